// noalloc.cu -- Wgrad entry point that allocates nothing and needs no
// caller-supplied scratch.
//
// Some callers cannot obtain device memory when they run the backward pass:
// plugin hosts (inference/training engines that own every device buffer and
// forbid allocations inside their execution callbacks), code on a
// latency-critical path where cudaMalloc's device-wide synchronisation is not
// acceptable, or a caller whose memory budget is fixed up front.  The normal
// puro_fp8_linear_wgrad wants such a caller to hand in scratch for its
// split-reduction schedule.  This variant instead keeps that scratch in a
// file-scope device array of fixed size, part of the library image, so the
// caller passes only inputs and outputs.
#include <mutex>

#include "internal.h"

namespace puro {
namespace {

// Scratch for the FP32 partial tiles of the split reduction.  Every GPU that
// loads this library holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_wgrad_scratch[PURO_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of g_wgrad_scratch on the current device.  In host code
// the array's name is only a host-side stand-in for the symbol, so the real
// device address is looked up once per device (with that device current)
// and cached for the life of the process: after cudaDeviceReset the cached
// address is stale (the header says so).
cudaError_t scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_wgrad_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace puro

using namespace puro;

extern "C" __attribute__((visibility("default"))) puro_status_t puro_fp8_linear_wgrad_noalloc(
    const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw, int32_t *dev_status, void *stream) {
    // The regular Wgrad's argument checks first, so a malformed call is
    // reported as such whatever its shape; then the split schedule this
    // shape would take must fit the fixed scratch.
    const puro_status_t st = fp8_gemm_validate(dy_t, x_t, dw);
    if (st != PURO_OK) return st;
    const size_t need = splitk_workspace_bytes(dy_t->rows, x_t->rows, dy_t->red, false);
    if (need > PURO_NOALLOC_SCRATCH_BYTES) return PURO_ERR_UNSUPPORTED;
    void *scratch = nullptr;
    if (need > 0 && dy_t->rows > 0 && x_t->rows > 0) {
        if (scratch_address(&scratch) != cudaSuccess) return PURO_ERR_CUDA;
    }
    return fp8_gemm_entry(dy_t, x_t, dw, scratch, scratch ? PURO_NOALLOC_SCRATCH_BYTES : 0, dev_status, stream);
}
