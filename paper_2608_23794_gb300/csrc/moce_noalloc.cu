// moce_forward_noalloc: the layer forward for callers that cannot allocate
// device memory.
//
// Some callers cannot call cudaMalloc at the point where they run a layer:
// code inside a custom allocator or a memory-pool callback, real-time loops
// that forbid allocation after start-up, plugins whose host framework owns
// every device buffer, or processes that have handed all free memory to a
// pool. They still own x, y and the packed tables, but cannot provide the
// forward's workspace. This entry point uses a fixed scratch array that lives
// in this library's device image instead, so it never allocates.
#include <mutex>

#include "moce_internal.cuh"

namespace {

// Scratch for one forward at a time. Every GPU that loads this library holds
// these bytes until the process exits. Layers whose workspace
// (moce_workspace_bytes) is larger are rejected.
constexpr size_t kNoAllocScratchBytes = 8u << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device. In host code
// the array's name is only a host-side stand-in, so the address must come
// from cudaGetSymbolAddress, once per device, with that device current.
cudaError_t scratch_address(void **out) {
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (err != cudaSuccess) return err;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" moce_status_t moce_forward_noalloc(
    const void *x, int N, int H, int W, int C_in, int C_out, int k, moce_dtype_t dtype,
    moce_layout_t layout, const int32_t *packed_idx, const float *packed_logits,
    const int32_t *resid_idx, int n_resid, const float *W1, const float *b1, const float *w2,
    const float *b2, float tau_min, float tau_max, void *y, moce_stream_t stream) {
    const size_t need = moce_workspace_bytes(N, H, W, C_in, C_out, k);
    if (need == 0) return MOCE_ERR_INVALID_VALUE;
    if (need > kNoAllocScratchBytes) return MOCE_ERR_UNSUPPORTED;
    void *scratch = nullptr;
    if (scratch_address(&scratch) != cudaSuccess) return MOCE_ERR_CUDA;
    // The array keeps whatever the previous call left in it. The stream
    // kernel's control words and tagged values must start from zero, so the
    // part this layer uses is cleared on the caller's stream first.
    if (cudaMemsetAsync(scratch, 0, need, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return MOCE_ERR_CUDA;
    return moce_forward(x, N, H, W, C_in, C_out, k, dtype, layout, packed_idx, packed_logits,
                        resid_idx, n_resid, W1, b1, w2, b2, tau_min, tau_max, y, scratch, need,
                        stream);
}

// The control words sit at the start of the scratch (the workspace layout
// every forward uses): the error word of the last forward on this device.
extern "C" moce_status_t moce_noalloc_check_device_error(moce_stream_t stream) {
    void *scratch = nullptr;
    if (scratch_address(&scratch) != cudaSuccess) return MOCE_ERR_CUDA;
    return moce_check_device_error(scratch, moce::kCtrlWords * 4, stream);
}
