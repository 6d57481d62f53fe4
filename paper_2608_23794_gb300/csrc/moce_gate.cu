// Standalone temperature-gate kernel (Eq. (tau), Eq. (weights)): one CTA per
// (block of GE experts, example). The arithmetic lives in moce_gate_block.cuh.
#include "moce_gate_block.cuh"

namespace moce {
namespace {

__global__ void __launch_bounds__(kThreads) gate_kernel(
    const float *__restrict__ z, int C, int R, int k, const int32_t *__restrict__ pidx,
    const float *__restrict__ plog, const float *__restrict__ W1, const float *__restrict__ b1,
    const float *__restrict__ w2, const float *__restrict__ b2, float tmin, float tmax,
    float *__restrict__ tau, float *__restrict__ a) {
    extern __shared__ __align__(16) float gsm[];
    gate_block(gsm, blockIdx.y, blockIdx.x * GE, z, C, R, k, pidx, plog, W1, b1, w2, b2, tmin, tmax,
               tau, a);
}

}  // namespace

cudaError_t launch_gate(const float *z, int N, int C, int R, int k, const int32_t *pidx,
                        const float *plog, const float *W1, const float *b1, const float *w2,
                        const float *b2, float tmin, float tmax, float *tau, float *a,
                        cudaStream_t s) {
    if (N == 0) return cudaSuccess;
    const size_t smem = gate_smem(k);
    if (smem > 48 * 1024) {
        cudaError_t err =
            cudaFuncSetAttribute(gate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
    }
    const dim3 grid((R + GE - 1) / GE, N);
    gate_kernel<<<grid, kThreads, smem, s>>>(z, C, R, k, pidx, plog, W1, b1, w2, b2, tmin, tmax,
                                             tau, a);
    return cudaGetLastError();
}

size_t gate_smem_bytes(int k) { return gate_smem(k); }

}  // namespace moce
