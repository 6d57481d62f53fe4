// Global average pooling z = GAP(x) (Sec. 3.3), fp32 accumulation in a fixed
// order so results are reproducible run to run.
//
// NHWC: pool_nhwc_partial_kernel reduces one tile of pool_px positions of one
// example into per-channel partial sums (16-byte vector loads, one channel
// vector per thread, several position rows per CTA reduced through shared
// memory); pool_finalize_kernel adds the tile partials in tile order and
// divides by H*W. NCHW: each channel plane is contiguous, one warp reduces a
// plane with a fixed shuffle tree.
#include "moce_internal.cuh"

namespace moce {
namespace {

template <typename T, int VEC> struct VecLoad;
template <> struct VecLoad<uint16_t, 8> {
    static __device__ __forceinline__ void add(const uint16_t *p, float *acc) {
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(p));
        acc[0] += bf16lo(v.x); acc[1] += bf16hi(v.x);
        acc[2] += bf16lo(v.y); acc[3] += bf16hi(v.y);
        acc[4] += bf16lo(v.z); acc[5] += bf16hi(v.z);
        acc[6] += bf16lo(v.w); acc[7] += bf16hi(v.w);
    }
};
template <> struct VecLoad<float, 4> {
    static __device__ __forceinline__ void add(const float *p, float *acc) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(p));
        acc[0] += v.x; acc[1] += v.y; acc[2] += v.z; acc[3] += v.w;
    }
};
template <typename T> struct VecLoad<T, 1> {
    static __device__ __forceinline__ void add(const T *p, float *acc) { acc[0] += load_elem<T>(p); }
};

// grid (pool_tiles, N); partial[(n*tiles + t)*C + c]
template <typename T, int VEC>
__global__ void __launch_bounds__(kThreads) pool_nhwc_partial_kernel(const T *__restrict__ x, int HW,
                                                                     int C, int PP, int tiles,
                                                                     float *__restrict__ partial) {
    __shared__ float red[kThreads * VEC];
    const int n = blockIdx.y, t = blockIdx.x;
    const int p0 = t * PP, p1 = min(HW, p0 + PP);
    const int V = C / VEC;
    const int span = V < kThreads ? V : kThreads;
    const int rows = kThreads / span;
    const int row = threadIdx.x / span, cvl = threadIdx.x % span;
    const T *xe = x + (size_t)n * HW * C;
    float *out = partial + ((size_t)n * tiles + t) * C;
    for (int cv0 = 0; cv0 < V; cv0 += span) {
        const int cv = cv0 + cvl;
        float acc[VEC];
#pragma unroll
        for (int j = 0; j < VEC; ++j) acc[j] = 0.f;
        if (row < rows && cv < V) {
            const T *col = xe + (size_t)cv * VEC;
            int p = p0 + row;
            for (; p + 3 * rows < p1; p += 4 * rows) {
                VecLoad<T, VEC>::add(col + (size_t)p * C, acc);
                VecLoad<T, VEC>::add(col + (size_t)(p + rows) * C, acc);
                VecLoad<T, VEC>::add(col + (size_t)(p + 2 * rows) * C, acc);
                VecLoad<T, VEC>::add(col + (size_t)(p + 3 * rows) * C, acc);
            }
            for (; p < p1; p += rows) VecLoad<T, VEC>::add(col + (size_t)p * C, acc);
        }
        if (rows == 1) {
            if (cv < V) {
#pragma unroll
                for (int j = 0; j < VEC; ++j) out[(size_t)cv * VEC + j] = acc[j];
            }
        } else {
            if (row < rows) {
#pragma unroll
                for (int j = 0; j < VEC; ++j) red[(row * span + cvl) * VEC + j] = acc[j];
            }
            __syncthreads();
            for (int q = threadIdx.x; q < span * VEC; q += kThreads) {
                float s = 0.f;
                for (int r = 0; r < rows; ++r) s += red[r * span * VEC + q];
                out[(size_t)cv0 * VEC + q] = s;
            }
            __syncthreads();
        }
    }
}

__global__ void __launch_bounds__(kThreads) pool_finalize_kernel(const float *__restrict__ partial,
                                                                 int N, int C, int tiles, int HW,
                                                                 float *__restrict__ z) {
    const size_t q = (size_t)blockIdx.x * kThreads + threadIdx.x;
    if (q >= (size_t)N * C) return;
    const size_t n = q / C, c = q % C;
    const float *p = partial + n * tiles * C + c;
    float s = 0.f;
    for (int t = 0; t < tiles; ++t) s += p[(size_t)t * C];
    z[q] = s / (float)HW;
}

// one warp per (n, c) plane
template <typename T>
__global__ void __launch_bounds__(kThreads) pool_nchw_kernel(const T *__restrict__ x, int N, int C,
                                                             int HW, float *__restrict__ z) {
    const size_t plane = (size_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (plane >= (size_t)N * C) return;
    const T *xp = x + plane * HW;
    float s = 0.f;
    for (int p = lane; p < HW; p += 32) s += load_elem<T>(xp + p);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) z[plane] = s / (float)HW;
}

}  // namespace

cudaError_t launch_pool(const void *x, int N, int HW, int C, moce_dtype_t dt, moce_layout_t lay,
                        float *z, const WsLayout &L, unsigned char *ws, cudaStream_t s) {
    if (N == 0) return cudaSuccess;
    if (lay == MOCE_NCHW) {
        const size_t planes = (size_t)N * C;
        const unsigned grid = (unsigned)((planes + 7) / 8);
        if (dt == MOCE_BF16)
            pool_nchw_kernel<uint16_t><<<grid, kThreads, 0, s>>>((const uint16_t *)x, N, C, HW, z);
        else
            pool_nchw_kernel<float><<<grid, kThreads, 0, s>>>((const float *)x, N, C, HW, z);
        return cudaGetLastError();
    }
    float *partial = reinterpret_cast<float *>(ws + L.partial);
    const dim3 grid(L.pool_tiles, N);
    const bool aligned = (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
    if (dt == MOCE_BF16) {
        if (aligned && C % 8 == 0)
            pool_nhwc_partial_kernel<uint16_t, 8><<<grid, kThreads, 0, s>>>(
                (const uint16_t *)x, HW, C, L.pool_px, L.pool_tiles, partial);
        else
            pool_nhwc_partial_kernel<uint16_t, 1><<<grid, kThreads, 0, s>>>(
                (const uint16_t *)x, HW, C, L.pool_px, L.pool_tiles, partial);
    } else {
        if (aligned && C % 4 == 0)
            pool_nhwc_partial_kernel<float, 4><<<grid, kThreads, 0, s>>>(
                (const float *)x, HW, C, L.pool_px, L.pool_tiles, partial);
        else
            pool_nhwc_partial_kernel<float, 1><<<grid, kThreads, 0, s>>>(
                (const float *)x, HW, C, L.pool_px, L.pool_tiles, partial);
    }
    const size_t nz = (size_t)N * C;
    pool_finalize_kernel<<<(unsigned)((nz + kThreads - 1) / kThreads), kThreads, 0, s>>>(
        partial, N, C, L.pool_tiles, HW, z);
    return cudaGetLastError();
}

}  // namespace moce
