// Global average pooling z = GAP(x) (Sec. 3.3), fp32 accumulation in a fixed
// order so results are reproducible run to run.
//
// NHWC: pool_nhwc_kernel gives a CTA one example, one block of CB channel
// vectors (16 bytes each: a warp reads 512 contiguous bytes of a position
// row) and one span of positions; its rows = 256 / CB thread rows take every
// rows-th position of the span, and the rows' sums are added in row order
// through shared memory; a thread keeps kPoolU loads in flight. One span
// per example (z written directly) when the (example, channel block) CTAs
// fill half the GPU; otherwise enough spans to fill it, whose tile sums
// pool_finalize_kernel adds in span order and divides by H*W. NCHW: each
// channel plane is contiguous, one warp reduces a plane with a fixed shuffle
// tree.
#include <algorithm>

#include "moce_internal.cuh"

namespace moce {
namespace {

#ifndef MOCE_POOL_CTAS
#define MOCE_POOL_CTAS (152 * 8)
#endif
#ifndef MOCE_POOL_HINT
#define MOCE_POOL_HINT 1
#endif
constexpr long long kPoolCtas = MOCE_POOL_CTAS;  // one wave of 8 CTAs per SM

#ifndef MOCE_POOL_UNROLL
#define MOCE_POOL_UNROLL 8
#endif
constexpr int kPoolU = MOCE_POOL_UNROLL;  // loads in flight per thread

// Vector loads of the NHWC pool: load() fetches one vector from a valid
// address and zeroes it when ok is false (past the span: no branch, so a
// thread's loads are all in flight), add() adds it to the channel sums.
template <typename T, int VEC> struct VecLoad;
template <> struct VecLoad<uint16_t, 8> {
    using V = uint4;
    static __device__ __forceinline__ V load(const uint16_t *p, bool ok) {
        V v;
#if MOCE_POOL_HINT
        asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "l"(p));
#else
        v = __ldg(reinterpret_cast<const uint4 *>(p));
#endif
        const uint32_t m = ok ? 0xffffffffu : 0u;
        v.x &= m; v.y &= m; v.z &= m; v.w &= m;
        return v;
    }
    static __device__ __forceinline__ void add(const V &v, float *acc) {
        acc[0] += bf16lo(v.x); acc[1] += bf16hi(v.x);
        acc[2] += bf16lo(v.y); acc[3] += bf16hi(v.y);
        acc[4] += bf16lo(v.z); acc[5] += bf16hi(v.z);
        acc[6] += bf16lo(v.w); acc[7] += bf16hi(v.w);
    }
};
template <> struct VecLoad<float, 4> {
    using V = float4;
    static __device__ __forceinline__ V load(const float *p, bool ok) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(p));
        return ok ? v : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    static __device__ __forceinline__ void add(const V &v, float *acc) {
        acc[0] += v.x; acc[1] += v.y; acc[2] += v.z; acc[3] += v.w;
    }
};
template <typename T> struct VecLoad<T, 1> {
    using V = float;
    static __device__ __forceinline__ V load(const T *p, bool ok) {
        const float v = load_elem<T>(p);
        return ok ? v : 0.f;
    }
    static __device__ __forceinline__ void add(const V &v, float *acc) { acc[0] += v; }
};

// grid (chunks, spans, N). Thread (row, cvl): channel vector ch CB + cvl,
// positions p0 + row, p0 + row + rows, ... of the span. One span: z[n][c]
// = sum / HW; otherwise partial[(n spans + t) C + c] = the span's sum.
template <typename T, int VEC>
__global__ void __launch_bounds__(kThreads) pool_nhwc_kernel(const T *__restrict__ x, int HW, int C,
                                                             int CB, int PT, int spans,
                                                             float *__restrict__ partial,
                                                             float *__restrict__ z) {
    __shared__ float red[kThreads * VEC];  // [row][j][cvl]
    const int ch = blockIdx.x, t = blockIdx.y, n = blockIdx.z;
    const int V = C / VEC, rows = kThreads / CB;
    const int row = threadIdx.x / CB, cvl = threadIdx.x - row * CB;
    const int cv = ch * CB + cvl;
    const int p0 = t * PT, p1 = min(HW, p0 + PT);
    float acc[VEC];
#pragma unroll
    for (int j = 0; j < VEC; ++j) acc[j] = 0.f;
    if (row < rows && cv < V) {
        using L = VecLoad<T, VEC>;
        const T *col = x + (size_t)n * HW * C + (size_t)cv * VEC;
        // kPoolU loads in flight (the last batch predicated), added in
        // position order
        for (int p = p0 + row; p < p1; p += kPoolU * rows) {
            typename L::V v[kPoolU];
#pragma unroll
            for (int u = 0; u < kPoolU; ++u) {
                const int pu = p + u * rows;
                v[u] = L::load(col + (size_t)(pu < p1 ? pu : p) * C, pu < p1);
            }
#pragma unroll
            for (int u = 0; u < kPoolU; ++u) L::add(v[u], acc);
        }
    }
    if (row < rows) {
#pragma unroll
        for (int j = 0; j < VEC; ++j) red[(row * VEC + j) * CB + cvl] = acc[j];
    }
    __syncthreads();
    for (int q = threadIdx.x; q < CB * VEC; q += kThreads) {
        const int j = q / CB, v = ch * CB + (q - j * CB);
        if (v >= V) continue;
        float s = 0.f;
        for (int r = 0; r < rows; ++r) s += red[r * VEC * CB + q];
        const size_t c = (size_t)v * VEC + j;
        if (spans == 1) z[(size_t)n * C + c] = s / (float)HW;
        else partial[((size_t)n * spans + t) * C + c] = s;
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

PoolPlan pool_plan(const void *x, int N, int HW, int C, moce_dtype_t dt) {
    PoolPlan pp;
    const bool aligned = (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
    pp.vec = dt == MOCE_BF16 ? (aligned && C % 8 == 0 ? 8 : 1) : (aligned && C % 4 == 0 ? 4 : 1);
    const int V = C / pp.vec;
    pp.CB = V < 32 ? V : 32;
    const int rows = kThreads / pp.CB;
    pp.chunks = (unsigned)((V + pp.CB - 1) / pp.CB);
    // spans per example: one (z written directly, no second launch) once the
    // (example, channel block) CTAs alone reach half a wave; otherwise about
    // kPoolCtas CTAs in all, at most one span per thread row of positions and
    // no more than the workspace's tile partials (ws_layout's pool_tiles)
    const long long base = (long long)N * pp.chunks;
    const int px = pool_tile_px(C), tiles = (HW + px - 1) / px;
    long long spans = 2 * base >= kPoolCtas ? 1 : (kPoolCtas + base - 1) / base;
    spans = std::min<long long>(spans, std::min<long long>(tiles, (HW + rows - 1) / rows));
    spans = std::max<long long>(1, std::min<long long>(spans, 65535));  // a grid dimension
    pp.PT = (int)((HW + spans - 1) / spans);
    pp.spans = (HW + pp.PT - 1) / pp.PT;
    return pp;
}

int pool_launches(const void *x, int N, int HW, int C, moce_dtype_t dt, moce_layout_t lay) {
    if (N == 0 || HW <= 0) return 0;
    if (lay == MOCE_NCHW) return 1;
    return pool_plan(x, N, HW, C, dt).spans > 1 ? 2 : 1;
}

cudaError_t launch_pool(const void *x, int N, int HW, int C, moce_dtype_t dt, moce_layout_t lay,
                        float *z, const WsLayout &L, unsigned char *ws, cudaStream_t s) {
    if (N == 0 || HW <= 0) return cudaSuccess;
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
    const PoolPlan pp = pool_plan(x, N, HW, C, dt);
    const int VEC = pp.vec, CB = pp.CB, PT = pp.PT, S = pp.spans;
    const unsigned chunks = pp.chunks;
    if (S > L.pool_tiles) return cudaErrorInvalidValue;  // the tile sums would not fit
    const dim3 grid(chunks, (unsigned)S, (unsigned)N);
    if (dt == MOCE_BF16) {
        if (VEC == 8)
            pool_nhwc_kernel<uint16_t, 8><<<grid, kThreads, 0, s>>>((const uint16_t *)x, HW, C, CB,
                                                                    PT, S, partial, z);
        else
            pool_nhwc_kernel<uint16_t, 1><<<grid, kThreads, 0, s>>>((const uint16_t *)x, HW, C, CB,
                                                                    PT, S, partial, z);
    } else {
        if (VEC == 4)
            pool_nhwc_kernel<float, 4><<<grid, kThreads, 0, s>>>((const float *)x, HW, C, CB, PT, S,
                                                                 partial, z);
        else
            pool_nhwc_kernel<float, 1><<<grid, kThreads, 0, s>>>((const float *)x, HW, C, CB, PT, S,
                                                                 partial, z);
    }
    if (S > 1) {
        const size_t nz = (size_t)N * C;
        pool_finalize_kernel<<<(unsigned)((nz + kThreads - 1) / kThreads), kThreads, 0, s>>>(
            partial, N, C, S, HW, z);
    }
    return cudaGetLastError();
}

}  // namespace moce
