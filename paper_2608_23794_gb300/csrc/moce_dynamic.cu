// Input-conditioned supports, Eq. (dynamic) (the variant of Sec. 5 that
// replaces the static support of Eq. (support) with a per-example one, at
// inference: deterministic hard TopK, no noise). Per example n:
//   h = ReLU(W_h z + b_h) in R^d                  router_hidden_kernel
//   L_e(X)_c = L_{e,c} + sum_j q_{e,j} h_j v_{c,j}  dyn_logits_kernel
//   S_e(X) = TopK(L_e(X), k), deployment order      launch_topk (moce_train.cu)
//                                                   over the N C_out rows
//   U(X) = channels no S_e(X) selects, ascending    dyn_resid_kernel
// then the gate (Eq. (tau), reading z at S_e(X)) and the weights (Eq.
// (weights), on the selected L_e(X) values) and the mix of the static path,
// with per-example supports. Every sum runs in a fixed order.
#include <math.h>

#include "moce_internal.cuh"

namespace moce {
namespace {

// h[n][j] = ReLU(b_h[j] + sum_c W_h[j][c] z[n][c]): a warp per (n, j), lanes
// over channels, then a fixed shuffle tree.
__global__ void __launch_bounds__(256) router_hidden_kernel(const float *__restrict__ z, int N,
                                                            int C, int d,
                                                            const float *__restrict__ Wh,
                                                            const float *__restrict__ bh,
                                                            float *__restrict__ h) {
    const int lane = threadIdx.x & 31;
    const size_t w = (size_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (w >= (size_t)N * d) return;
    const int n = (int)(w / d), j = (int)(w - (size_t)n * d);
    const float *wr = Wh + (size_t)j * C, *zn = z + (size_t)n * C;
    float s = 0.f;
    for (int c = lane; c < C; c += 32) s = fmaf(__ldg(wr + c), zn[c], s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) h[w] = fmaxf(s + __ldg(bh + j), 0.f);
}

// Ldyn[n][e][c] = L[e][c] + sum_j (q_{e,j} h[n][j]) v_{c,j}: a 64 x 64 tile of
// (expert, channel) per CTA, the rank-d product through shared memory in
// slices of 32, 4 x 4 outputs per thread, j in order.
constexpr int kDynT = 64, kDynJ = 32;
__global__ void __launch_bounds__(256) dyn_logits_kernel(const float *__restrict__ L,
                                                         const float *__restrict__ Q,
                                                         const float *__restrict__ V,
                                                         const float *__restrict__ h, int R, int C,
                                                         int d, float *__restrict__ Ld) {
    __shared__ __align__(16) float Gs[kDynJ][kDynT + 4], Vs[kDynJ][kDynT + 4];
    const int c0 = blockIdx.x * kDynT, e0 = blockIdx.y * kDynT, n = blockIdx.z;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const float *hn = h + (size_t)n * d;
    float acc[4][4] = {};
    for (int j0 = 0; j0 < d; j0 += kDynJ) {
        for (int q = tid; q < kDynT * kDynJ; q += 256) {
            const int r = q / kDynJ, jj = q - r * kDynJ, j = j0 + jj;
            const int e = e0 + r, c = c0 + r;
            Gs[jj][r] = (e < R && j < d) ? __ldg(Q + (size_t)e * d + j) * hn[j] : 0.f;
            Vs[jj][r] = (c < C && j < d) ? __ldg(V + (size_t)c * d + j) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int jj = 0; jj < kDynJ; ++jj) {
            const float4 g = *reinterpret_cast<const float4 *>(&Gs[jj][ty * 4]);
            const float4 v = *reinterpret_cast<const float4 *>(&Vs[jj][tx * 4]);
            const float gr[4] = {g.x, g.y, g.z, g.w}, vr[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(gr[a], vr[b], acc[a][b]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int e = e0 + ty * 4 + a;
        if (e >= R) continue;
        const float *Lr = L + (size_t)e * C;
        float *out = Ld + ((size_t)n * R + e) * C;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int c = c0 + tx * 4 + b;
            if (c < C) out[c] = __ldg(Lr + c) + acc[a][b];
        }
    }
}

// U(X) of example n: the channels that none of the example's R k selections
// hits, ascending, and their count. One CTA of 1024 threads per example: a
// bitmap of C bits in shared memory, then runs of words counted, scanned and
// written in order.
__global__ void __launch_bounds__(1024) dyn_resid_kernel(const int32_t *__restrict__ sidx, int R,
                                                         int k, int C,
                                                         int32_t *__restrict__ resid,
                                                         int32_t *__restrict__ nU) {
    extern __shared__ uint32_t bits[];
    __shared__ int32_t part[1024];
    const int n = blockIdx.x, t = threadIdx.x;
    const int nw = (C + 31) >> 5;
    for (int w = t; w < nw; w += 1024) bits[w] = 0u;
    __syncthreads();
    const int32_t *sn = sidx + (size_t)n * R * k;
    for (int q = t; q < R * k; q += 1024) {
        const int c = __ldg(sn + q);
        if ((unsigned)c < (unsigned)C) atomicOr(bits + (c >> 5), 1u << (c & 31));
    }
    __syncthreads();
    const int per = (nw + 1023) / 1024, w0 = min(nw, t * per), w1 = min(nw, w0 + per);
    auto free_bits = [&](int w) {
        uint32_t m = ~bits[w];
        if (w == nw - 1 && (C & 31)) m &= (1u << (C & 31)) - 1u;  // channels past C
        return m;
    };
    int cnt = 0;
    for (int w = w0; w < w1; ++w) cnt += __popc(free_bits(w));
    part[t] = cnt;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {  // inclusive scan of the run counts
        const int v = t >= o ? part[t - o] : 0;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    int pos = part[t] - cnt;
    int32_t *rn = resid + (size_t)n * C;
    for (int w = w0; w < w1; ++w) {
        uint32_t m = free_bits(w);
        while (m) {
            const int b = __ffs(m) - 1;
            rn[pos++] = (w << 5) + b;
            m &= m - 1u;
        }
    }
    if (t == 1023) nU[n] = part[1023];
}

}  // namespace

DynLayout dyn_layout(int N, int HW, int C, int R, int k, int d) {
    DynLayout D;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
    D.err = take(4);
    D.h = take((size_t)N * d * 4);
    D.Ld = take((size_t)N * R * C * 4);
    D.sidx = take((size_t)N * R * k * 4);
    D.slog = take((size_t)N * R * k * 4);
    D.resid = take((size_t)N * C * 4);
    D.nU = take((size_t)N * 4);
    D.routing = off;  // the buffers above do not depend on H W
    D.fwd_off = off;
    D.fwd = ws_layout(N, HW, C, R, k);
    D.total = off + D.fwd.total;
    return D;
}

bool dynamic_supported(int C, int k) {
    return topk_smem_bytes(C, k) <= 227 * 1024 && (size_t)((C + 31) / 32) * 4 <= 64 * 1024;
}

cudaError_t launch_dynamic_supports(const float *z, int N, int C, int R, int k, int d,
                                    const float *L, const float *Wh, const float *bh,
                                    const float *V, const float *Q, float *h, float *Ld,
                                    int32_t *sidx, float *slog, int32_t *resid, int32_t *nU,
                                    uint32_t *err, cudaStream_t s) {
    if (N == 0) return cudaSuccess;
    router_hidden_kernel<<<(unsigned)(((size_t)N * d + 7) / 8), 256, 0, s>>>(z, N, C, d, Wh, bh, h);
    const dim3 grid((C + kDynT - 1) / kDynT, (R + kDynT - 1) / kDynT, N);
    dyn_logits_kernel<<<grid, 256, 0, s>>>(L, Q, V, h, R, C, d, Ld);
    cudaError_t e = cudaMemsetAsync(err, 0, 4, s);
    if (e != cudaSuccess) return e;
    e = launch_topk(Ld, N * R, C, k, sidx, slog, err, s);
    if (e != cudaSuccess) return e;
    const size_t smem = (size_t)((C + 31) / 32) * 4;
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(dyn_resid_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
    }
    dyn_resid_kernel<<<N, 1024, smem, s>>>(sidx, R, k, C, resid, nU);
    return cudaGetLastError();
}

}  // namespace moce
