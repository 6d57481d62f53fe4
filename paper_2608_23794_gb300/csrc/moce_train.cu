// Support maintenance on the full routing matrix L [R][C] (training side):
//
//   topk_warp_kernel,     Eq. (support), Sec. 3.2: S_e = TopK(L_e, k), written in
//   topk_cta_kernel       deployment order (descending logit, equal logits by
//                         ascending channel; -0.0 equals +0.0), so the result
//                         is already packed. One warp (many rows, small k) or
//                         one CTA (few rows or large k) per row: a radix select
//                         of the k-th order key, an ordered compaction of the
//                         k selected (key, channel) pairs, then a bitonic sort
//                         of only those, as 64-bit keys whose low word is the
//                         channel.
//   coverage kernels      Sec. 3.4: p_{e,c} = softmax(L_e)_c over all C channels,
//                         u_c = (1/R) sum_e p_{e,c}, ubar = (1/C) sum_c u_c,
//                         L_cov = sum_c (u_c - ubar)^2 / (ubar^2 + eps), and
//                         dL_cov/dL_{e,c} = (1/R) p_{e,c} (g_c - sum_c' p_{e,c'} g_c')
//                         with g_c = dL_cov/du_c. Row statistics (max, sum of
//                         exponentials), then partial column sums over chunks
//                         of kRowChunk rows (in row order, in double), then u
//                         (the chunks in order), then the loss and g (one CTA,
//                         double), then the gradient by rows.
// Every sum runs in a fixed order: the results do not depend on scheduling.
#include <math.h>

#include "moce_select.cuh"

namespace moce {
namespace {

constexpr int kTrainThreads = 512;
constexpr int kRowChunk = 32;  // rows per partial column sum
constexpr uint32_t kTopkBadLogit = 1u;

__device__ float block_sum_f(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float s = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];  // warp order
    return s;
}
__device__ float block_max_f(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float s = -INFINITY;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s = fmaxf(s, red[w]);
    return s;
}
__device__ double block_sum_d(double v, double *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    double s = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
    return s;
}

// Shared memory of one warp's row: the KP selected pairs, 256 histogram bins
// and the row's C order keys.
__host__ __device__ inline size_t topk_warp_smem(int C, int k) {
    int kp = 1;
    while (kp < k) kp <<= 1;
    return align_up((size_t)kp * 8 + 256 * 4 + (size_t)C * 4, 16);
}

// One row per warp (W warps per CTA, no block barriers): the row's C order
// keys in the warp's shared memory, then warp_select (moce_select.cuh).
__global__ void __launch_bounds__(256) topk_warp_kernel(const float *__restrict__ L, int R,
                                                          int C, int k, int KP,
                                                          int32_t *__restrict__ idx_out,
                                                          float *__restrict__ lg_out,
                                                          uint32_t *err) {
    extern __shared__ __align__(8) unsigned char ksm[];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const size_t per_warp = topk_warp_smem(C, k);
    unsigned char *base = ksm + (size_t)w * per_warp;
    unsigned long long *sel = reinterpret_cast<unsigned long long *>(base);   // [KP]
    uint32_t *hist = reinterpret_cast<uint32_t *>(base + (size_t)KP * 8);    // [256]
    uint32_t *key = hist + 256;                                               // [C]
    const size_t e = (size_t)blockIdx.x * (blockDim.x >> 5) + w;
    if (e >= (size_t)R) return;
    const float *Le = L + e * C;
    for (int c = lane; c < C; c += 32) {
        const float v = Le[c];
        if (!isfinite(v)) atomicOr(err, kTopkBadLogit);
        key[c] = desc_key(v);
    }
    __syncwarp();
    warp_select(key, C, k, KP, hist, sel);
    for (int i = lane; i < k; i += 32) {
        const uint32_t c = (uint32_t)(sel[i] & 0xffffffffu);
        idx_out[e * k + i] = (int32_t)c;
        lg_out[e * k + i] = Le[c];
    }
}

// One row per CTA (256 threads): the row's C order keys in shared memory;
// four 8-bit radix passes find T, the k-th smallest key, and how many of the
// keys equal to T are taken (the lowest channels first, as the tie rule
// orders them); an ordered compaction (ballots, in channel order) collects
// the k selected (key, channel) pairs; a bitonic sort of those KP = k rounded
// up to a power of two pairs gives deployment order.
constexpr int kSelThreads = 256;
__global__ void __launch_bounds__(kSelThreads) topk_cta_kernel(const float *__restrict__ L,
                                                                   int C, int k, int KP,
                                                                   int32_t *__restrict__ idx_out,
                                                                   float *__restrict__ lg_out,
                                                                   uint32_t *err) {
    extern __shared__ __align__(8) unsigned char ksm[];
    unsigned long long *sel = reinterpret_cast<unsigned long long *>(ksm);  // [KP]
    uint32_t *key = reinterpret_cast<uint32_t *>(ksm + (size_t)KP * 8);    // [C]
    __shared__ uint32_t hist[256], wl[kSelThreads / 32], we[kSelThreads / 32];
    __shared__ uint32_t s_prefix, s_kk;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const size_t e = blockIdx.x;
    const float *Le = L + e * C;
    for (int c = tid; c < C; c += kSelThreads) {
        const float v = Le[c];
        if (!isfinite(v)) atomicOr(err, kTopkBadLogit);
        key[c] = desc_key(v);
    }
    for (int i = tid; i < KP; i += kSelThreads) sel[i] = ~0ull;
    uint32_t prefix = 0u, mask = 0u, kk = (uint32_t)k;  // kk: rank sought among the prefix's keys
    for (int shift = 24; shift >= 0; shift -= 8) {
        hist[tid] = 0u;
        __syncthreads();
        for (int c = tid; c < C; c += kSelThreads) {
            const uint32_t kc = key[c];
            if ((kc & mask) == prefix) atomicAdd(hist + ((kc >> shift) & 255u), 1u);
        }
        __syncthreads();
        const uint32_t h = hist[tid];
        uint32_t incl = h;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) wl[warp] = incl;
        __syncthreads();
        for (int w = 0; w < warp; ++w) incl += wl[w];
        const uint32_t excl = incl - h;
        if (excl < kk && kk <= incl) {
            s_prefix = prefix | ((uint32_t)tid << shift);
            s_kk = kk - excl;
        }
        __syncthreads();
        prefix = s_prefix;
        kk = s_kk;
        mask |= 0xffu << shift;
        __syncthreads();
    }
    // prefix = T; the k - kk keys below T all belong, then the first kk equal to T
    const uint32_t T = prefix, nless = (uint32_t)k - kk;
    uint32_t run_l = 0u, run_e = 0u;
    const uint32_t lt = (1u << lane) - 1u;
    for (int j0 = 0; j0 < C; j0 += kSelThreads) {
        const int c = j0 + tid;
        const uint32_t kc = c < C ? key[c] : 0xffffffffu;
        const bool isl = c < C && kc < T, ise = c < C && kc == T;
        const uint32_t bl = __ballot_sync(0xffffffffu, isl), be = __ballot_sync(0xffffffffu, ise);
        if (lane == 0) {
            wl[warp] = __popc(bl);
            we[warp] = __popc(be);
        }
        __syncthreads();
        uint32_t ol = run_l, oe = run_e, tl = 0u, te = 0u;
        for (int w = 0; w < kSelThreads / 32; ++w) {
            if (w < warp) {
                ol += wl[w];
                oe += we[w];
            }
            tl += wl[w];
            te += we[w];
        }
        const unsigned long long k64 = ((unsigned long long)kc << 32) | (uint32_t)c;
        if (isl) sel[ol + __popc(bl & lt)] = k64;
        if (ise) {
            const uint32_t r = oe + __popc(be & lt);
            if (r < kk) sel[nless + r] = k64;
        }
        run_l += tl;
        run_e += te;
        __syncthreads();
    }
    // bitonic sort of the KP pairs, ascending keys (padding sorts last)
    for (int size = 2; size <= KP; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = tid; i < KP / 2; i += kSelThreads) {
                const int lo = 2 * i - (i & (stride - 1));  // pair (lo, lo + stride)
                const int hi = lo + stride;
                const bool up = (lo & size) == 0;
                const unsigned long long a = sel[lo], b = sel[hi];
                if ((a > b) == up) {
                    sel[lo] = b;
                    sel[hi] = a;
                }
            }
            __syncthreads();
        }
    }
    for (int i = tid; i < k; i += kSelThreads) {
        const uint32_t c = (uint32_t)(sel[i] & 0xffffffffu);
        idx_out[e * k + i] = (int32_t)c;
        lg_out[e * k + i] = Le[c];
    }
}

// Row statistics: stat[e] = {max_c L_{e,c}, sum_c exp(L_{e,c} - max)}.
__global__ void __launch_bounds__(kTrainThreads) cov_rows_kernel(const float *__restrict__ L,
                                                                  int C, float2 *__restrict__ stat) {
    __shared__ float red[kTrainThreads / 32];
    const int e = blockIdx.x;
    const float *Le = L + (size_t)e * C;
    float m = -INFINITY;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) m = fmaxf(m, Le[c]);
    m = block_max_f(m, red);
    float s = 0.f;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) s += expf(Le[c] - m);
    s = block_sum_f(s, red);
    if (threadIdx.x == 0) stat[e] = make_float2(m, s);
}

// Partial column sums: part[j][c] = sum over rows j kRowChunk .. + kRowChunk - 1
// (in order) of p_{e,c}, in double; thread c of a 256-column block, chunk
// j = blockIdx.y (coalesced row segments).
__global__ void __launch_bounds__(256) cov_cols_kernel(const float *__restrict__ L, int R, int C,
                                                       const float2 *__restrict__ stat,
                                                       double *__restrict__ part) {
    const int c = blockIdx.x * 256 + threadIdx.x;
    if (c >= C) return;
    const int e0 = blockIdx.y * kRowChunk, e1 = min(R, e0 + kRowChunk);
    double s = 0.0;
#pragma unroll 8
    for (int e = e0; e < e1; ++e) {
        const float2 st = stat[e];
        s += (double)(expf(L[(size_t)e * C + c] - st.x) / st.y);
    }
    part[(size_t)blockIdx.y * C + c] = s;
}

// u_c = (1/R) sum_j part[j][c], the chunks in order; kept in the part
// buffer's row 0 (thread c alone reads column c).
__global__ void __launch_bounds__(256) cov_usage_kernel(double *__restrict__ part, int R, int C,
                                                        int chunks) {
    const int c = blockIdx.x * 256 + threadIdx.x;
    if (c >= C) return;
    double t = 0.0;
#pragma unroll 8
    for (int j = 0; j < chunks; ++j) t += part[(size_t)j * C + c];
    part[c] = t / (double)R;
}

// The loss and g_c = dL_cov/du_c from u; one CTA, double.
__global__ void __launch_bounds__(kTrainThreads) cov_loss_kernel(const double *__restrict__ u,
                                                                  int C, double eps,
                                                                  float *__restrict__ loss,
                                                                  float *__restrict__ u_out,
                                                                  float *__restrict__ g) {
    __shared__ double red[kTrainThreads / 32];
    double s = 0.0;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) s += u[c];
    const double ubar = block_sum_d(s, red) / (double)C;
    double S = 0.0, dev = 0.0;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) {
        const double d = u[c] - ubar;
        S += d * d;
        dev += d;
    }
    S = block_sum_d(S, red);
    dev = block_sum_d(dev, red);
    const double D = ubar * ubar + eps;
    if (threadIdx.x == 0) *loss = (float)(S / D);
    // g_c = 2 (u_c - ubar) / D + shift, the shift (the same for every c) from
    // the dependence of ubar on u; the divisions once per CTA
    const double twoD = 2.0 / D;
    const double shift = -2.0 * dev / ((double)C * D) - 2.0 * ubar * S / ((double)C * D * D);
    for (int c = threadIdx.x; c < C; c += kTrainThreads) {
        if (u_out) u_out[c] = (float)u[c];
        if (g) g[c] = (float)(twoD * (u[c] - ubar) + shift);
    }
}

// dL_cov/dL_{e,c} = (1/R) p_{e,c} (g_c - sum_c' p_{e,c'} g_c'), one CTA per row.
__global__ void __launch_bounds__(kTrainThreads) cov_grad_kernel(const float *__restrict__ L, int R,
                                                                  int C,
                                                                  const float2 *__restrict__ stat,
                                                                  const float *__restrict__ g,
                                                                  float *__restrict__ grad) {
    __shared__ float red[kTrainThreads / 32];
    const int e = blockIdx.x;
    const float *Le = L + (size_t)e * C;
    const float2 st = stat[e];
    float dot = 0.f;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) dot += expf(Le[c] - st.x) / st.y * g[c];
    dot = block_sum_f(dot, red);
    const float inv_R = 1.f / (float)R;
    for (int c = threadIdx.x; c < C; c += kTrainThreads) {
        const float p = expf(Le[c] - st.x) / st.y;
        grad[(size_t)e * C + c] = p * (g[c] - dot) * inv_R;
    }
}

}  // namespace

static int pow2_at_least(int v) {
    int p = 1;
    while (p < v) p <<= 1;
    return p;
}

size_t topk_smem_bytes(int C, int k) { return topk_warp_smem(C, k); }  // >= the CTA kernel's

// Workspace of the support-maintenance calls: the error word, the row
// statistics, u in double and g.
size_t train_ws_bytes(int R, int C) {
    const size_t chunks = (size_t)(R + kRowChunk - 1) / kRowChunk;
    return align_up(16, 256) + align_up((size_t)R * 8, 256) + align_up(chunks * C * 8, 256) +
           align_up((size_t)C * 4, 256);
}

// Many rows with a small k (the per-example rows of the input-conditioned
// variant) go one per warp; few rows or a large k one per CTA (more threads
// per row for the sort, and every SM busy).
cudaError_t launch_topk(const float *L, int R, int C, int k, int32_t *idx, float *lg,
                        uint32_t *err, cudaStream_t s) {
    if (R == 0) return cudaSuccess;
    const int KP = pow2_at_least(k);
    cudaError_t e;
    if (KP <= 128 && R >= 8192) {
        const size_t pw = topk_warp_smem(C, k);
        int W = (int)((200 * 1024) / pw);  // rows (warps) per CTA
        W = W < 1 ? 1 : (W > 8 ? 8 : W);
        const size_t smem = pw * (size_t)W;
        e = cudaFuncSetAttribute(topk_warp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        topk_warp_kernel<<<(unsigned)((R + W - 1) / W), 32 * W, smem, s>>>(L, R, C, k, KP, idx, lg,
                                                                           err);
        return cudaGetLastError();
    }
    const size_t smem = (size_t)KP * 8 + (size_t)C * 4;
    e = cudaFuncSetAttribute(topk_cta_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    topk_cta_kernel<<<(unsigned)R, kSelThreads, smem, s>>>(L, C, k, KP, idx, lg, err);
    return cudaGetLastError();
}

cudaError_t launch_coverage(const float *L, int R, int C, double eps, float *loss, float *u,
                            float *grad, unsigned char *ws, cudaStream_t s) {
    const int chunks = (R + kRowChunk - 1) / kRowChunk;
    float2 *stat = reinterpret_cast<float2 *>(ws + align_up(16, 256));
    double *ud = reinterpret_cast<double *>(ws + align_up(16, 256) + align_up((size_t)R * 8, 256));
    float *g = reinterpret_cast<float *>(ws + align_up(16, 256) + align_up((size_t)R * 8, 256) +
                                         align_up((size_t)chunks * C * 8, 256));
    cov_rows_kernel<<<R, kTrainThreads, 0, s>>>(L, C, stat);
    cov_cols_kernel<<<dim3((C + 255) / 256, chunks), 256, 0, s>>>(L, R, C, stat, ud);
    cov_usage_kernel<<<(C + 255) / 256, 256, 0, s>>>(ud, R, C, chunks);
    cov_loss_kernel<<<1, kTrainThreads, 0, s>>>(ud, C, eps, loss, u, grad ? g : nullptr);
    if (grad) cov_grad_kernel<<<R, kTrainThreads, 0, s>>>(L, R, C, stat, g, grad);
    return cudaGetLastError();
}

}  // namespace moce
