// Standalone temperature-gate kernels (Eq. (tau), Eq. (weights)).
//
// gate_kernel: one CTA per (block of GE experts, example); the arithmetic
// lives in moce_gate_block.cuh (any k).
//
// gate_tiled_kernel (k a multiple of 16): the hidden layer of the gate of
// every expert of one example is the product H = U W1^T (U [R][k]: row e =
// z[n, S_e] in deployment order; W1 [k][k], shared by every expert), a dense
// contraction. One CTA of 256 threads takes 64 experts: z of the example is
// staged once; then, in chunks of KC = 32 inputs, the chunk's support
// indices, its rows of U^T [KC][64] (gathered from z) and of W1^T [KC][k]
// pass through shared memory (about 42 KB at k = 128, so several CTAs share
// an SM), and thread (te, th) accumulates experts 4 te .. 4 te + 3 times
// hidden units TN th .. TN th + TN - 1 (TN = k / 16) in registers, over the
// inputs in order (fma.rn.f32x2 on pairs of hidden units). Each expert's 16
// partial sums w2 . ReLU(h + b1) are added by shuffles in a fixed order; then
// tau and the softmax weights as in moce_gate_block.cuh.
#include "moce_gate_block.cuh"

namespace moce {
namespace {

__global__ void __launch_bounds__(kThreads) gate_kernel(
    const float *__restrict__ z, int C, int R, int k, const int32_t *__restrict__ pidx,
    const float *__restrict__ plog, const float *__restrict__ W1, const float *__restrict__ b1,
    const float *__restrict__ w2, const float *__restrict__ b2, float tmin, float tmax,
    float *__restrict__ tau, float *__restrict__ a, size_t sup_stride) {
    extern __shared__ __align__(16) float gsm[];
    const size_t so = (size_t)blockIdx.y * sup_stride;  // per-example supports (0: shared)
    gate_block(gsm, blockIdx.y, blockIdx.x * GE, z, C, R, k, pidx + so, plog + so, W1, b1, w2, b2,
               tmin, tmax, tau, a);
}

constexpr int kTE = 64;        // experts per tiled-gate CTA
constexpr int kUS = kTE + 4;   // padded row of U^T (float4-aligned, rows 4 banks apart)

constexpr int kKC = 32;        // inputs per chunk of the tiled gate

// Floats of the tiled gate's shared memory: U^T and W1^T chunks, tau, the
// chunk's index rows (KC + 1 apart: the gather reads them without bank
// conflicts) and z of the example.
__host__ __device__ inline size_t tiled_smem(int k, int C) {
    return ((size_t)kKC * kUS + (size_t)kKC * k + kTE + (size_t)kTE * (kKC + 1) + (size_t)C) *
           sizeof(float);
}

template <int TN>
__global__ void __launch_bounds__(256) gate_tiled_kernel(
    const float *__restrict__ z, int C, int R, const int32_t *__restrict__ pidx,
    const float *__restrict__ plog, const float *__restrict__ W1, const float *__restrict__ b1,
    const float *__restrict__ w2, const float *__restrict__ b2, float tmin, float tmax,
    float *__restrict__ tau, float *__restrict__ a, size_t sup_stride) {
    constexpr int k = 16 * TN;
    pidx += (size_t)blockIdx.y * sup_stride;  // per-example supports (0: shared)
    plog += (size_t)blockIdx.y * sup_stride;
    extern __shared__ __align__(16) float tsm[];
    float *Ut = tsm;                                   // [KC][kUS]: Ut[i][el] = z[n, S_(e0+el)][i0+i]
    float *Wt = Ut + (size_t)kKC * kUS;                // [KC][k]: Wt[i][j] = W1[j][i0 + i]
    float *tau_s = Wt + (size_t)kKC * k;               // [kTE]
    int32_t *is = reinterpret_cast<int32_t *>(tau_s + kTE);  // [kTE][KC + 1]
    float *zs = reinterpret_cast<float *>(is + kTE * (kKC + 1));  // [C]
    const int n = blockIdx.y, e0 = blockIdx.x * kTE;
    const int tid = threadIdx.x, te = tid >> 4, th = tid & 15;
    const int ne = min(kTE, R - e0);
    {
        const float *zn = z + (size_t)n * C;
        for (int c = tid; c < C; c += 256) zs[c] = __ldcg(zn + c);
    }
    // thread th's hidden units, in pairs: pair p < 2 (TN / 4) is units
    // 64 (p / 2) + 4 th + 2 (p mod 2) + {0, 1}; a last pair (TN mod 4 = 2) is
    // units 64 (TN / 4) + 2 th + {0, 1}. Sixteen threads then read 256
    // consecutive bytes of a W^T row per float4, without bank conflicts.
    constexpr int NP = TN / 2, NQ = TN / 4;
    auto unit = [&](int p, int h) {
        return p < 2 * NQ ? 64 * (p >> 1) + 4 * th + 2 * (p & 1) + h : 64 * NQ + 2 * th + h;
    };
    float2 acc[4][NP];
#pragma unroll
    for (int m = 0; m < 4; ++m)
#pragma unroll
        for (int p = 0; p < NP; ++p) acc[m][p] = make_float2(0.f, 0.f);
    for (int i0 = 0; i0 < k; i0 += kKC) {
        const int kc = min(kKC, k - i0);
        __syncthreads();  // z staged / the previous chunk consumed
        // the chunk's support indices (consecutive threads on consecutive
        // inputs of an expert: coalesced loads, conflict-free stores)
        for (int q = tid; q < ne * kc; q += 256) {
            const int el = q / kc, i = q - el * kc;
            is[el * (kKC + 1) + i] = __ldg(pidx + (size_t)(e0 + el) * k + i0 + i);
        }
        // Wt[i][j] = W1[j][i0 + i]: a thread reads 4 inputs of one hidden unit
#pragma unroll 4
        for (int q = tid; q < k * (kc >> 2); q += 256) {
            const int j = q % k, i4 = q / k;
            const float4 w = __ldg(reinterpret_cast<const float4 *>(W1 + (size_t)j * k + i0) + i4);
            Wt[(4 * i4 + 0) * k + j] = w.x;
            Wt[(4 * i4 + 1) * k + j] = w.y;
            Wt[(4 * i4 + 2) * k + j] = w.z;
            Wt[(4 * i4 + 3) * k + j] = w.w;
        }
        __syncthreads();
        // U^T rows of the chunk, consecutive threads on consecutive experts
        // (conflict-free stores); experts past R read as zero
        for (int q = tid; q < kTE * kc; q += 256) {
            const int el = q & (kTE - 1), i = q / kTE;
            Ut[i * kUS + el] = el < ne ? zs[is[el * (kKC + 1) + i]] : 0.f;
        }
        __syncthreads();
#pragma unroll 2
        for (int i = 0; i < kc; ++i) {
            const float4 u = *reinterpret_cast<const float4 *>(Ut + (size_t)i * kUS + 4 * te);
            const float *wr = Wt + (size_t)i * k;
            float2 w[NP];
#pragma unroll
            for (int r = 0; r < NQ; ++r) {
                const float4 v = *reinterpret_cast<const float4 *>(wr + 64 * r + 4 * th);
                w[2 * r] = make_float2(v.x, v.y);
                w[2 * r + 1] = make_float2(v.z, v.w);
            }
            if constexpr (NP > 2 * NQ) w[NP - 1] = *reinterpret_cast<const float2 *>(wr + 64 * NQ + 2 * th);
            const float2 u0 = make_float2(u.x, u.x), u1 = make_float2(u.y, u.y),
                         u2 = make_float2(u.z, u.z), u3 = make_float2(u.w, u.w);
#pragma unroll
            for (int p = 0; p < NP; ++p) {
                acc[0][p] = __ffma2_rn(u0, w[p], acc[0][p]);
                acc[1][p] = __ffma2_rn(u1, w[p], acc[1][p]);
                acc[2][p] = __ffma2_rn(u2, w[p], acc[2][p]);
                acc[3][p] = __ffma2_rn(u3, w[p], acc[3][p]);
            }
        }
    }
    // g = w2 . ReLU(h + b1) + b2: this thread's hidden units, then the 16
    // threads of the expert group (consecutive lanes) in a fixed order
    float gp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int p = 0; p < NP; ++p) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int jj = unit(p, h);
            const float bj = __ldg(b1 + jj), wj = __ldg(w2 + jj);
#pragma unroll
            for (int m = 0; m < 4; ++m)
                gp[m] = fmaf(wj, fmaxf((h ? acc[m][p].y : acc[m][p].x) + bj, 0.f), gp[m]);
        }
    }
#pragma unroll
    for (int m = 0; m < 4; ++m) {
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) gp[m] += __shfl_xor_sync(0xffffffffu, gp[m], o);
    }
    if (th == 0) {
        const float bb = __ldg(b2);
#pragma unroll
        for (int m = 0; m < 4; ++m) {
            const int el = 4 * te + m, e = e0 + el;
            const float t = tmin + (tmax - tmin) / (1.f + expf(-(gp[m] + bb)));
            tau_s[el] = t;
            if (e < R) tau[(size_t)n * R + e] = t;
        }
    }
    if (a == nullptr) return;
    __syncthreads();
    // a[n, e, i] = exp((L_i - L_max) / tau) / sum_j exp((L_j - L_max) / tau), a
    // warp per expert, the lane's k / 32 logits loaded at once
    constexpr int LK = (k + 31) / 32;
    const int warp = tid >> 5, lane = tid & 31;
    for (int el = warp; el < kTE; el += 8) {
        const int e = e0 + el;
        if (e >= R) break;
        const float t = tau_s[el];
        const float *L = plog + (size_t)e * k;
        float lv[LK];
#pragma unroll
        for (int r = 0; r < LK; ++r) lv[r] = lane + 32 * r < k ? __ldg(L + lane + 32 * r) : -INFINITY;
        float m = lv[0];
#pragma unroll
        for (int r = 1; r < LK; ++r) m = fmaxf(m, lv[r]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        float s = 0.f;
#pragma unroll
        for (int r = 0; r < LK; ++r) {
            lv[r] = lane + 32 * r < k ? expf((lv[r] - m) / t) : 0.f;
            s += lv[r];
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        float *ae = a + ((size_t)n * R + e) * k;
#pragma unroll
        for (int r = 0; r < LK; ++r)
            if (lane + 32 * r < k) ae[lane + 32 * r] = lv[r] / s;
    }
}

template <int TN>
cudaError_t launch_tiled_gate(const float *z, int N, int C, int R, const int32_t *pidx,
                              const float *plog, const float *W1, const float *b1,
                              const float *w2, const float *b2, float tmin, float tmax,
                              float *tau, float *a, size_t ss, cudaStream_t s) {
    constexpr int k = 16 * TN;
    const size_t smem = tiled_smem(k, C);
    cudaError_t err = cudaFuncSetAttribute(gate_tiled_kernel<TN>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    const dim3 grid((R + kTE - 1) / kTE, N);
    gate_tiled_kernel<TN><<<grid, 256, smem, s>>>(z, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax,
                                                  tau, a, ss);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gate(const float *z, int N, int C, int R, int k, const int32_t *pidx,
                        const float *plog, const float *W1, const float *b1, const float *w2,
                        const float *b2, float tmin, float tmax, float *tau, float *a,
                        cudaStream_t s, size_t ss) {
    if (N == 0) return cudaSuccess;
    // the tiled kernel reads W1 rows as float4
    const bool w1v = (reinterpret_cast<uintptr_t>(W1) & 15u) == 0 &&
                     (reinterpret_cast<uintptr_t>(pidx) & 15u) == 0 && ss % 4 == 0;
    if (w1v && k >= 32 && tiled_smem(k, C) <= 227 * 1024) {
        switch (k) {
        case 32: return launch_tiled_gate<2>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 64: return launch_tiled_gate<4>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 96: return launch_tiled_gate<6>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 128: return launch_tiled_gate<8>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 192: return launch_tiled_gate<12>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 256: return launch_tiled_gate<16>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        case 384: return launch_tiled_gate<24>(z, N, C, R, pidx, plog, W1, b1, w2, b2, tmin, tmax, tau, a, ss, s);
        default: break;
        }
    }
    const size_t smem = gate_smem(k);
    if (smem > 48 * 1024) {
        cudaError_t err =
            cudaFuncSetAttribute(gate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
    }
    const dim3 grid((R + GE - 1) / GE, N);
    gate_kernel<<<grid, kThreads, smem, s>>>(z, C, R, k, pidx, plog, W1, b1, w2, b2, tmin, tmax,
                                             tau, a, ss);
    return cudaGetLastError();
}

size_t gate_smem_bytes(int k) { return gate_smem(k); }

}  // namespace moce
