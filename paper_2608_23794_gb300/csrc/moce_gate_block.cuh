// Temperature gate, Eq. (tau), and mixing weights, Eq. (weights), for one
// block of experts of one example, for the standalone gate kernel (any k).
//
// For each (example n, routed expert e) the gate input is u = z[n, S_e] in
// deployment order (position i = the expert's i-th most preferred channel,
// Sec. 3.3). The shared gate g(u) = w2 . ReLU(W1 u + b1) + b2 (two-layer MLP
// of hidden width k, Sec. 4.1) is evaluated for a block of GE experts at once
// as a small batched product H = U W1^T: U [GE x k] is gathered into shared
// memory, W1 streams through shared memory in chunks of HJ hidden units, and
// each thread accumulates 4 hidden units of one expert in registers. Then
// tau = tau_min + (tau_max - tau_min) * sigma(g) and, if requested,
// a[n,e,i] = exp((L_i - L_max)/tau) / sum_j exp((L_j - L_max)/tau).
// All sums run in a fixed order (deterministic).
#pragma once

#include "moce_internal.cuh"

namespace moce {

constexpr int GE = 32;  // experts per gate block
constexpr int HJ = 32;  // hidden units per W1 chunk
constexpr int HJS = HJ + 4;  // padded row of the transposed W1 chunk (keeps float4 alignment)

__host__ __device__ inline int gate_ks(int k) { return (k % 2 == 0) ? k + 1 : k; }

__host__ __device__ inline size_t gate_smem(int k) {
    return ((size_t)GE * gate_ks(k) + (size_t)k * HJS + GE) * sizeof(float);
}

// One block of GE experts of example n: 256 threads = GE experts x 8 threads
// (4 hidden units each). gsm: gate_smem(k) bytes of shared memory.
__device__ __forceinline__ void gate_block(float *gsm, int n, int e0, const float *__restrict__ z,
                                           int C, int R, int k, const int32_t *__restrict__ pidx,
                                           const float *__restrict__ plog,
                                           const float *__restrict__ W1,
                                           const float *__restrict__ b1,
                                           const float *__restrict__ w2,
                                           const float *__restrict__ b2, float tmin, float tmax,
                                           float *__restrict__ tau, float *__restrict__ a) {
    const int ks = gate_ks(k);
    float *U = gsm;                        // [GE][ks]
    float *Wt = U + (size_t)GE * ks;       // [k][HJS]
    float *tau_s = Wt + (size_t)k * HJS;   // [GE]
    const int tid = threadIdx.x, te = tid >> 3, jq = tid & 7;
    const float *zn = z + (size_t)n * C;

    for (int q = tid; q < GE * k; q += kThreads) {
        const int el = q / k, i = q - el * k, e = e0 + el;
        U[el * ks + i] = (e < R) ? __ldcg(zn + __ldg(pidx + (size_t)e * k + i)) : 0.f;
    }
    float gacc = 0.f;
    for (int j0 = 0; j0 < k; j0 += HJ) {
        __syncthreads();  // U ready / previous chunk consumed
        for (int q = tid; q < HJ * k; q += kThreads) {
            const int jj = q / k, i = q - jj * k, j = j0 + jj;
            Wt[i * HJS + jj] = (j < k) ? __ldg(W1 + (size_t)j * k + i) : 0.f;
        }
        __syncthreads();
        float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
        const float *ur = U + te * ks;
        const float *wc = Wt + jq * 4;
#pragma unroll 4
        for (int i = 0; i < k; ++i) {
            const float u = ur[i];
            const float4 w = *reinterpret_cast<const float4 *>(wc + i * HJS);
            acc0 = fmaf(u, w.x, acc0);
            acc1 = fmaf(u, w.y, acc1);
            acc2 = fmaf(u, w.z, acc2);
            acc3 = fmaf(u, w.w, acc3);
        }
        const int j = j0 + jq * 4;
        if (j + 0 < k) gacc = fmaf(__ldg(w2 + j + 0), fmaxf(acc0 + __ldg(b1 + j + 0), 0.f), gacc);
        if (j + 1 < k) gacc = fmaf(__ldg(w2 + j + 1), fmaxf(acc1 + __ldg(b1 + j + 1), 0.f), gacc);
        if (j + 2 < k) gacc = fmaf(__ldg(w2 + j + 2), fmaxf(acc2 + __ldg(b1 + j + 2), 0.f), gacc);
        if (j + 3 < k) gacc = fmaf(__ldg(w2 + j + 3), fmaxf(acc3 + __ldg(b1 + j + 3), 0.f), gacc);
    }
    // the 8 threads of an expert are consecutive lanes: fixed-order tree
    gacc += __shfl_xor_sync(0xffffffffu, gacc, 4);
    gacc += __shfl_xor_sync(0xffffffffu, gacc, 2);
    gacc += __shfl_xor_sync(0xffffffffu, gacc, 1);
    const int e = e0 + te;
    if (jq == 0) {
        const float g = gacc + __ldg(b2);
        const float t = tmin + (tmax - tmin) / (1.f + expf(-g));
        tau_s[te] = t;
        if (e < R) tau[(size_t)n * R + e] = t;
    }
    if (a == nullptr) return;
    __syncthreads();
    const int warp = tid >> 5, lane = tid & 31;
    for (int el = warp; el < GE; el += kThreads / 32) {
        const int ee = e0 + el;
        if (ee >= R) break;
        const float t = tau_s[el];
        const float *L = plog + (size_t)ee * k;
        float m = -INFINITY;
        for (int i = lane; i < k; i += 32) m = fmaxf(m, __ldg(L + i));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        float s = 0.f;
        for (int i = lane; i < k; i += 32) s += expf((__ldg(L + i) - m) / t);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        float *ae = a + ((size_t)n * R + ee) * k;
        for (int i = lane; i < k; i += 32) ae[i] = expf((__ldg(L + i) - m) / t) / s;
    }
}


}  // namespace moce
