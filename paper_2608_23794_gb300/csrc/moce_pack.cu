// Deployment packing of static supports (Sec. 3.2, Sec. 3.3 ordering rule,
// Sec. 3.4 residual set U, Sec. 3.5 "Storage").
//
// pack_rows_kernel: one CTA per expert. Entry j of the row goes to position
//   rank(j) = #{m : L_m > L_j, or L_m == L_j and c_m < c_j},
// which sorts the row by descending logit with ties by ascending channel.
// Because channels within a valid row are distinct, the ranks are a
// permutation and the output does not depend on the input order. The kernel
// also validates the row and marks the selected channels in a bitmap.
// pack_resid_kernel: one CTA lists the unmarked channels in ascending order.
#include "moce_internal.cuh"

namespace moce {
namespace {

constexpr uint32_t kBadRange = 1u, kBadDup = 2u, kBadLogit = 4u;

// ws words: [0] error bits, [1] |U|, [2..] coverage bitmap (ceil(C/32) words)
__global__ void __launch_bounds__(128) pack_rows_kernel(int C, int k, const int32_t *__restrict__ idx,
                                                        const float *__restrict__ lg,
                                                        int32_t *__restrict__ pidx,
                                                        float *__restrict__ plog,
                                                        uint32_t *__restrict__ words) {
    const int e = blockIdx.x;
    const int32_t *ri = idx + (size_t)e * k;
    const float *rl = lg + (size_t)e * k;
    uint32_t *covered = words + 2;
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        const int cj = __ldg(ri + j);
        const float lj = __ldg(rl + j);
        uint32_t bad = 0;
        if (cj < 0 || cj >= C) bad |= kBadRange;
        if (!isfinite(lj)) bad |= kBadLogit;
        int rank = 0;
        for (int m = 0; m < k; ++m) {
            const int cm = __ldg(ri + m);
            const float lm = __ldg(rl + m);
            if (m != j && cm == cj) bad |= kBadDup;
            rank += (lm > lj) || (lm == lj && cm < cj);
        }
        if (bad) {
            atomicOr(words, bad);
        } else if (rank < k) {
            pidx[(size_t)e * k + rank] = cj;
            plog[(size_t)e * k + rank] = lj;
            atomicOr(covered + (cj >> 5), 1u << (cj & 31));
        }
    }
}

__global__ void __launch_bounds__(1024) pack_resid_kernel(int C, uint32_t *__restrict__ words,
                                                          int32_t *__restrict__ resid) {
    __shared__ int warp_tot[32];
    const uint32_t *covered = words + 2;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int base = 0;
    for (int c0 = 0; c0 < C; c0 += 1024) {
        const int c = c0 + (int)threadIdx.x;
        const bool flag = c < C && !((covered[c >> 5] >> (c & 31)) & 1u);
        const uint32_t bal = __ballot_sync(0xffffffffu, flag);
        if (lane == 0) warp_tot[warp] = __popc(bal);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < 32; ++w) {
            const int t = warp_tot[w];
            before += (w < warp) ? t : 0;
            total += t;
        }
        if (flag) resid[base + before + __popc(bal & ((1u << lane) - 1u))] = c;
        base += total;
        __syncthreads();
    }
    if (threadIdx.x == 0) words[1] = (uint32_t)base;
}

}  // namespace

cudaError_t launch_pack(int C, int R, int k, const int32_t *idx, const float *lg, int32_t *pidx,
                        float *plog, int32_t *resid, uint32_t *ws_words, cudaStream_t s) {
    const size_t nwords = 2 + (size_t)(C + 31) / 32;
    cudaError_t err = cudaMemsetAsync(ws_words, 0, nwords * 4, s);
    if (err != cudaSuccess) return err;
    pack_rows_kernel<<<R, 128, 0, s>>>(C, k, idx, lg, pidx, plog, ws_words);
    pack_resid_kernel<<<1, 1024, 0, s>>>(C, ws_words, resid);
    return cudaGetLastError();
}

}  // namespace moce
