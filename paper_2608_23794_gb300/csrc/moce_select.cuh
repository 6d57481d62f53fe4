// Selection of the k smallest 32-bit order keys of a row by one warp
// (Eq. (support), Sec. 3.2: TopK in deployment order). Shared by the TopK
// kernels and the input-conditioned route.
#pragma once

#include "moce_internal.cuh"

namespace moce {

// Order key of a logit: larger logit -> smaller key; -0.0 and +0.0 equal.
__device__ __forceinline__ uint32_t desc_key(float v) {
    uint32_t b = __float_as_uint(v == 0.f ? 0.f : v);
    b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);  // increasing with v
    return ~b;
}

// key[0..C): the row's order keys (shared memory of the calling warp);
// hist: 256 words of its shared memory; sel: KP = k rounded up to a power of
// two 64-bit slots. On return sel[0..k) holds (key << 32) | channel of the k
// selected channels in ascending order (descending logit, equal logits by
// ascending channel). Four 8-bit radix passes (a histogram and a warp scan)
// find T, the k-th smallest key, and how many of the keys equal to T belong
// (the lowest channels); an ordered compaction by ballots collects the k; a
// bitonic sort of the KP slots (padding sorts last) orders them. The whole
// warp calls it; it synchronises the warp only.
__device__ __forceinline__ void warp_select(const uint32_t *key, int C, int k, int KP,
                                            uint32_t *hist, unsigned long long *sel) {
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < KP; i += 32) sel[i] = ~0ull;
    __syncwarp();
    uint32_t prefix = 0u, mask = 0u, kk = (uint32_t)k;  // kk: rank sought among the prefix's keys
    for (int shift = 24; shift >= 0; shift -= 8) {
#pragma unroll
        for (int b = 0; b < 8; ++b) hist[lane * 8 + b] = 0u;
        __syncwarp();
        for (int c = lane; c < C; c += 32) {
            const uint32_t kc = key[c];
            if ((kc & mask) == prefix) atomicAdd(hist + ((kc >> shift) & 255u), 1u);
        }
        __syncwarp();
        uint32_t hb[8], own = 0u;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            hb[b] = hist[lane * 8 + b];
            own += hb[b];
        }
        uint32_t incl = own;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        uint32_t run = incl - own, found = 0u, fb = 0u, fk = 0u;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            if (!found && run < kk && kk <= run + hb[b]) {
                found = 1u;
                fb = (uint32_t)(lane * 8 + b);
                fk = kk - run;
            }
            run += hb[b];
        }
        const int src = __ffs(__ballot_sync(0xffffffffu, found != 0u)) - 1;
        fb = __shfl_sync(0xffffffffu, fb, src);
        fk = __shfl_sync(0xffffffffu, fk, src);
        prefix |= fb << shift;
        kk = fk;
        mask |= 0xffu << shift;
        __syncwarp();
    }
    // prefix = T; the k - kk keys below T all belong, then the first kk equal to T
    const uint32_t T = prefix, nless = (uint32_t)k - kk, lt = (1u << lane) - 1u;
    uint32_t run_l = 0u, run_e = 0u;
    for (int j0 = 0; j0 < C; j0 += 32) {
        const int c = j0 + lane;
        const uint32_t kc = c < C ? key[c] : 0xffffffffu;
        const bool isl = c < C && kc < T, ise = c < C && kc == T;
        const uint32_t bl = __ballot_sync(0xffffffffu, isl), be = __ballot_sync(0xffffffffu, ise);
        const unsigned long long k64 = ((unsigned long long)kc << 32) | (uint32_t)c;
        if (isl) sel[run_l + __popc(bl & lt)] = k64;
        if (ise) {
            const uint32_t r = run_e + __popc(be & lt);
            if (r < kk) sel[nless + r] = k64;
        }
        run_l += __popc(bl);
        run_e += __popc(be);
    }
    __syncwarp();
    // bitonic sort of the KP pairs, ascending keys (padding sorts last)
    for (int size = 2; size <= KP; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = lane; i < KP / 2; i += 32) {
                const int lo = 2 * i - (i & (stride - 1));  // pair (lo, lo + stride)
                const int hi = lo + stride;
                const bool up = (lo & size) == 0;
                const unsigned long long a = sel[lo], b = sel[hi];
                if ((a > b) == up) {
                    sel[lo] = b;
                    sel[hi] = a;
                }
            }
            __syncwarp();
        }
    }
}

}  // namespace moce
