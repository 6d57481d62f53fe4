// Single-pass streaming forward of a MoCE layer (Sec. 3.3-3.4) for NHWC bf16
// layers with 64 <= C_in <= 256, C_in % 64 == 0, C_out <= 64, k <= 16 and at
// most 255 tiles of 64 positions per example: x is read from HBM once.
//
// Every expert's temperature needs the whole-image pool of its example
// (Sec. 3.3, Eq. (tau)), so no position can be mixed before its example has
// been pooled. Here a tile stays in shared memory from the moment it is
// pooled until its example's gate has run, and is mixed from there.
//
// Work: tiles of 64 positions of one example (tile t of example n is item
// it = n T + t, T = ceil(HW / 64)); CTA b of G (one per SM, cooperative
// launch) takes items b, b + G, ... through a ring of D shared-memory slots.
// Roles (640 threads):
//   producer (warp 16)   : one TMA tensor load per 64-channel group of the
//                          tile ([64 positions][64 channels], 128-byte
//                          swizzle) into slot j mod D;
//   transpose (0-3)      : warp g owns channel group g of the slot and, on
//                          its own (no barrier with the other warps): reads
//                          it with ldmatrix.trans, adds the tile's channel
//                          sums (the pool, Sec. 3.3), writes the words back
//                          in place as channel-major rows (row c = the
//                          tile's 64 positions of channel c, bf16 pairs) and
//                          signals the slot;
//   publish (18)         : adds the tile's channel sums to the example's
//                          accumulator words by one bulk reduction;
//   residual (19)        : sums the unselected channels of every position
//                          (Eq. (res));
//   gate (4-7)           : for every example whose last tile this CTA
//                          holds, wait (bounded) until every accumulator
//                          word of the example counts all T tiles, decode z,
//                          run the gate of every expert (Eq. (tau)) and the
//                          softmax weights (Eq. (weights)), publish them with
//                          a tag. These warps wait for nothing else (no slot,
//                          no other gate), so no chain of waits passes
//                          through a gate;
//   mix (8-15)           : each 8-lane group owns one expert pair with their
//                          row offsets and weights in registers; a lane reads
//                          one 16-byte chunk (8 positions) of a support row
//                          and adds it with fma.rn.f32x2 (Eq. (expert)); y
//                          with the residual column is staged in shared
//                          memory; the mix warps synchronise only through
//                          mbarriers, never with a CTA barrier;
//   table + store (17)   : brings the weights of item j's example (waiting,
//                          bounded, for its tag) into one of two tables;
//                          each staged y tile leaves by one bulk copy.
// Accumulator word of (example, channel): bits 56-63 count the tiles added,
// bits 48-55 the tiles whose sum was kept as a tagged fp32 word instead,
// bits 0-47 the sum of 2^39 + round(2^20 s) over the other tiles (s = the
// tile's channel sum, |s| < 2^19). Integer sums do not depend on the order of
// the additions, so z is deterministic, and the count in the same word makes
// a fence between the sum and the count unnecessary. Forward e uses bank
// e mod 2 of the words and clears the other bank, which the previous forward
// used and the next one will.
// Every wait is bounded (MOCE_ERR_TIMEOUT); none traps.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kTP = 64;             // positions per tile
constexpr int kThreads_ = 640;
// Warps are ordered by how short their critical path is: the transpose and
// gate warps come first (the scheduler favours older warps when several are
// ready, and the mix warps, with many independent loads in flight, are
// nearly always ready), the mix warps after them.
constexpr int kTr0 = 0;             // warps 0-3
constexpr int kGate0 = 128;         // warps 4-7
constexpr int kMix0 = 256;          // warps 8-15
constexpr int kMixT = 256;
constexpr int kProdW = 16;          // warp 17: y stores; 18: pool words; 19: residual
constexpr int kStoreW = 17;
constexpr int kPubW = 18;
constexpr int kResW = 19;
constexpr int kMaxD = 6;            // x slots at most
constexpr int kNT = 2;              // weight tables
constexpr int kKMax = 16;
constexpr int kRMax = 64;
constexpr int kMaxT = 255;          // tiles per example (8-bit count field)
constexpr int kBarGate = 3;
// mbarriers: raw (TMA landed), staged (transposed), empty (mixed), tready /
// tfree (gate -> mix tables), ydone / yfree (mix -> store staging buffers)
constexpr int kMbRaw = 0, kMbStaged = kMaxD, kMbEmpty = 2 * kMaxD, kMbTReady = 3 * kMaxD,
              kMbTFree = 3 * kMaxD + kNT, kMbYDone = 3 * kMaxD + 2 * kNT,
              kMbYFree = 3 * kMaxD + 2 * kNT + 1, kMbPooled = 3 * kMaxD + 2 * kNT + 2,
              kMbPFree = 3 * kMaxD + 2 * kNT + 4, kMbResDone = 3 * kMaxD + 2 * kNT + 6,
              kMbCount = 4 * kMaxD + 2 * kNT + 6;
// registers: 96 per thread at launch; mix 136, transpose 104, gate 56, the rest 48
// (setmaxnreg.inc waits for registers the other warpgroups release: the
// shares must add up to no more than the launch allocation)
constexpr int kRegLaunch = 96, kRegMix = 136, kRegTr = 104, kRegGate = 56, kRegMisc = 48;
static_assert(2 * 128 * kRegMix + 128 * kRegTr + 128 * kRegGate + 128 * kRegMisc <=
                  kThreads_ * kRegLaunch,
              "register split exceeds the launch allocation");

constexpr float kFixScale = 1048576.0f;  // 2^20
constexpr float kFixMax = 524288.0f;     // 2^19
constexpr unsigned long long kFixBias = 1ull << 39;
constexpr unsigned long long kWideOne = 1ull << 48;
constexpr unsigned long long kTileOne = 1ull << 56;

// round(2^20 s) for |s| < 2^19 from two 32-bit conversions (no 64-bit
// float conversion): hi = round(16 s), then the remainder s - hi / 16
// (exact in fp32: |s| < 2^20 makes it a multiple of ulp(s), below 1/32) at
// 2^-20 resolution; hi 2^16 + lo is within one unit of 2^20 s.
__device__ __forceinline__ long long fix20(float v) {
    const int hi = __float2int_rn(v * 16.f);
    const int lo = __float2int_rn(fmaf((float)hi, -0.0625f, v) * kFixScale);
    return ((long long)hi << 16) + lo;
}
// fx 2^-20 as fp32 from two 32-bit conversions: the integer part and the
// 20-bit fraction.
__device__ __forceinline__ float unfix20(long long fx) {
    return (float)(int)(fx >> 20) + (float)(int)(fx & 0xfffffll) * (1.0f / kFixScale);
}

struct StreamParams {
    uint16_t *y;
    int N, HW, C, R, k, nU, T, nreg, G, D;
    uint32_t items;
    const int32_t *pidx;
    const float *plog;
    const int32_t *resid;
    const float *W1, *b1, *w2, *b2;
    float tmin, tmax, inv_HW, inv_nU;
    uint32_t *ctrl;
    unsigned long long *zacc;   // [2][N][C] accumulator words, bank = epoch mod 2
    unsigned long long *wide;   // [N][T][C] tagged fp32 tile sums beyond the fixed-point range
    uint32_t *flag;             // [N] tag of the forward whose gate wrote example n's weights
    float *wblk;                // [N][tb_bytes / 4] weight blocks (table layout)
    float *z, *tau;             // [N][C], [N][R]
    uint32_t tb_bytes;          // bytes of one weight table
    uint32_t ysb;               // bytes of one y staging buffer
    uint32_t off_x, off_tab, off_ys, off_res, off_U, off_zs, off_w1t, off_b1, off_w2, off_psum,
        off_pword, off_bar;
    uint32_t smem_bytes;
};

// Float offset of expert e's 16 weights in a table: experts 8 apart (the
// four lane groups of a mix warp) start 16 bytes apart mod 128, so the
// groups' reads of their weights hit different banks.
__host__ __device__ __forceinline__ int wofs(int e) { return 16 * e + 4 * (e >> 3); }
inline uint32_t table_bytes(int R) { return (uint32_t)stream_table_bytes(R); }

// ---------------------------------------------------------------- PTX helpers
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *tm, int x, int y,
                                            uint32_t mbar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(mbar), "l"(policy)
        : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t a, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a)
                 : "memory");
}
__device__ __forceinline__ void sts128(uint32_t a, const uint32_t (&r)[4]) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(r[0]), "r"(r[1]),
                 "r"(r[2]), "r"(r[3])
                 : "memory");
}
__device__ __forceinline__ uint4 lds128a(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(a)
                 : "memory");
    return v;
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void bulk_store(void *dst, uint32_t src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                 "r"(src), "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Bulk stores of this thread still reading shared memory: at most N groups.
template <int N> __device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// acc + lo, then + hi, for the two bf16 of a word (exact widening, fp32 add)
__device__ __forceinline__ float add_bf16x2(float acc, uint32_t w) {
    asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\t"
        "add.rn.f32.bf16 %0, lo, %0;\n\tadd.rn.f32.bf16 %0, hi, %0;\n\t}"
        : "+f"(acc)
        : "r"(w));
    return acc;
}
// acc.x + lo, acc.y + hi
__device__ __forceinline__ float2 add_bf16_pair(float2 acc, uint32_t w) {
    asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %2;\n\t"
        "add.rn.f32.bf16 %0, lo, %0;\n\tadd.rn.f32.bf16 %1, hi, %1;\n\t}"
        : "+f"(acc.x), "+f"(acc.y)
        : "r"(w));
    return acc;
}
// Bulk reduction (TMA engine, async proxy): dst[i] += src[i] for the u64
// words of a shared-memory buffer, each element added atomically.
__device__ __forceinline__ void bulk_reduce_add_u64(void *dst, uint32_t src, uint32_t bytes) {
    asm volatile(
        "cp.reduce.async.bulk.global.shared::cta.bulk_group.add.u64 [%0], [%1], %2;" ::"l"(dst),
        "r"(src), "r"(bytes)
        : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

struct Item {
    int n, t, valid;
    uint32_t it;
};
__device__ __forceinline__ Item item_of(const StreamParams &P, int j) {
    Item r;
    r.it = (uint32_t)blockIdx.x + (uint32_t)j * (uint32_t)P.G;
    r.n = (int)(r.it / (uint32_t)P.T);
    r.t = (int)(r.it - (uint32_t)r.n * (uint32_t)P.T);
    r.valid = min(kTP, P.HW - r.t * kTP);
    return r;
}
__device__ __forceinline__ int items_of_cta(const StreamParams &P) {
    const uint32_t b = blockIdx.x;
    return b < P.items ? (int)((P.items - 1u - b) / (uint32_t)P.G) + 1 : 0;
}
__device__ __forceinline__ float *res_of(const StreamParams &P, unsigned char *sm, int s) {
    return reinterpret_cast<float *>(sm + P.off_res) + s * kTP;
}

// ================================================================ roles

// Producer: one TMA tensor load per 64-channel group of each tile.
__device__ void role_producer(const StreamParams &P, const CUtensorMap *tm, unsigned char *sm) {
    if ((threadIdx.x & 31) != 0) return;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_x);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
    const int nj = items_of_cta(P);
    int issued = 0;
    for (int j = 0; j < nj; ++j) {
        const int s = j % P.D;
        if (j >= P.D &&
            !mbar_wait(bar + 8u * (kMbEmpty + s), (uint32_t)((j / P.D) - 1) & 1u, P.ctrl, 0u))
            break;
        const Item I = item_of(P, j);
        const int row = I.n * P.HW + I.t * kTP;
        const uint32_t full = bar + 8u * (kMbRaw + s);
        mbar_expect_tx(full, (uint32_t)P.nreg * 8192u);
        for (int g = 0; g < P.nreg; ++g)
            tma_load_2d(xs0 + (uint32_t)s * sb + 8192u * (uint32_t)g, tm, 64 * g, row, full, pol);
        ++issued;
    }
    // no copy may still be writing shared memory when the CTA exits
    for (int j = issued > P.D ? issued - P.D : 0; j < issued; ++j)
        mbar_wait(bar + 8u * (kMbRaw + j % P.D), (uint32_t)(j / P.D) & 1u, P.ctrl, 0u);
}

// Transpose + pool, warp g on channel group g alone. Region g of the slot
// (8 KB) holds [64 positions][64 channels] as the TMA wrote it (128-byte
// swizzle: 16-byte chunk c of row p at chunk c ^ (p & 7)). ldmatrix.trans of
// 8x8 blocks gives lane l (cl = l / 4, q = l mod 4) the words
// {x[p][c], x[p + 1][c]} for channel c = 8 jj + cl of the region and
// positions p = 32 h + 8 m + 2 q (m = 0..3 over the four matrices). The lane
// adds them to its channel sums (the pool, Sec. 3.3) and stores its four
// words as one 16-byte chunk at logical chunk 4 h + q of row c (physical
// chunk (4 h + q) ^ (4 (c & 1))): row c then holds the tile's 64 positions
// of channel c, word 16 h + 4 q + m holding positions 2 (16 h + 4 m + q) and
// the next. The channel sums go to the publish warp, the slot to the
// residual and mix warps: nothing else stands on this warp's path.
__device__ void role_transpose(const StreamParams &P, unsigned char *sm) {
    const int tt = threadIdx.x - kTr0;  // 0..127
    const int g = tt >> 5, lane = tt & 31;
    const int q = lane & 3, cl = lane >> 2;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_x);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    const bool own = g < P.nreg;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.D, pb = j & 1;
        bool ok = mbar_wait(bar + 8u * (kMbRaw + s), (uint32_t)(j / P.D) & 1u, P.ctrl, I.it);
        // the publish warp has read this sum buffer (item j - 2)
        ok = ok && (j < 2 || mbar_wait(bar + 8u * (kMbPFree + pb), (uint32_t)((j >> 1) - 1) & 1u,
                                       P.ctrl, I.it));
        if (!__all_sync(0xffffffffu, ok)) break;  // warp-uniform exit
        if (own) {
            const uint32_t rb = xs0 + (uint32_t)s * sb + 8192u * (uint32_t)g;
            uint32_t r[16][4];
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int jj = 0; jj < 8; ++jj)
                    ldsm_x4_t(rb + (uint32_t)(32 * h + lane) * 128u +
                                  ((uint32_t)(jj ^ (lane & 7)) << 4),
                              r[8 * h + jj]);
            float pacc[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) pacc[jj] = 0.f;
            // the tile's channel sums (positions beyond the example excluded)
            if (I.valid == kTP) {
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int m = 0; m < 4; ++m)
#pragma unroll
                        for (int jj = 0; jj < 8; ++jj)
                            pacc[jj] = add_bf16x2(pacc[jj], r[8 * h + jj][m]);
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        // keep position p (low half) and p + 1 (high half) when in the example
                        const int p = 32 * h + 8 * m + 2 * q;
                        const uint32_t keep = (p < I.valid ? 0x0000ffffu : 0u) |
                                              (p + 1 < I.valid ? 0xffff0000u : 0u);
#pragma unroll
                        for (int jj = 0; jj < 8; ++jj)
                            pacc[jj] = add_bf16x2(pacc[jj], r[8 * h + jj][m] & keep);
                    }
            }
            __syncwarp();
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) {
                    const int c = 8 * jj + cl;
                    sts128(rb + (uint32_t)c * 128u + ((uint32_t)((4 * h + q) ^ ((c & 1) << 2)) << 4),
                           r[8 * h + jj]);
                }
            // sums over the four position subsets (lanes q = 0..3), in a fixed order
            float *ps = reinterpret_cast<float *>(sm + P.off_psum) + pb * P.C + 64 * g;
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                float v = pacc[jj];
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                if ((jj & 3) == q) ps[8 * jj + cl] = v;
            }
            __syncwarp();
        }
        if (lane == 0) {
            mbar_arrive(bar + 8u * (kMbStaged + s));
            mbar_arrive(bar + 8u * (kMbPooled + pb));
        }
    }
}

// Publish: the tile's channel sums as accumulator words (fixed point, with
// the tile count) into a shared buffer, and from there into the example's
// words by one bulk reduction (TMA engine, each element added atomically).
__device__ void role_publish(const StreamParams &P, unsigned char *sm) {
    const int lane = threadIdx.x & 31;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    const uint32_t tag = ld_relaxed(P.ctrl + kCtrlEpoch) + 1u;
    unsigned long long *zb = P.zacc + (size_t)((tag - 1u) & 1u) * P.N * P.C;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int pb = j & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(bar + 8u * (kMbPooled + pb), (uint32_t)(j >> 1) & 1u,
                                                P.ctrl, I.it)))
            break;  // warp-uniform exit
        const float *ps = reinterpret_cast<const float *>(sm + P.off_psum) + pb * P.C;
        const uint32_t pw = smem_u32(sm + P.off_pword) + (uint32_t)pb * (uint32_t)P.C * 8u;
        if (lane == 0) bulk_wait_read<1>();  // the reduction of item j - 2 has read pw
        __syncwarp();
        for (int c = lane; c < P.C; c += 32) {
            const float v = ps[c];
            unsigned long long add;
            if (fabsf(v) < kFixMax) {
                add = kTileOne + kFixBias + (unsigned long long)fix20(v);
            } else {  // beyond the fixed-point range (or not finite)
                st_tagged(P.wide + ((size_t)I.n * P.T + I.t) * P.C + c, v, tag);
                add = kTileOne + kWideOne;
            }
            asm volatile("st.shared.u64 [%0], %1;" ::"r"(pw + 8u * (uint32_t)c), "l"(add) : "memory");
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(bar + 8u * (kMbPFree + pb));
            if (I.it + 1u != drop)  // fault injection: never counted
                bulk_reduce_add_u64(zb + (size_t)I.n * P.C, pw, (uint32_t)P.C * 8u);
        }
    }
    if (lane == 0) bulk_wait_all();  // the last reductions are complete
}

// Residual expert (Eq. (res)): the mean of the unselected channels at each
// position of the transposed tile; lane (part = lane / 8, chunk jc = lane
// mod 8) adds U entries part, part + 4, ... over its chunk's 8 positions,
// then the four parts are added in a fixed order.
__device__ void role_residual(const StreamParams &P, unsigned char *sm) {
    const int lane = threadIdx.x & 31;
    const int jc = lane & 7, part = lane >> 3;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_x);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    const uint16_t *Us = reinterpret_cast<const uint16_t *>(sm + P.off_U);
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.D;
        if (!__all_sync(0xffffffffu, mbar_wait(bar + 8u * (kMbStaged + s), (uint32_t)(j / P.D) & 1u,
                                                P.ctrl, I.it)))
            break;  // warp-uniform exit
        const uint32_t xs = xs0 + (uint32_t)s * sb;
        float2 ra[4];
#pragma unroll
        for (int m = 0; m < 4; ++m) ra[m] = make_float2(0.f, 0.f);
#pragma unroll 2
        for (int u = part; u < P.nU; u += 4) {
            const int c = Us[u];
            const uint4 v = lds128a(xs + (uint32_t)c * 128u + ((uint32_t)(jc ^ ((c & 1) << 2)) << 4));
            ra[0] = add_bf16_pair(ra[0], v.x);
            ra[1] = add_bf16_pair(ra[1], v.y);
            ra[2] = add_bf16_pair(ra[2], v.z);
            ra[3] = add_bf16_pair(ra[3], v.w);
        }
#pragma unroll
        for (int m = 0; m < 4; ++m) {
#pragma unroll
            for (int o = 8; o <= 16; o <<= 1) {
                ra[m].x += __shfl_xor_sync(0xffffffffu, ra[m].x, o);
                ra[m].y += __shfl_xor_sync(0xffffffffu, ra[m].y, o);
            }
        }
        if (lane < 8) {
            // positions 32 (jc / 4) + 8 m + 2 (jc mod 4) + {0, 1}
            float *rp = res_of(P, sm, s);
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const int p = 32 * (jc >> 2) + 8 * m + 2 * (jc & 3);
                rp[p] = ra[m].x * P.inv_nU;
                rp[p + 1] = ra[m].y * P.inv_nU;
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar + 8u * (kMbResDone + s));
    }
}

// Gate of every expert of example n (Eq. (tau)) and its softmax weights
// (Eq. (weights)) into the example's weight block in global memory, by the
// 128 threads of the gate role; thread (e = gt / 2, h = gt mod 2) holds
// hidden units 8 h .. 8 h + 7 and support positions 8 h .. 8 h + 7 of expert
// e. W1 is kept transposed and zero-padded to 16 x 16 (W1t[i][j] = W1[j][i]),
// b1 and w2 zero-padded to 16, so padded units and positions contribute
// nothing. z and tau of the example are written out as well.
template <int KT>
__device__ bool gate_example(const StreamParams &P, unsigned char *sm, int n, uint32_t tag,
                             uint32_t item) {
    const int gt = threadIdx.x - kGate0;
    float *zs = reinterpret_cast<float *>(sm + P.off_zs);
    const float4 *W1t = reinterpret_cast<const float4 *>(sm + P.off_w1t);
    const float *b1s = reinterpret_cast<const float *>(sm + P.off_b1);
    const float *w2s = reinterpret_cast<const float *>(sm + P.off_w2);
    constexpr int k = KT;
    const unsigned long long T = (unsigned long long)P.T;
    const unsigned long long *zb = P.zacc + ((size_t)((tag - 1u) & 1u) * P.N + n) * P.C;
    // z from the accumulator words, once each counts every tile (bounded)
    bool ok = true;
    for (int c = gt; c < P.C; c += 128) {
        unsigned long long w = ld_relaxed64(zb + c);
        for (uint32_t i = 0; (w >> 56) != T && i < kSpinLimit; ++i) {
            if ((i & 15u) == 15u && ld_relaxed(P.ctrl + kCtrlError) != 0u) break;
            __nanosleep(i < 64 ? 20 : 200);
            w = ld_relaxed64(zb + c);
        }
        if ((w >> 56) != T) {
            ok = false;
            break;
        }
        const unsigned long long nw = (w >> 48) & 0xffull;
        const long long fx =
            (long long)(w & ((1ull << 48) - 1ull)) - (long long)((T - nw) * kFixBias);
        float sum = unfix20(fx);
        if (nw != 0ull) {
            // the tagged fp32 sums of the wide tiles, in tile order, once each
            // carries this forward's tag (bounded)
            const unsigned long long *wp = P.wide + (size_t)n * P.T * P.C + c;
            bool got = false;
            for (uint32_t rep = 0; rep < kSpinLimit && !got; ++rep) {
                float acc = 0.f;
                unsigned long long seen = 0;
                for (int t = 0; t < P.T; ++t) {
                    const unsigned long long wv = ld_tagged(wp + (size_t)t * P.C);
                    if (tag_ok(wv, tag)) {
                        acc += tag_val(wv);
                        ++seen;
                    }
                }
                if (seen == nw) {
                    sum += acc;
                    got = true;
                } else if (ld_relaxed(P.ctrl + kCtrlError) != 0u) {
                    break;
                } else {
                    __nanosleep(200);
                }
            }
            if (!got) {
                ok = false;
                break;
            }
        }
        const float zv = sum * P.inv_HW;
        zs[c] = zv;
        P.z[(size_t)n * P.C + c] = zv;
    }
    if (!ok && ld_relaxed(P.ctrl + kCtrlError) == 0u) report_timeout(P.ctrl, item);
    if (!bar_and(kBarGate, 128, ok)) return false;
    const int e = gt >> 1, h = gt & 1;
    const bool act = e < P.R;
    const int ec = act ? e : 0;
    const int32_t *pi = P.pidx + ec * k;
    const float *pl = P.plog + ec * k;
    float u[KT];
#pragma unroll
    for (int i = 0; i < KT; ++i) u[i] = zs[__ldg(pi + i)];
    // hidden units 8h .. 8h + 7: h_j = b1_j + sum_i W1[j][i] u_i, in input order
    float2 hv[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) hv[m] = make_float2(b1s[8 * h + 2 * m], b1s[8 * h + 2 * m + 1]);
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const float2 uu = make_float2(u[i], u[i]);
        const float4 wa = W1t[4 * i + 2 * h], wb = W1t[4 * i + 2 * h + 1];
        hv[0] = __ffma2_rn(make_float2(wa.x, wa.y), uu, hv[0]);
        hv[1] = __ffma2_rn(make_float2(wa.z, wa.w), uu, hv[1]);
        hv[2] = __ffma2_rn(make_float2(wb.x, wb.y), uu, hv[2]);
        hv[3] = __ffma2_rn(make_float2(wb.z, wb.w), uu, hv[3]);
    }
    float gp = 0.f;
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        gp = fmaf(w2s[8 * h + 2 * m], fmaxf(hv[m].x, 0.f), gp);
        gp = fmaf(w2s[8 * h + 2 * m + 1], fmaxf(hv[m].y, 0.f), gp);
    }
    const float go = __shfl_xor_sync(0xffffffffu, gp, 1);
    const float g = (h ? go + gp : gp + go) + __ldg(P.b2);
    const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-g));
    // a_i = exp((L_i - L_0) / tau) / sum_j exp((L_j - L_0) / tau)
    const float L0 = __ldg(pl);  // position 0 holds the largest logit
    const float rt = 1.f / tau;
    float ex[8], sp = 0.f;
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const int i = 8 * h + m;
        ex[m] = i < k ? expf((__ldg(pl + i) - L0) * rt) : 0.f;
        sp += ex[m];
    }
    const float so = __shfl_xor_sync(0xffffffffu, sp, 1);
    const float S = h ? so + sp : sp + so;
    const float inv = 1.f / S;
    if (act) {
        float4 *wt = reinterpret_cast<float4 *>(P.wblk + (size_t)n * (P.tb_bytes >> 2) + wofs(e) + 8 * h);
        wt[0] = make_float4(ex[0] * inv, ex[1] * inv, ex[2] * inv, ex[3] * inv);
        wt[1] = make_float4(ex[4] * inv, ex[5] * inv, ex[6] * inv, ex[7] * inv);
        if (h == 0) P.tau[(size_t)n * P.R + e] = tau;
    }
    // the weights, z and tau are visible before the tag
    __threadfence();
    bar_sync(kBarGate, 128);
    if (gt == 0) st_release(P.flag + n, tag);
    return true;
}

// Gate role: the examples whose last tile is one of this CTA's items, in order.
template <int KT>
__device__ void role_gate(const StreamParams &P, unsigned char *sm, uint32_t tag) {
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        if (I.t != P.T - 1) continue;
        if (!gate_example<KT>(P, sm, I.n, tag, I.it)) break;
    }
}

// Table + store: for item j, the weights of its example (waiting, bounded,
// for the tag its gate publishes) into table j mod kNT; then the staged y
// tile of item j - 1 leaves by one bulk copy (its 16-byte aligned body) and
// plain stores (the unaligned head and tail, under 16 bytes each), and the
// staging buffer is handed back once the copy has read it. The table of
// item j never waits for a store, so the two duties share the warp without
// a cycle of waits.
__device__ void role_table_store(const StreamParams &P, unsigned char *sm, uint32_t tag) {
    const int lane = threadIdx.x & 31;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const int Rp = P.R + 1;
    const int n16 = (int)(P.tb_bytes >> 4);
    const int nj = items_of_cta(P);
    for (int j = 0; j <= nj; ++j) {
        if (j < nj) {
            const Item I = item_of(P, j);
            const int q = j % kNT;
            bool ok = j < kNT || mbar_wait(bar + 8u * (kMbTFree + q), (uint32_t)((j / kNT) - 1) & 1u,
                                           P.ctrl, I.it);
            if (ok && lane == 0) {
                ok = false;
                for (uint32_t i = 0; i < kSpinLimit; ++i) {
                    if (ld_acquire(P.flag + I.n) == tag) { ok = true; break; }
                    if ((i & 15u) == 15u && ld_relaxed(P.ctrl + kCtrlError) != 0u) break;
                    __nanosleep(i < 64 ? 20 : 200);
                }
                if (!ok && ld_relaxed(P.ctrl + kCtrlError) == 0u) report_timeout(P.ctrl, I.it);
            }
            if (!__shfl_sync(0xffffffffu, ok, 0)) break;
            const uint4 *src =
                reinterpret_cast<const uint4 *>(P.wblk + (size_t)I.n * (P.tb_bytes >> 2));
            uint4 *dst = reinterpret_cast<uint4 *>(sm + P.off_tab + (size_t)q * P.tb_bytes);
            for (int i = lane; i < n16; i += 32) dst[i] = __ldcg(src + i);
            __syncwarp();
            if (lane == 0) mbar_arrive(bar + 8u * (kMbTReady + q));
        }
        if (j > 0) {
            const int js = j - 1;
            const Item I = item_of(P, js);
            if (!__all_sync(0xffffffffu,
                            mbar_wait(bar + 8u * kMbYDone, (uint32_t)js & 1u, P.ctrl, I.it)))
                break;  // warp-uniform exit
            uint16_t *ydst = P.y + ((size_t)I.n * P.HW + (size_t)I.t * kTP) * Rp;
            const uint32_t dmis = (uint32_t)(reinterpret_cast<uintptr_t>(ydst) & 15u);
            const uint16_t *ys = reinterpret_cast<const uint16_t *>(sm + P.off_ys + dmis);
            // byte offsets from ydst: [0, a0) head, [a0, a1) body, [a1, nbytes) tail
            const uint32_t nbytes = (uint32_t)I.valid * (uint32_t)Rp * 2u;
            const uint32_t hi = (dmis + nbytes) & ~15u;
            const uint32_t a0 = min((16u - dmis) & 15u, nbytes);
            const uint32_t a1 = max(a0, hi - min(dmis, hi));
            if (lane == 0 && a1 > a0)
                bulk_store(reinterpret_cast<unsigned char *>(ydst) + a0,
                           smem_u32(reinterpret_cast<const unsigned char *>(ys) + a0), a1 - a0);
            if (lane < 8) {
                const uint32_t e = (uint32_t)lane;
                if (2u * e < a0) ydst[e] = ys[e];
                const uint32_t te = (a1 >> 1) + e;
                if (2u * te < nbytes) ydst[te] = ys[te];
            }
            if (lane == 0) bulk_wait_read<0>();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar + 8u * kMbYFree);
        }
    }
    if (lane == 0) bulk_wait_all();
}

// Mix: group (warp w, lanes 8 G4 .. 8 G4 + 7) owns expert pair
// P = (w mod 4) + 16 (w / 4) + 4 G4 (experts 2P, 2P + 1; the four groups of a
// warp hold pairs 4 apart, so their 16-bit output stores hit distinct banks);
// lane chunk jc covers positions 32 (jc / 4) + 8 m + 2 (jc mod 4) + {0, 1}.
template <int KT>
__device__ void role_mix(const StreamParams &P, unsigned char *sm) {
    const int tid = threadIdx.x - kMix0, w = tid >> 5, lane = tid & 31;
    const int G4 = lane >> 3, jc = lane & 7;
    const int pair = (w & 3) + 16 * (w >> 2) + 4 * G4;
    const int e0 = 2 * pair, e1 = e0 + 1;
    const bool v0 = e0 < P.R, v1 = e1 < P.R;
    constexpr int k = KT;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_x);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    uint32_t off0[KT], off1[KT];
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const int c0 = v0 ? __ldg(P.pidx + e0 * k + i) : 0;
        const int c1 = v1 ? __ldg(P.pidx + e1 * k + i) : 0;
        off0[i] = (uint32_t)c0 * 128u + ((uint32_t)(jc ^ ((c0 & 1) << 2)) << 4);
        off1[i] = (uint32_t)c1 * 128u + ((uint32_t)(jc ^ ((c1 & 1) << 2)) << 4);
    }
    const int Rp = P.R + 1;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.D, q = j % kNT;
        bool ok = mbar_wait(bar + 8u * (kMbStaged + s), (uint32_t)(j / P.D) & 1u, P.ctrl, I.it);
        ok = ok && mbar_wait(bar + 8u * (kMbTReady + q), (uint32_t)(j / kNT) & 1u, P.ctrl, I.it);
        if (!__all_sync(0xffffffffu, ok)) break;  // warp-uniform exit
        // the pair's weights of this example
        constexpr int KQ = (KT + 3) / 4;
        float w0[4 * KQ], w1[4 * KQ];
        {
            const uint32_t tb = smem_u32(sm + P.off_tab) + (uint32_t)q * P.tb_bytes;
            const uint32_t t0 = tb + 4u * (uint32_t)wofs(v0 ? e0 : 0);
            const uint32_t t1 = tb + 4u * (uint32_t)wofs(v1 ? e1 : 0);
#pragma unroll
            for (int i4 = 0; i4 < KQ; ++i4) {
                const uint4 a = lds128a(t0 + 16u * i4), b = lds128a(t1 + 16u * i4);
                w0[4 * i4] = __uint_as_float(a.x); w0[4 * i4 + 1] = __uint_as_float(a.y);
                w0[4 * i4 + 2] = __uint_as_float(a.z); w0[4 * i4 + 3] = __uint_as_float(a.w);
                w1[4 * i4] = __uint_as_float(b.x); w1[4 * i4 + 1] = __uint_as_float(b.y);
                w1[4 * i4 + 2] = __uint_as_float(b.z); w1[4 * i4 + 3] = __uint_as_float(b.w);
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar + 8u * (kMbTFree + q));
        // Eq. (expert) for the lane's 8 positions of both experts
        float2 a[4], b[4];
#pragma unroll
        for (int m = 0; m < 4; ++m) a[m] = b[m] = make_float2(0.f, 0.f);
        const uint32_t xs = xs0 + (uint32_t)s * sb;
        // k is a compile-time constant: no guard stands between one
        // support's loads and the next, so they are issued ahead
#pragma unroll
        for (int i = 0; i < KT; ++i) {
            const uint4 x0 = lds128a(xs + off0[i]);
            const uint4 x1 = lds128a(xs + off1[i]);
            const float2 c0 = make_float2(w0[i], w0[i]), c1 = make_float2(w1[i], w1[i]);
            a[0] = __ffma2_rn(c0, unpack2(x0.x), a[0]);
            a[1] = __ffma2_rn(c0, unpack2(x0.y), a[1]);
            a[2] = __ffma2_rn(c0, unpack2(x0.z), a[2]);
            a[3] = __ffma2_rn(c0, unpack2(x0.w), a[3]);
            b[0] = __ffma2_rn(c1, unpack2(x1.x), b[0]);
            b[1] = __ffma2_rn(c1, unpack2(x1.y), b[1]);
            b[2] = __ffma2_rn(c1, unpack2(x1.z), b[2]);
            b[3] = __ffma2_rn(c1, unpack2(x1.w), b[3]);
        }
        // y tile: [positions][R + 1] bf16 in the staging buffer, placed so that
        // it has the alignment mod 16 of its destination in y
        const size_t row0 = (size_t)I.n * P.HW + (size_t)I.t * kTP;
        const uint32_t dmis = (uint32_t)(reinterpret_cast<uintptr_t>(P.y + row0 * Rp) & 15u);
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys + dmis);
        // the store of item j - 1 has read the staging buffer
        ok = j < 1 || mbar_wait(bar + 8u * kMbYFree, (uint32_t)(j - 1) & 1u, P.ctrl, I.it);
        if (!__all_sync(0xffffffffu, ok)) break;
#pragma unroll
        for (int m = 0; m < 4; ++m) {
            const int p = 32 * (jc >> 2) + 8 * m + 2 * (jc & 3);
            if (v0) {
                ys[p * Rp + e0] = f32_to_bf16(a[m].x);
                ys[(p + 1) * Rp + e0] = f32_to_bf16(a[m].y);
            }
            if (v1) {
                ys[p * Rp + e1] = f32_to_bf16(b[m].x);
                ys[(p + 1) * Rp + e1] = f32_to_bf16(b[m].y);
            }
        }
        if (tid < kTP) {  // mix warps 0, 1: the residual column, once it is summed
            ok = mbar_wait(bar + 8u * (kMbResDone + s), (uint32_t)(j / P.D) & 1u, P.ctrl, I.it);
            if (!__all_sync(0xffffffffu, ok)) break;
            ys[tid * Rp + P.R] = f32_to_bf16(res_of(P, sm, s)[tid]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(bar + 8u * (kMbEmpty + s));
            mbar_arrive(bar + 8u * kMbYDone);
        }
    }
}

template <int KT>
__global__ void __launch_bounds__(kThreads_, 1)
    moce_stream_kernel(const __grid_constant__ CUtensorMap tmx, const StreamParams P) {
    extern __shared__ unsigned char smraw[];
    unsigned char *sm = smraw + ((1024u - (smem_u32(smraw) & 1023u)) & 1023u);
    const int tid = threadIdx.x, warp = tid >> 5;
    const uint32_t tag = ld_relaxed(P.ctrl + kCtrlEpoch) + 1u;
    if (tid == 0) {
        const uint32_t bar = smem_u32(sm + P.off_bar);
        for (int d = 0; d < P.D; ++d) {
            mbar_init(bar + 8u * (kMbRaw + d), 1);
            mbar_init(bar + 8u * (kMbStaged + d), 4);
            mbar_init(bar + 8u * (kMbEmpty + d), kMixT / 32);
        }
        for (int q = 0; q < kNT; ++q) {
            mbar_init(bar + 8u * (kMbTReady + q), 1);
            mbar_init(bar + 8u * (kMbTFree + q), kMixT / 32);
        }
        mbar_init(bar + 8u * kMbYDone, kMixT / 32);
        mbar_init(bar + 8u * kMbYFree, 1);
        for (int q = 0; q < 2; ++q) {
            mbar_init(bar + 8u * (kMbPooled + q), 4);
            mbar_init(bar + 8u * (kMbPFree + q), 1);
        }
        for (int d = 0; d < P.D; ++d) mbar_init(bar + 8u * (kMbResDone + d), 1);
        fence_mbar_init();
    }
    // resident tables: U and the gate parameters (W1 transposed, zero-padded
    // to 16 x 16; b1 and w2 zero-padded to 16)
    {
        uint16_t *Us = reinterpret_cast<uint16_t *>(sm + P.off_U);
        for (int i = tid; i < P.nU; i += kThreads_) Us[i] = (uint16_t)__ldg(P.resid + i);
        float *W1t = reinterpret_cast<float *>(sm + P.off_w1t);
        for (int q = tid; q < kKMax * kKMax; q += kThreads_) {
            const int i = q / kKMax, jh = q % kKMax;
            W1t[q] = (i < P.k && jh < P.k) ? __ldg(P.W1 + jh * P.k + i) : 0.f;
        }
        for (int i = tid; i < kKMax; i += kThreads_) {
            reinterpret_cast<float *>(sm + P.off_b1)[i] = i < P.k ? __ldg(P.b1 + i) : 0.f;
            reinterpret_cast<float *>(sm + P.off_w2)[i] = i < P.k ? __ldg(P.w2 + i) : 0.f;
        }
        // the accumulator bank of the previous (and the next) forward
        unsigned long long *other = P.zacc + (size_t)(tag & 1u) * P.N * P.C;
        const size_t nw = (size_t)P.N * P.C;
        for (size_t i = (size_t)blockIdx.x * kThreads_ + tid; i < nw; i += (size_t)gridDim.x * kThreads_)
            other[i] = 0ull;
    }
    __syncthreads();
    if (warp < 4) {
        set_role_regs<kRegTr, kRegLaunch>();
        role_transpose(P, sm);
    } else if (warp < 8) {
        set_role_regs<kRegGate, kRegLaunch>();
        role_gate<KT>(P, sm, tag);
    } else if (warp < 16) {
        set_role_regs<kRegMix, kRegLaunch>();
        role_mix<KT>(P, sm);
    } else {
        set_role_regs<kRegMisc, kRegLaunch>();
        if (warp == kProdW) role_producer(P, &tmx, sm);
        else if (warp == kStoreW) role_table_store(P, sm, tag);
        else if (warp == kPubW) role_publish(P, sm);
        else if (warp == kResW) role_residual(P, sm);
    }
    __syncthreads();
    if (tid == 0) {
        // the last CTA to finish advances the epoch for the next forward
        __threadfence();
        const uint32_t done = atomicAdd(P.ctrl + kCtrlExitCounter, 1u);
        if (done == gridDim.x - 1u) {
            P.ctrl[kCtrlExitCounter] = 0u;
            __threadfence();
            atomicAdd(P.ctrl + kCtrlEpoch, 1u);
        }
    }
}

// ---------------------------------------------------------------- host

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

int sm_count() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms;
}

struct StreamPlan {
    StreamParams p;
    size_t smem = 0;
};

bool plan_stream(int N, int HW, int C, int R, int k, int sms, StreamPlan *out) {
    if (C < 64 || C > 256 || C % 64 != 0 || R < 1 || R > kRMax || k < 1 || k > kKMax) return false;
    if (N < 1 || HW < 1 || sms < 1) return false;
    if ((long long)N * HW > (1ll << 31) - 1) return false;
    StreamParams &p = out->p;
    p = StreamParams{};
    p.N = N;
    p.HW = HW;
    p.C = C;
    p.R = R;
    p.k = k;
    p.T = (HW + kTP - 1) / kTP;
    if (p.T > kMaxT) return false;
    const long long items = (long long)N * p.T;
    if (items > 0x7fffffffll) return false;
    p.items = (uint32_t)items;
    p.G = (int)std::min<long long>(sms, items);
    p.nreg = C / 64;
    p.tb_bytes = table_bytes(R);
    p.ysb = (uint32_t)align_up((size_t)kTP * (R + 1) * 2, 16) + 16u;
    size_t off = 0;
    auto take = [&](size_t bytes, size_t al) {
        off = align_up(off, al);
        const size_t o = off;
        off += bytes;
        return (uint32_t)o;
    };
    p.off_tab = take((size_t)kNT * p.tb_bytes, 16);
    p.off_ys = take((size_t)p.ysb, 16);
    p.off_res = take((size_t)kMaxD * kTP * 4, 16);
    p.off_U = take((size_t)C * 2, 16);
    p.off_zs = take((size_t)C * 4, 16);
    p.off_w1t = take((size_t)kKMax * kKMax * 4, 16);
    p.off_b1 = take((size_t)kKMax * 4, 16);
    p.off_w2 = take((size_t)kKMax * 4, 16);
    p.off_psum = take((size_t)2 * C * 4, 16);
    p.off_pword = take((size_t)2 * C * 8, 16);
    p.off_bar = take((size_t)kMbCount * 8, 8);
    const size_t fixed = align_up(off, 1024);
    const size_t sb = (size_t)kTP * C * 2;
    const size_t budget = 227 * 1024 - 1024;  // 1 KB for aligning the dynamic base
    if (fixed + 3 * sb > budget) return false;
    p.D = (int)std::min<size_t>(kMaxD, (budget - fixed) / sb);
    // an example's tiles span ceil(T / G) + 1 rounds at most: with D slots a
    // CTA can hold what the gates of its oldest item still wait for
    if ((p.G - 1 + p.T - 1) / p.G > p.D - 1) return false;
    // slots first (1024-aligned for the 128-byte swizzle), then the rest
    const uint32_t shift = (uint32_t)(p.D * sb);
    p.off_x = 0;
    for (uint32_t *o : {&p.off_tab, &p.off_ys, &p.off_res, &p.off_U, &p.off_zs, &p.off_w1t,
                        &p.off_b1, &p.off_w2, &p.off_psum, &p.off_pword, &p.off_bar})
        *o += shift;
    p.smem_bytes = (uint32_t)(shift + off + 1024);
    out->smem = p.smem_bytes;
    return true;
}

}  // namespace

bool stream_supported(int N, int HW, int C, int R, int k) {
    StreamPlan plan;
    return encode_fn() != nullptr && plan_stream(N, HW, C, R, k, sm_count(), &plan);
}

cudaError_t launch_stream(const uint16_t *x, int N, int HW, int C, int R, int k,
                          const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                          const float *W1, const float *b1, const float *w2, const float *b2,
                          float tmin, float tmax, uint16_t *y, const WsLayout &L,
                          unsigned char *ws, cudaStream_t s) {
    StreamPlan plan;
    if (!plan_stream(N, HW, C, R, k, sm_count(), &plan)) return cudaErrorNotSupported;
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    CUtensorMap tm;
    const cuuint64_t dims[2] = {(cuuint64_t)C, (cuuint64_t)N * (cuuint64_t)HW};
    const cuuint64_t strides[1] = {(cuuint64_t)C * 2};
    const cuuint32_t box[2] = {64, kTP};
    const cuuint32_t es[2] = {1, 1};
    if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<uint16_t *>(x), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    StreamParams P = plan.p;
    P.y = y;
    P.nU = nU;
    P.pidx = pidx;
    P.plog = plog;
    P.resid = resid;
    P.W1 = W1;
    P.b1 = b1;
    P.w2 = w2;
    P.b2 = b2;
    P.tmin = tmin;
    P.tmax = tmax;
    P.inv_HW = 1.f / (float)HW;
    P.inv_nU = nU > 0 ? 1.f / (float)nU : 0.f;
    P.ctrl = reinterpret_cast<uint32_t *>(ws + L.ctrl);
    P.zacc = reinterpret_cast<unsigned long long *>(ws + L.zacc);
    P.wide = reinterpret_cast<unsigned long long *>(ws + L.partial);
    P.flag = reinterpret_cast<uint32_t *>(ws + L.sync) + N;
    P.wblk = reinterpret_cast<float *>(ws + L.sblk);
    P.z = reinterpret_cast<float *>(ws + L.z);
    P.tau = reinterpret_cast<float *>(ws + L.tau);
    // one instantiation per support size: the mixing and gate loops are
    // fully unrolled over k
    using Kern = void (*)(const CUtensorMap, const StreamParams);
    static const Kern kerns[kKMax] = {
        moce_stream_kernel<1>,  moce_stream_kernel<2>,  moce_stream_kernel<3>,
        moce_stream_kernel<4>,  moce_stream_kernel<5>,  moce_stream_kernel<6>,
        moce_stream_kernel<7>,  moce_stream_kernel<8>,  moce_stream_kernel<9>,
        moce_stream_kernel<10>, moce_stream_kernel<11>, moce_stream_kernel<12>,
        moce_stream_kernel<13>, moce_stream_kernel<14>, moce_stream_kernel<15>,
        moce_stream_kernel<16>};
    const Kern kern = kerns[k - 1];
    static std::mutex mu;
    static size_t configured[kKMax] = {};
    {
        std::lock_guard<std::mutex> lock(mu);
        if (plan.smem > configured[k - 1]) {
            cudaError_t err = cudaFuncSetAttribute(
                kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem);
            if (err != cudaSuccess) return err;
            configured[k - 1] = plan.smem;
        }
    }
    void *args[] = {&tm, &P};
    return cudaLaunchCooperativeKernel((const void *)kern, dim3(P.G), dim3(kThreads_), args,
                                       plan.smem, s);
}

}  // namespace moce
