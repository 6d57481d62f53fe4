// Streaming forward of a MoCE layer (Sec. 3.3-3.4) for NHWC bf16 layers with
// 64 <= C_in <= 256, C_in % 64 == 0, C_out <= 64, k <= 16 and at most 255
// tiles of 64 positions per example, in one cooperative launch: x crosses
// HBM once.
//
// Every expert's temperature needs the whole-image pool of its example
// (Sec. 3.3, Eq. (tau)), so no position can be mixed before its example has
// been pooled. Each tile is therefore read twice through the GPU but once
// from HBM: a pool stream reads it from HBM a few items ahead of the mix
// stream, adds its channel sums to the example's accumulator words and lets
// the slot go at once; the mix stream reads it again, from L2, once the
// example's gate has (usually long) run. The streams wait on each other
// only through two counters: the pool stream runs at most `lead` items ahead
// of the mix stream's loads, and the mix stream loads only tiles the pool
// stream has read. The latency from a tile's pooling to its example's
// weights thus stalls no shared-memory slot.
//
// Work: tiles of 64 positions of one example (tile t of example n is item
// it = n T + t, T = ceil(HW / 64)). Stream CTA b of Gs takes items b,
// b + Gs, ... in both streams; the other Gg CTAs (a few SMs) run the gates:
// on a stream SM a gate would share issue slots and shared memory with the
// mixing and come late. Roles of a stream CTA (640 threads):
//   pool (warps 0-3)     : warp g reads channel group g of the pool slot
//                          (ldmatrix.trans of the TMA's 128-byte swizzled
//                          [64 positions][64 channels] block) and adds the
//                          tile's channel sums (the pool, Sec. 3.3);
//   transpose (4-7)      : warp g transposes channel group g of the mix slot
//                          in place into channel-major rows (row c = the
//                          tile's 64 positions of channel c, bf16 pairs) and
//                          sums the group's unselected channels at every
//                          position (Eq. (res));
//   mix (8-15)           : each 8-lane group owns one expert pair, with their
//                          row offsets and weights in registers; a lane reads
//                          one 16-byte chunk (8 positions) of a support row
//                          and adds it with fma.rn.f32x2 (Eq. (expert)); the
//                          y tile with the residual column is staged in
//                          shared memory;
//   pool producer (16), mix producer (17): one 32 KB TMA tensor load per tile
//                          (the pool stream's with an L2 evict_last policy and
//                          an L2 prefetch a few items ahead, the mix stream's
//                          evict_first); the mix producer also brings the
//                          weights of each item's example (waiting, bounded,
//                          for the tag its gate publishes) into one of two
//                          tables by one bulk copy;
//   store (18)           : each staged y tile (two staging buffers) leaves by
//                          one bulk copy;
//   publish (19)         : the channel sums go to the example's accumulator
//                          words by one bulk reduction.
// A gate CTA takes the examples g, g + Gg, ...: it waits (bounded) until
// every accumulator word of the example counts all T tiles, decodes z, runs
// the gate of every expert (Eq. (tau)) and the softmax weights
// (Eq. (weights)), and publishes them with a tag.
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

#ifndef MOCE_STREAM_LEAD
#define MOCE_STREAM_LEAD 12
#endif
#ifndef MOCE_STREAM_DP
#define MOCE_STREAM_DP 2
#endif
#ifndef MOCE_STREAM_PF
#define MOCE_STREAM_PF 1
#endif
#ifndef MOCE_STREAM_GATES
#define MOCE_STREAM_GATES 4
#endif

namespace moce {
namespace {

constexpr int kTP = 64;             // positions per tile
constexpr int kThreads_ = 640;
constexpr int kPool0 = 0;           // warps 0-3
constexpr int kTr0 = 128;           // warps 4-7
constexpr int kMix0 = 256;          // warps 8-15
constexpr int kMixT = 256;
constexpr int kPoolProdW = 16, kMixProdW = 17, kStoreW = 18;  // warp 19 publishes
constexpr int kDP = MOCE_STREAM_DP; // pool slots
constexpr int kMaxDM = 6;           // mix slots at most
constexpr int kNT = 2;              // weight tables
constexpr int kKMax = 16;
constexpr int kRMax = 64;
constexpr int kMaxT = 255;          // tiles per example (8-bit count field)
constexpr int kBarPool = 1;
static_assert(kDP >= 2 && kDP <= 4, "pool slots");
// mbarriers: praw / pfree (pool ring), mraw / staged / empty (mix ring),
// tready / tfree (tables), ydone / yfree (y staging buffers), pooled / psfree
// (channel-sum buffers)
constexpr int kNY = 2;              // y staging buffers
constexpr int kMbPRaw = 0, kMbPFree = kDP, kMbMRaw = 2 * kDP, kMbStaged = 2 * kDP + kMaxDM,
              kMbEmpty = 2 * kDP + 2 * kMaxDM, kMbTReady = 2 * kDP + 3 * kMaxDM,
              kMbTFree = kMbTReady + kNT, kMbYDone = kMbTFree + kNT, kMbYFree = kMbYDone + kNY,
              kMbPooled = kMbYFree + kNY, kMbPsFree = kMbPooled + 2, kMbCount = kMbPsFree + 2;
// registers: 96 per thread at launch; mix 136, transpose 96, pool 64 and
// warps 16-19 48 (setmaxnreg.inc waits for registers the other warpgroups
// release: the shares must add up to no more than the launch allocation)
constexpr int kRegLaunch = 96, kRegMix = 136, kRegTr = 96, kRegPool = 64, kRegMisc = 48;
static_assert(2 * 128 * kRegMix + 128 * kRegTr + 128 * kRegPool + 128 * kRegMisc <=
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
    int N, HW, C, R, k, nU, T, nreg, Gs, Gg, DM, lead, PF;
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
    // stream CTAs
    uint32_t off_pool, off_mix, off_tab, off_ys, off_res, off_U, off_Ur, off_psum, off_pword,
        off_ctr, off_bar;
    // gate CTAs
    uint32_t g_zs, g_w1t, g_b1, g_w2, g_idx, g_dl;
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
// Tile t of example n: the box {64 channels, 64 positions, 1, all channel
// groups} of the four-dimensional view of x (see launch_stream) at position
// 64 t of example n; positions past the example's last read as zeros.
__device__ __forceinline__ void tma_load_tile(uint32_t dst, const CUtensorMap *tm, int t, int n,
                                              uint32_t mbar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(0), "r"(kTP * t), "r"(n), "r"(0), "r"(mbar),
        "l"(policy)
        : "memory");
}
// Untiled bulk copy global -> shared (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes,
                                          uint32_t mbar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(dst), "l"(src), "r"(bytes), "r"(mbar)
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
__device__ __forceinline__ void bulk_commit() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void bulk_store(void *dst, uint32_t src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                 "r"(src), "r"(bytes)
                 : "memory");
    bulk_commit();
}
// Bulk operations of this thread still reading shared memory: at most N groups.
template <int N> __device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// acc + lo, then + hi, for the two bf16 of a word (exact widening, fp32 add);
// volatile, so that the adds keep their place between the ldmatrix loads
// (hoisting all loads first would need more registers than the pool has)
__device__ __forceinline__ float add_bf16x2(float acc, uint32_t w) {
    asm volatile("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\t"
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
    bulk_commit();
}
// The two stream counters live in shared memory; the producers poll them.
__device__ __forceinline__ uint32_t ld_ctr(uint32_t a) {
    uint32_t v;
    asm volatile("ld.volatile.shared.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void st_ctr(uint32_t a, uint32_t v) {
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
// Bounded wait until the counter at a exceeds v.
__device__ bool wait_ctr(uint32_t a, uint32_t v, uint32_t *ctrl, uint32_t item) {
    for (uint32_t i = 0; i < kSpinLimit; ++i) {
        if (ld_ctr(a) > v) return true;
        if ((i & 15u) == 15u && ld_relaxed(ctrl + kCtrlError) != 0u) return false;
        __nanosleep(i < 64 ? 20 : 200);
    }
    report_timeout(ctrl, item);
    return false;
}

struct Item {
    int n, t, valid;
    uint32_t it;
};
__device__ __forceinline__ Item item_of(const StreamParams &P, int j) {
    Item r;
    r.it = (uint32_t)blockIdx.x + (uint32_t)j * (uint32_t)P.Gs;
    r.n = (int)(r.it / (uint32_t)P.T);
    r.t = (int)(r.it - (uint32_t)r.n * (uint32_t)P.T);
    r.valid = min(kTP, P.HW - r.t * kTP);
    return r;
}
__device__ __forceinline__ int items_of_cta(const StreamParams &P) {
    const uint32_t b = blockIdx.x;
    return b < P.items ? (int)((P.items - 1u - b) / (uint32_t)P.Gs) + 1 : 0;
}
// residual partial of channel group g for mix slot s: [64 positions] fp32
__device__ __forceinline__ float *res_part(const StreamParams &P, unsigned char *sm, int s, int g) {
    return reinterpret_cast<float *>(sm + P.off_res) + (s * 4 + g) * kTP;
}
// counter 0: items the pool stream has pooled; counter 1: items the mix
// stream has loaded
__device__ __forceinline__ uint32_t ctr_addr(const StreamParams &P, unsigned char *sm, int i) {
    return smem_u32(sm + P.off_ctr) + 4u * (uint32_t)i;
}

// ================================================================ roles

// Pool producer: the pool stream's TMA loads (evict_last: the mix stream
// reads the same lines again from L2), at most `lead` items ahead of the mix
// stream's loads.
__device__ void role_pool_producer(const StreamParams &P, const CUtensorMap *tm,
                                   unsigned char *sm) {
    if ((threadIdx.x & 31) != 0) return;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_pool);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
    const int nj = items_of_cta(P);
    // L2 prefetch of item j + PF with the load of item j: HBM gets PF tiles in
    // flight without holding shared memory, and the loads hit L2
    auto prefetch = [&](int j) {
        const Item I = item_of(P, j);
        asm volatile(
            "cp.async.bulk.prefetch.tensor.4d.L2.global.tile.L2::cache_hint"
            " [%0, {%1, %2, %3, %4}], %5;"
            ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(0), "r"(kTP * I.t), "r"(I.n), "r"(0),
            "l"(pol)
            : "memory");
    };
    for (int j = 0; j < min(P.PF, nj); ++j) prefetch(j);
    int issued = 0;
    for (int j = 0; j < nj; ++j) {
        const int s = j % kDP;
        if (j >= kDP &&
            !mbar_wait(bar + 8u * (kMbPFree + s), (uint32_t)((j / kDP) - 1) & 1u, P.ctrl, 0u))
            break;
        if (j >= P.lead && !wait_ctr(ctr_addr(P, sm, 1), (uint32_t)(j - P.lead), P.ctrl, 0u))
            break;
        const Item I = item_of(P, j);
        if (j + P.PF < nj) prefetch(j + P.PF);
        const uint32_t full = bar + 8u * (kMbPRaw + s);
        mbar_expect_tx(full, sb);
        tma_load_tile(xs0 + (uint32_t)s * sb, tm, I.t, I.n, full, pol);
        ++issued;
    }
    // no copy may still be writing shared memory when the CTA exits
    for (int j = issued > kDP ? issued - kDP : 0; j < issued; ++j)
        mbar_wait(bar + 8u * (kMbPRaw + j % kDP), (uint32_t)(j / kDP) & 1u, P.ctrl, 0u);
}

// Mix producer: the mix stream's TMA loads (evict_first: the lines are dead
// after this read), each once the pool stream has read the tile, so that it
// comes from L2; then the weights of the item's example, once its gate has
// published them (bounded wait on the tag), into table j mod kNT by one bulk
// copy, once the mix warps have read that table's item j - kNT.
__device__ void role_mix_producer(const StreamParams &P, const CUtensorMap *tm,
                                  unsigned char *sm, uint32_t tag) {
    if ((threadIdx.x & 31) != 0) return;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_mix);
    const uint32_t tb0 = smem_u32(sm + P.off_tab);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    const int nj = items_of_cta(P);
    int issued = 0, tabs = 0;
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.DM, q = j % kNT;
        if (j >= P.DM && !mbar_wait(bar + 8u * (kMbEmpty + s), (uint32_t)((j / P.DM) - 1) & 1u,
                                    P.ctrl, I.it))
            break;
        if (!wait_ctr(ctr_addr(P, sm, 0), (uint32_t)j, P.ctrl, I.it)) break;
        const uint32_t full = bar + 8u * (kMbMRaw + s);
        mbar_expect_tx(full, sb);
        tma_load_tile(xs0 + (uint32_t)s * sb, tm, I.t, I.n, full, pol);
        ++issued;
        st_ctr(ctr_addr(P, sm, 1), (uint32_t)issued);
        if (j >= kNT && !mbar_wait(bar + 8u * (kMbTFree + q), (uint32_t)((j / kNT) - 1) & 1u,
                                   P.ctrl, I.it))
            break;
        bool ok = false;
        for (uint32_t i = 0; i < kSpinLimit; ++i) {
            if (ld_acquire(P.flag + I.n) == tag) { ok = true; break; }
            if ((i & 15u) == 15u && ld_relaxed(P.ctrl + kCtrlError) != 0u) break;
            __nanosleep(i < 64 ? 20 : 100);
        }
        if (!ok) {
            if (ld_relaxed(P.ctrl + kCtrlError) == 0u) report_timeout(P.ctrl, I.it);
            break;
        }
        // the gate's stores (generic proxy, seen through the acquire) before
        // the bulk copy's reads (async proxy)
        asm volatile("fence.proxy.async.global;" ::: "memory");
        const uint32_t tfull = bar + 8u * (kMbTReady + q);
        mbar_expect_tx(tfull, P.tb_bytes);
        bulk_load(tb0 + (uint32_t)q * P.tb_bytes, P.wblk + (size_t)I.n * (P.tb_bytes >> 2),
                  P.tb_bytes, tfull);
        ++tabs;
    }
    // no copy may still be writing shared memory when the CTA exits
    for (int j = issued > P.DM ? issued - P.DM : 0; j < issued; ++j)
        mbar_wait(bar + 8u * (kMbMRaw + j % P.DM), (uint32_t)(j / P.DM) & 1u, P.ctrl, 0u);
    for (int j = tabs > kNT ? tabs - kNT : 0; j < tabs; ++j)
        mbar_wait(bar + 8u * (kMbTReady + j % kNT), (uint32_t)(j / kNT) & 1u, P.ctrl, 0u);
}

// Pool, warp g on channel group g. Region g of the pool slot (8 KB) holds
// [64 positions][64 channels] as the TMA wrote it (128-byte swizzle: 16-byte
// chunk c of row p at chunk c ^ (p & 7)); ldmatrix.trans of 8x8 blocks gives
// lane l (cl = l / 4, q = l mod 4) the words {x[p][c], x[p + 1][c]} for
// channel c = 8 jj + cl of the region and positions p = 32 h + 8 m + 2 q.
// The lane adds them per channel; the four lanes of a channel (q) are added
// in a fixed order and the tile's channel sums go to sum buffer j mod 2 for
// the publish warp. Once every warp has read the slot it goes back to the
// producer, and the item counts as loaded for the mix stream.
__device__ void role_pool(const StreamParams &P, unsigned char *sm) {
    const int tt = threadIdx.x - kPool0;  // 0..127
    const int g = tt >> 5, lane = tt & 31;
    const int q = lane & 3, cl = lane >> 2;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_pool);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    const bool own = g < P.nreg;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % kDP, pb = j & 1;
        bool ok = mbar_wait(bar + 8u * (kMbPRaw + s), (uint32_t)(j / kDP) & 1u, P.ctrl, I.it);
        // the publish warp has read sum buffer pb (item j - 2)
        ok = ok && (j < 2 || mbar_wait(bar + 8u * (kMbPsFree + pb), (uint32_t)((j >> 1) - 1) & 1u,
                                       P.ctrl, I.it));
        if (ok && own) {
            float pacc[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) pacc[jj] = 0.f;
            const uint32_t rb = xs0 + (uint32_t)s * sb + 8192u * (uint32_t)g;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint32_t r[8][4];
#pragma unroll
                for (int jj = 0; jj < 8; ++jj)
                    ldsm_x4_t(rb + (uint32_t)(32 * h + lane) * 128u +
                                  ((uint32_t)(jj ^ (lane & 7)) << 4),
                              r[jj]);
                // positions past the example are zeros (the TMA fill)
#pragma unroll
                for (int m = 0; m < 4; ++m)
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj) pacc[jj] = add_bf16x2(pacc[jj], r[jj][m]);
            }
            float *ps = reinterpret_cast<float *>(sm + P.off_psum) + pb * P.C + 64 * g;
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                float v = pacc[jj];
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                if ((jj & 3) == q) ps[8 * jj + cl] = v;
            }
        }
        if (!bar_and(kBarPool, 128, ok)) break;  // every warp has read the slot
        if (tt == 0) {
            mbar_arrive(bar + 8u * (kMbPFree + s));
            mbar_arrive(bar + 8u * (kMbPooled + pb));
            st_ctr(ctr_addr(P, sm, 0), (uint32_t)(j + 1));
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
        if (!__all_sync(0xffffffffu, mbar_wait(bar + 8u * (kMbPooled + pb),
                                                (uint32_t)(j >> 1) & 1u, P.ctrl, I.it)))
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
            asm volatile("st.shared.u64 [%0], %1;" ::"r"(pw + 8u * (uint32_t)c), "l"(add)
                         : "memory");
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(bar + 8u * (kMbPsFree + pb));
            if (I.it + 1u != drop)  // fault injection: never counted
                bulk_reduce_add_u64(zb + (size_t)I.n * P.C, pw, (uint32_t)P.C * 8u);
            else
                bulk_commit();  // an empty group keeps one group per item
        }
    }
    if (lane == 0) bulk_wait_all();  // the last reductions are complete
}

// Transpose, warp g on channel group g of the mix slot, in place: the lane's
// four ldmatrix words (positions 32 h + 8 m + 2 q, m = 0..3, of channel
// c = 8 jj + cl) go as one 16-byte chunk to logical chunk 4 h + q of row c
// (physical chunk (4 h + q) ^ (4 (c & 1))): row c then holds the tile's 64
// positions of channel c, word 16 h + 4 q + m holding positions
// 2 (16 h + 4 m + q) and the next. Then the residual expert (Eq. (res)) over
// the group's unselected channels: lane (part = lane / 8, chunk jc = lane
// mod 8) adds the group's entries of U part, part + 4, ... over its chunk's
// 8 positions, the four parts in a fixed order.
__device__ void role_transpose(const StreamParams &P, unsigned char *sm) {
    const int tt = threadIdx.x - kTr0;  // 0..127
    const int g = tt >> 5, lane = tt & 31;
    const int q = lane & 3, cl = lane >> 2;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_mix);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    const bool own = g < P.nreg;
    // the entries of U in channel group g, in U's order (ballot compaction)
    const uint16_t *Us = reinterpret_cast<const uint16_t *>(sm + P.off_U);
    uint16_t *Ur = reinterpret_cast<uint16_t *>(sm + P.off_Ur) + g * P.C;
    int nr = 0;
    for (int u0 = 0; u0 < P.nU; u0 += 32) {
        const int u = u0 + lane;
        const int c = u < P.nU ? (int)Us[u] : -1;
        const bool mine = own && (c >> 6) == g;
        const uint32_t bal = __ballot_sync(0xffffffffu, mine);
        if (mine) Ur[nr + __popc(bal & ((1u << lane) - 1u))] = (uint16_t)c;
        nr += __popc(bal);
    }
    __syncwarp();
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.DM;
        if (!__all_sync(0xffffffffu,
                        mbar_wait(bar + 8u * (kMbMRaw + s), (uint32_t)(j / P.DM) & 1u, P.ctrl, I.it)))
            break;  // warp-uniform exit
        const uint32_t xs = xs0 + (uint32_t)s * sb;
        if (own) {
            const uint32_t rb = xs + 8192u * (uint32_t)g;
            uint32_t r[16][4];
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int jj = 0; jj < 8; ++jj)
                    ldsm_x4_t(rb + (uint32_t)(32 * h + lane) * 128u +
                                  ((uint32_t)(jj ^ (lane & 7)) << 4),
                              r[8 * h + jj]);
            __syncwarp();
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) {
                    const int c = 8 * jj + cl;
                    sts128(rb + (uint32_t)c * 128u + ((uint32_t)((4 * h + q) ^ ((c & 1) << 2)) << 4),
                           r[8 * h + jj]);
                }
            __syncwarp();
            const int jc = lane & 7, part = lane >> 3;
            float2 ra[4];
#pragma unroll
            for (int m = 0; m < 4; ++m) ra[m] = make_float2(0.f, 0.f);
#pragma unroll 2
            for (int u = part; u < nr; u += 4) {
                const int c = Ur[u];
                const uint4 v =
                    lds128a(xs + (uint32_t)c * 128u + ((uint32_t)(jc ^ ((c & 1) << 2)) << 4));
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
                float *rp = res_part(P, sm, s, g);
#pragma unroll
                for (int m = 0; m < 4; ++m) {
                    const int p = 32 * (jc >> 2) + 8 * m + 2 * (jc & 3);
                    rp[p] = ra[m].x;
                    rp[p + 1] = ra[m].y;
                }
            }
            __syncwarp();
        }
        if (lane == 0) mbar_arrive(bar + 8u * (kMbStaged + s));
    }
}

// Gate CTA: the examples n = g, g + Gg, ... (g = its index among the Gg gate
// CTAs), in order. For each, thread c waits (bounded) until accumulator word
// c of the example counts all T tiles and decodes z_c; then thread
// 4 e + q runs hidden units 4 q .. 4 q + 3 of expert e's gate (Eq. (tau))
// and its softmax weights 4 q .. 4 q + 3 (Eq. (weights)), the four threads
// of an expert adding their partial sums in a fixed order; the weights go to
// the example's weight block in global memory, published with a tag. W1 is
// kept transposed and zero-padded to 16 x 16 (W1t[i][j] = W1[j][i]), b1 and w2
// zero-padded to 16, and per expert its support channels and logit offsets
// L_i - L_0 (L_0 the largest), so padded units and entries add nothing.
template <int KT>
__device__ void gate_cta(const StreamParams &P, unsigned char *sm, uint32_t tag) {
    const int tid = threadIdx.x;
    float *zs = reinterpret_cast<float *>(sm + P.g_zs);
    const float4 *W1t = reinterpret_cast<const float4 *>(sm + P.g_w1t);
    const float *b1s = reinterpret_cast<const float *>(sm + P.g_b1);
    const float *w2s = reinterpret_cast<const float *>(sm + P.g_w2);
    const uint16_t *gidx = reinterpret_cast<const uint16_t *>(sm + P.g_idx);
    const float4 *gdl = reinterpret_cast<const float4 *>(sm + P.g_dl);
    const unsigned long long T = (unsigned long long)P.T;
    const float b2 = __ldg(P.b2);
    for (int n = (int)blockIdx.x - P.Gs; n < P.N; n += P.Gg) {
        const uint32_t item = (uint32_t)n * (uint32_t)P.T + (uint32_t)P.T - 1u;
        // z from the accumulator words, once each counts every tile (bounded)
        bool ok = true;
        if (tid < P.C) {
            const int c = tid;
            const unsigned long long *zb = P.zacc + ((size_t)((tag - 1u) & 1u) * P.N + n) * P.C;
            unsigned long long w = ld_relaxed64(zb + c);
            for (uint32_t i = 0; (w >> 56) != T && i < kSpinLimit; ++i) {
                if ((i & 15u) == 15u && ld_relaxed(P.ctrl + kCtrlError) != 0u) break;
                __nanosleep(i < 256 ? 20 : 100);
                w = ld_relaxed64(zb + c);
            }
            ok = (w >> 56) == T;
            float sum = 0.f;
            if (ok) {
                const unsigned long long nw = (w >> 48) & 0xffull;
                const long long fx =
                    (long long)(w & ((1ull << 48) - 1ull)) - (long long)((T - nw) * kFixBias);
                sum = unfix20(fx);
                if (nw != 0ull) {
                    // the tagged fp32 sums of the wide tiles, in tile order, once
                    // each carries this forward's tag (bounded)
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
                    ok = got;
                }
            }
            const float zv = sum * P.inv_HW;
            zs[c] = zv;
            P.z[(size_t)n * P.C + c] = zv;
            if (!ok && ld_relaxed(P.ctrl + kCtrlError) == 0u) report_timeout(P.ctrl, item);
        }
        if (!__syncthreads_and(ok)) break;
        // whole warps (the shuffles need every lane); only threads below 4 R write
        if (tid < ((4 * P.R + 31) & ~31)) {
            const int e = min(tid >> 2, P.R - 1), q = tid & 3;
            const bool wr = tid < 4 * P.R;
            // h_j = b1_j + sum_i W1[j][i] u_i, in input order, for j = 4 q .. 4 q + 3
            float4 h = reinterpret_cast<const float4 *>(b1s)[q];
#pragma unroll
            for (int i = 0; i < KT; ++i) {
                const float ui = zs[gidx[e * 16 + i]];
                const float4 w = W1t[4 * i + q];
                h.x = fmaf(w.x, ui, h.x);
                h.y = fmaf(w.y, ui, h.y);
                h.z = fmaf(w.z, ui, h.z);
                h.w = fmaf(w.w, ui, h.w);
            }
            const float4 w2 = reinterpret_cast<const float4 *>(w2s)[q];
            float g = w2.x * fmaxf(h.x, 0.f);
            g = fmaf(w2.y, fmaxf(h.y, 0.f), g);
            g = fmaf(w2.z, fmaxf(h.z, 0.f), g);
            g = fmaf(w2.w, fmaxf(h.w, 0.f), g);
            g += __shfl_xor_sync(0xffffffffu, g, 1);
            g += __shfl_xor_sync(0xffffffffu, g, 2);
            const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-(g + b2)));
            // a_i = exp((L_i - L_0) / tau) / sum_j exp((L_j - L_0) / tau)
            const float rt = 1.f / tau;
            const float4 d = gdl[e * 4 + q];
            float4 ex;
            ex.x = 4 * q + 0 < KT ? expf(d.x * rt) : 0.f;
            ex.y = 4 * q + 1 < KT ? expf(d.y * rt) : 0.f;
            ex.z = 4 * q + 2 < KT ? expf(d.z * rt) : 0.f;
            ex.w = 4 * q + 3 < KT ? expf(d.w * rt) : 0.f;
            float S = (ex.x + ex.y) + (ex.z + ex.w);
            S += __shfl_xor_sync(0xffffffffu, S, 1);
            S += __shfl_xor_sync(0xffffffffu, S, 2);
            const float inv = 1.f / S;
            if (wr) {
                reinterpret_cast<float4 *>(P.wblk + (size_t)n * (P.tb_bytes >> 2) + wofs(e))[q] =
                    make_float4(ex.x * inv, ex.y * inv, ex.z * inv, ex.w * inv);
                if (q == 0) P.tau[(size_t)n * P.R + e] = tau;
            }
        }
        // every thread's weights, z and tau are visible before the tag (the
        // barrier orders them before thread 0's fence, which is cumulative)
        __syncthreads();
        if (tid == 0) {
            __threadfence();
            st_release(P.flag + n, tag);
        }
    }
}

// Store: the staged y tile of item j (buffer j mod kNY) leaves by one bulk
// copy (its 16-byte aligned body) and plain stores (the unaligned head and
// tail, under 16 bytes each); the buffer goes back to the mix warps as soon
// as the copy has read it.
__device__ void role_store(const StreamParams &P, unsigned char *sm) {
    const int lane = threadIdx.x & 31;
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const int Rp = P.R + 1;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int b = j % kNY;
        if (!__all_sync(0xffffffffu, mbar_wait(bar + 8u * (kMbYDone + b),
                                                (uint32_t)(j / kNY) & 1u, P.ctrl, I.it)))
            break;  // warp-uniform exit
        uint16_t *ydst = P.y + ((size_t)I.n * P.HW + (size_t)I.t * kTP) * Rp;
        const uint32_t dmis = (uint32_t)(reinterpret_cast<uintptr_t>(ydst) & 15u);
        const uint16_t *ys =
            reinterpret_cast<const uint16_t *>(sm + P.off_ys + (size_t)b * P.ysb + dmis);
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
        // the buffer goes back once the copy has read it
        if (lane == 0) {
            bulk_wait_read<0>();
            mbar_arrive(bar + 8u * (kMbYFree + b));
        }
        __syncwarp();
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
    const uint32_t bar = smem_u32(sm + P.off_bar);
    const uint32_t xs0 = smem_u32(sm + P.off_mix);
    const uint32_t sb = (uint32_t)P.C * kTP * 2u;
    uint32_t off0[KT], off1[KT];
#pragma unroll
    for (int i = 0; i < KT; ++i) {
        const int c0 = v0 ? __ldg(P.pidx + e0 * KT + i) : 0;
        const int c1 = v1 ? __ldg(P.pidx + e1 * KT + i) : 0;
        off0[i] = (uint32_t)c0 * 128u + ((uint32_t)(jc ^ ((c0 & 1) << 2)) << 4);
        off1[i] = (uint32_t)c1 * 128u + ((uint32_t)(jc ^ ((c1 & 1) << 2)) << 4);
    }
    const int Rp = P.R + 1;
    const int nj = items_of_cta(P);
    for (int j = 0; j < nj; ++j) {
        const Item I = item_of(P, j);
        const int s = j % P.DM, q = j % kNT;
        bool ok = mbar_wait(bar + 8u * (kMbStaged + s), (uint32_t)(j / P.DM) & 1u, P.ctrl, I.it);
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
        // the residual partials of the channel groups, in group order
        float rv = 0.f;
        if (tid < kTP)
            for (int g = 0; g < P.nreg; ++g) rv += res_part(P, sm, s, g)[tid];
        // the slot is read: it goes back to the mix producer
        __syncwarp();
        if (lane == 0) mbar_arrive(bar + 8u * (kMbEmpty + s));
        // y tile: [positions][R + 1] bf16 in staging buffer j mod kNY, placed so
        // that it has the alignment mod 16 of its destination in y
        const int yb = j % kNY;
        const size_t row0 = (size_t)I.n * P.HW + (size_t)I.t * kTP;
        const uint32_t dmis = (uint32_t)(reinterpret_cast<uintptr_t>(P.y + row0 * Rp) & 15u);
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys + (size_t)yb * P.ysb + dmis);
        // the store of item j - kNY has read the staging buffer
        ok = j < kNY || mbar_wait(bar + 8u * (kMbYFree + yb), (uint32_t)((j / kNY) - 1) & 1u,
                                  P.ctrl, I.it);
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
        if (tid < kTP) ys[tid * Rp + P.R] = f32_to_bf16(rv * P.inv_nU);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar + 8u * (kMbYDone + yb));
    }
}

// Stream CTA: barriers, U, then the roles.
template <int KT>
__device__ void stream_cta(const StreamParams &P, const CUtensorMap *tm, unsigned char *sm,
                           uint32_t tag) {
    const int tid = threadIdx.x, warp = tid >> 5;
    if (tid == 0) {
        const uint32_t bar = smem_u32(sm + P.off_bar);
        for (int d = 0; d < kDP; ++d) {
            mbar_init(bar + 8u * (kMbPRaw + d), 1);
            mbar_init(bar + 8u * (kMbPFree + d), 1);
        }
        for (int d = 0; d < P.DM; ++d) {
            mbar_init(bar + 8u * (kMbMRaw + d), 1);
            mbar_init(bar + 8u * (kMbStaged + d), 4);
            mbar_init(bar + 8u * (kMbEmpty + d), kMixT / 32);
        }
        for (int q = 0; q < kNT; ++q) {
            mbar_init(bar + 8u * (kMbTReady + q), 1);
            mbar_init(bar + 8u * (kMbTFree + q), kMixT / 32);
        }
        for (int b = 0; b < kNY; ++b) {
            mbar_init(bar + 8u * (kMbYDone + b), kMixT / 32);
            mbar_init(bar + 8u * (kMbYFree + b), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar + 8u * (kMbPooled + b), 1);
            mbar_init(bar + 8u * (kMbPsFree + b), 1);
        }
        st_ctr(ctr_addr(P, sm, 0), 0u);
        st_ctr(ctr_addr(P, sm, 1), 0u);
        fence_mbar_init();
    }
    uint16_t *Us = reinterpret_cast<uint16_t *>(sm + P.off_U);
    for (int i = tid; i < P.nU; i += kThreads_) Us[i] = (uint16_t)__ldg(P.resid + i);
    __syncthreads();
    if (warp < 4) {
        set_role_regs<kRegPool, kRegLaunch>();
        role_pool(P, sm);
    } else if (warp < 8) {
        set_role_regs<kRegTr, kRegLaunch>();
        role_transpose(P, sm);
    } else if (warp < 16) {
        set_role_regs<kRegMix, kRegLaunch>();
        role_mix<KT>(P, sm);
    } else {
        set_role_regs<kRegMisc, kRegLaunch>();
        if (warp == kPoolProdW) role_pool_producer(P, tm, sm);
        else if (warp == kMixProdW) role_mix_producer(P, tm, sm, tag);
        else if (warp == kStoreW) role_store(P, sm);
        else role_publish(P, sm);
    }
}

// Gate CTA: the resident gate parameters, then its examples.
template <int KT>
__device__ void gate_cta_main(const StreamParams &P, unsigned char *sm, uint32_t tag) {
    const int tid = threadIdx.x;
    float *W1t = reinterpret_cast<float *>(sm + P.g_w1t);
    for (int q = tid; q < kKMax * kKMax; q += kThreads_) {
        const int i = q / kKMax, jh = q % kKMax;
        W1t[q] = (i < KT && jh < KT) ? __ldg(P.W1 + jh * KT + i) : 0.f;
    }
    for (int i = tid; i < kKMax; i += kThreads_) {
        reinterpret_cast<float *>(sm + P.g_b1)[i] = i < KT ? __ldg(P.b1 + i) : 0.f;
        reinterpret_cast<float *>(sm + P.g_w2)[i] = i < KT ? __ldg(P.w2 + i) : 0.f;
    }
    uint16_t *gidx = reinterpret_cast<uint16_t *>(sm + P.g_idx);
    float *gdl = reinterpret_cast<float *>(sm + P.g_dl);
    for (int q = tid; q < P.R * kKMax; q += kThreads_) {
        const int e = q / kKMax, i = q % kKMax;
        gidx[q] = i < KT ? (uint16_t)__ldg(P.pidx + e * KT + i) : 0;
        gdl[q] = i < KT ? __ldg(P.plog + e * KT + i) - __ldg(P.plog + e * KT) : 0.f;
    }
    __syncthreads();
    gate_cta<KT>(P, sm, tag);
}

// CTAs 0 .. Gs - 1 stream the items; CTAs Gs .. Gs + Gg - 1 run the gates.
template <int KT>
__global__ void __launch_bounds__(kThreads_, 1)
    moce_stream_kernel(const __grid_constant__ CUtensorMap tmx, const StreamParams P) {
    extern __shared__ unsigned char smraw[];
    unsigned char *sm = smraw + ((1024u - (smem_u32(smraw) & 1023u)) & 1023u);
    const int tid = threadIdx.x;
    const uint32_t tag = ld_relaxed(P.ctrl + kCtrlEpoch) + 1u;
    {
        // the accumulator bank of the previous (and the next) forward
        unsigned long long *other = P.zacc + (size_t)(tag & 1u) * P.N * P.C;
        const size_t nw = (size_t)P.N * P.C;
        for (size_t i = (size_t)blockIdx.x * kThreads_ + tid; i < nw;
             i += (size_t)gridDim.x * kThreads_)
            other[i] = 0ull;
    }
    if ((int)blockIdx.x < P.Gs) stream_cta<KT>(P, &tmx, sm, tag);
    else gate_cta_main<KT>(P, sm, tag);
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

// Items the pool stream may run ahead of the mix stream's loads: enough to
// cover the latency from a tile's pooling to its example's weights, few
// enough that the lines it has read stay in L2 until the mix stream reads
// them (Gs (lead + pool slots) tiles, about 66 MB at 148 stream CTAs and
// C_in 256; on the 256-channel, 64-example layer leads of 10 to 22 measure
// alike, 6 is 12 % slower).
constexpr int kLead = MOCE_STREAM_LEAD;
// Items the pool producer prefetches into L2 ahead of its loads.
constexpr int kPrefetch = MOCE_STREAM_PF;
// SMs that run gates only.
constexpr int kGateCtas = MOCE_STREAM_GATES;

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
    // a few whole SMs run the gates: on a stream SM they would share the issue
    // slots and shared memory with the mixing and come late
    p.Gg = std::min(kGateCtas, N);
    if (sms <= p.Gg) return false;
    p.Gs = (int)std::min<long long>(sms - p.Gg, items);
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
    p.off_ys = take((size_t)kNY * p.ysb, 16);
    p.off_U = take((size_t)C * 2, 16);
    p.off_Ur = take((size_t)4 * C * 2, 16);
    p.off_psum = take((size_t)2 * C * 4, 16);
    p.off_pword = take((size_t)2 * C * 8, 16);
    p.off_ctr = take(16, 16);
    p.off_bar = take((size_t)kMbCount * 8, 8);
    // the residual partials: 4 groups x 64 positions of fp32 per mix slot
    const size_t sb = (size_t)kTP * C * 2, resb = (size_t)4 * kTP * 4;
    const size_t budget = 227 * 1024 - 1024;  // 1 KB for aligning the dynamic base
    p.DM = 0;
    for (int dm = kMaxDM; dm >= 2 && p.DM == 0; --dm)
        if (align_up(align_up(off, 16) + dm * resb, 1024) + (kDP + dm) * sb <= budget) p.DM = dm;
    if (p.DM == 0) return false;
    p.off_res = take((size_t)p.DM * resb, 16);
    const size_t fixed_end = off;
    p.lead = kLead;
    p.PF = kPrefetch;
    // Progress: the pool stream's item j waits for the mix producer to load
    // item j - lead, which it does after the weights of item j - lead - 1's
    // example are published. That example must be an earlier one than every
    // example item j belongs to, so (lead + 1) Gs must exceed the tiles of one
    // example (with one round to spare).
    if ((long long)p.lead * p.Gs < (long long)p.T) return false;
    // slots first (1024-aligned for the 128-byte swizzle), then the rest
    p.off_pool = 0;
    p.off_mix = (uint32_t)(kDP * sb);
    const uint32_t shift = (uint32_t)((kDP + p.DM) * sb);
    for (uint32_t *o : {&p.off_tab, &p.off_ys, &p.off_U, &p.off_Ur, &p.off_psum, &p.off_pword,
                        &p.off_ctr, &p.off_bar, &p.off_res})
        *o += shift;
    // the gate CTAs' resident tables, from the start of shared memory
    off = 0;
    p.g_zs = take((size_t)C * 4, 16);
    p.g_w1t = take((size_t)kKMax * kKMax * 4, 16);
    p.g_b1 = take((size_t)kKMax * 4, 16);
    p.g_w2 = take((size_t)kKMax * 4, 16);
    p.g_idx = take((size_t)R * kKMax * 2, 16);
    p.g_dl = take((size_t)R * kKMax * 4, 16);
    if (off > shift) return false;  // never: the slots alone exceed it
    p.smem_bytes = (uint32_t)(shift + fixed_end + 1024);
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
    // x viewed as [channel group][example][position][64 channels]: one box
    // of {64, 64, 1, C / 64} is a whole tile, landing as C / 64 regions of
    // [64 positions][128 bytes] (128-byte swizzle) in one copy (copies of
    // 32 KB keep HBM busy where 8 KB ones, a box per channel group, do not);
    // positions past the example's HW are outside the view and read as zeros.
    CUtensorMap tm;
    const cuuint64_t dims[4] = {64, (cuuint64_t)HW, (cuuint64_t)N, (cuuint64_t)(C / 64)};
    const cuuint64_t strides[3] = {(cuuint64_t)C * 2, (cuuint64_t)HW * C * 2, 128};
    const cuuint32_t box[4] = {64, kTP, 1, (cuuint32_t)(C / 64)};
    const cuuint32_t es[4] = {1, 1, 1, 1};
    if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_UINT16, 4, const_cast<uint16_t *>(x), dims, strides, box,
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
    return cudaLaunchCooperativeKernel((const void *)kern, dim3(P.Gs + P.Gg), dim3(kThreads_), args,
                                       plan.smem, s);
}

}  // namespace moce
