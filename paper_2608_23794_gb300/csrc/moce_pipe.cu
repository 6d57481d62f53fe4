// Warp-specialised persistent forward kernel of a MoCE layer (Sec. 3.3-3.4):
// pooling, gate, softmax weights, routed mixing and the residual expert in one
// launch, for NHWC bf16 layers with C_in <= 256.
//
// The temperature of every expert depends on the whole-image average of its
// support (Sec. 3.3), so an example can only be mixed after all of it has been
// pooled: x is read twice, the second time shortly after the first (mostly
// from L2). One CTA per SM (cooperative launch, so all CTAs are resident)
// runs three warp roles:
//
//   pool   (warps 16-23) pools slices of examples ("units"). Each warp owns a
//          slice of the channels and streams the unit's rows of those
//          channels with a rolling window of 16-byte loads; at the end of a
//          unit its lanes combine their row sums with shuffles and write the
//          unit's channel sums as tagged words (value + forward epoch).
//   stage  (warps 8-15) prepares mixing tiles in two buffers. Tiles come in
//          runs of consecutive tiles of one example; at the start of a run it
//          reduces z from the unit sums (unit order, so z is deterministic)
//          and evaluates the gate of every expert (Eq. (tau)) and the softmax
//          weights (Eq. (weights)). For every tile it writes the weights into
//          the tile's table of {row offset, weight} entries, stages x of the
//          tile transposed to channel-major rows of pixel pairs, and writes
//          the previous finished tile of y to HBM (one bulk copy when rows
//          allow it).
//   mix    (warps 0-7) mixes the full buffer: each group of 8 lanes owns 8
//          positions per lane and computes an expert pair (Eq. (expert)) with
//          one 16-byte shared load per support and packed fp32 FMAs, plus a
//          slice of the residual sum (Eq. (res)).
//
// Stage and mix hand buffers over through shared-memory mbarriers. Every wait
// is bounded: one that gives up records MOCE_ERR_TIMEOUT in the workspace and
// makes every other wait return. Waits form no cycle: mix waits for stage,
// stage for mix (an earlier tile) and for unit sums, which the pool roles
// write without waiting for anything.
#include <algorithm>

#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kGS = 8;                // lanes of a mixing group
constexpr int kGPW = 32 / kGS;        // mixing groups per warp
constexpr int kTP = 8 * kGS;          // positions per mixing tile
constexpr int kRB = 16 * kGS;         // bytes per staged channel row
constexpr int kFM = 7;                // chunk swizzle mask of the staged rows
constexpr int kMixT = 256;            // mix role: warps 0-7
constexpr int kStageT = 256;          // stage role: warps 8-15
constexpr int kPoolT = 256;           // pool role: warps 16-23
constexpr int kPipeT = kMixT + kStageT + kPoolT;
constexpr int kMixWarps = kMixT / 32;
constexpr int kPoolWarps = kPoolT / 32;
constexpr int kGroups = kMixT / kGS;  // mixing groups per CTA
constexpr int kRPS = kTP + 8;         // row stride (floats) of the residual partial sums
constexpr int kBarStage = 2, kBarPrologue = 3;
constexpr int kBufs = 2;              // tile buffers (x, y, residual sums) between stage and mix
constexpr int kWTabs = kBufs + 1;     // run tables: the mix role may still read kBufs runs
constexpr int kStageU = 4;            // staging units (2 x 16 bytes) per stage thread and tile
constexpr int kRun = 7;               // mixing tiles per run (one gate per run)
constexpr int kPoolWin = 6;           // rolling window of 16-byte loads per pool thread
constexpr int kMaxUnits = 16;         // pooling units per example (z reads them at once)
constexpr int kGateMaxK = 64;         // gate width of the one-warp-per-expert gate
// Registers per thread of each role. The launch gives every thread 80
// (kPipeT * 80 <= 65536); the roles then trade them with setmaxnreg within
// the launch's total.
constexpr int kLaunchRegs = 80, kMixRegs = 80, kStageRegs = 96, kPoolRegs = 64;
static_assert(kMixT * kMixRegs + kStageT * kStageRegs + kPoolT * kPoolRegs <= kPipeT * kLaunchRegs,
              "register split exceeds the launch allocation");
static_assert(kPipeT * kLaunchRegs <= 65536, "launch registers");

struct PipeParams {
    const uint16_t *x;
    uint16_t *y;
    int N, HW, C, R, k, nU;
    const int32_t *pidx;
    const float *plog;
    const int32_t *resid;
    const float *W1, *b1, *w2, *b2;
    float tmin, tmax;
    uint32_t *ctrl;
    unsigned long long *part;     // tagged unit sums [N][S][C]
    float *z, *tau;
    int S;                        // pooling units per example
    int MT, RN;                   // mixing tiles and runs per example
    uint32_t pool_items, runs;
    int cpw, rpi;                 // pool: 8-channel blocks per warp, rows per load instruction
    int kp, Es, ks, Kg, gate_tabs;  // Kg: padded gate width of the group gate, 0: warp gate
    int bulk_y;                   // output tiles leave by one bulk copy (rows of E = R + 1)
    uint32_t off_xs[kBufs], off_ys[kBufs], off_rp[kBufs], off_tab[kWTabs];
    uint32_t off_zs, off_zbuf, off_uw, off_W1, off_b1, off_w2, off_pidx, off_plog, off_U, off_bar;
    float inv_perq, inv_E, inv_kp;
};


// This CTA's mixing tiles, in order: runs q = blockIdx.x, blockIdx.x + G, ...
// of up to kRun consecutive tiles of one example.
struct TileIter {
    uint32_t q;  // run
    int j;       // tile within the run
};
struct TileRef {
    int n, p0, np;
};

__device__ __forceinline__ int run_len(const PipeParams &P, uint32_t q) {
    const int r = (int)(q % (uint32_t)P.RN);
    return min(kRun, P.MT - r * kRun);
}
__device__ __forceinline__ TileRef tile_of(const PipeParams &P, const TileIter &it) {
    TileRef t;
    t.n = (int)(it.q / (uint32_t)P.RN);
    const int r = (int)(it.q - (uint32_t)t.n * P.RN);
    t.p0 = (r * kRun + it.j) * kTP;
    t.np = min(kTP, P.HW - t.p0);
    return t;
}
__device__ __forceinline__ void tile_next(const PipeParams &P, TileIter &it) {
    if (++it.j >= run_len(P, it.q)) {
        it.q += gridDim.x;
        it.j = 0;
    }
}

// ---------------------------------------------------------------- mbarriers
// Shared words: full[kBufs] (stage -> mix), done[kBufs] (mix -> stage), zbar
// (unit sums of the next run's example copied into shared memory).
constexpr uint32_t kFullBar = 0, kDoneBar = 8 * kBufs, kZBar = 16 * kBufs;

// ================================================================ mix role
__device__ void mix_role(const PipeParams &P, unsigned char *sm) {
    set_role_regs<kMixRegs, kLaunchRegs>();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = lane / kGS, lig = lane % kGS;
    const uint32_t lx = (uint32_t)lig << 4;
    const int g = warp * kGPW + h;
    const int R = P.R, kp = P.kp, NP = (R + 1) >> 1, Es = P.Es;
    const int32_t *s_resid = reinterpret_cast<const int32_t *>(sm + P.off_U);
    const uint32_t bars = smem_u32(sm + P.off_bar);
    uint32_t t = 0, run = 0;
    for (TileIter it{blockIdx.x, 0}; it.q < P.runs; ++t) {
        const int b = (int)(t % kBufs);
        if (!mbar_wait(bars + kFullBar + 8 * b, (t / kBufs) & 1u, P.ctrl, it.q)) break;
        const unsigned char *xs = sm + P.off_xs[b];
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys[b]);
        const uint4 *tab = reinterpret_cast<const uint4 *>(sm + P.off_tab[run % kWTabs]);
        // expert pairs: warp w's groups take pairs w + 8h of each block of 32,
        // so the groups' output stores and table reads hit different banks
        for (int blk = 0; blk < NP; blk += kMixWarps * kGPW) {
            const int pr = blk + warp + kMixWarps * h;
            if (pr >= NP) continue;
            const int ea = 2 * pr, eb = ea + 1;
            float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
            float2 b0 = a0, b1 = a0, b2 = a0, b3 = a0;
            // an odd last expert pairs with itself; its twin's result is dropped
            const int ebb = eb < R ? eb : ea;
            mix_entries2(xs, tab + pslot(ea, kp, 0), tab + pslot(ebb, kp, 0), kp >> 1, lx, a0, a1,
                         a2, a3, b0, b1, b2, b3);
            // lane lig's positions are lig + 8 m, m = 0..7
            if (P.bulk_y) {
                // rows of odd length: 16-bit stores
                uint16_t *yh = ys + lig * Es + ea;
                const int st = kGS * Es;
                const float av[8] = {a0.x, a0.y, a1.x, a1.y, a2.x, a2.y, a3.x, a3.y};
                const float bv[8] = {b0.x, b0.y, b1.x, b1.y, b2.x, b2.y, b3.x, b3.y};
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    yh[q * st] = f32_to_bf16(av[q]);
                    yh[q * st + 1] = f32_to_bf16(bv[q]);
                }
            } else {
                uint32_t *yw = reinterpret_cast<uint32_t *>(ys + lig * Es + ea);
                const int st = (kGS * Es) >> 1;
                yw[0 * st] = pack_bf16x2(a0.x, b0.x);
                yw[1 * st] = pack_bf16x2(a0.y, b0.y);
                yw[2 * st] = pack_bf16x2(a1.x, b1.x);
                yw[3 * st] = pack_bf16x2(a1.y, b1.y);
                yw[4 * st] = pack_bf16x2(a2.x, b2.x);
                yw[5 * st] = pack_bf16x2(a2.y, b2.y);
                yw[6 * st] = pack_bf16x2(a3.x, b3.x);
                yw[7 * st] = pack_bf16x2(a3.y, b3.y);
            }
        }
        // residual: group g sums U entries g, g + kGroups, ... for its positions
        if (P.nU > 0) {
            float2 r0 = make_float2(0.f, 0.f), r1 = r0, r2 = r0, r3 = r0;
            for (int u = g; u < P.nU; u += kGroups) {
                const uint32_t c = (uint32_t)s_resid[u];
                const uint4 v = lds128(xs + (((c * kRB) | (((c >> 3) & kFM) << 4)) ^ lx));
                r0 = __fadd2_rn(r0, unpack2(v.x));
                r1 = __fadd2_rn(r1, unpack2(v.y));
                r2 = __fadd2_rn(r2, unpack2(v.z));
                r3 = __fadd2_rn(r3, unpack2(v.w));
            }
            float *rg = reinterpret_cast<float *>(sm + P.off_rp[b]) + g * kRPS + lig;
            rg[0 * kGS] = r0.x; rg[1 * kGS] = r0.y; rg[2 * kGS] = r1.x; rg[3 * kGS] = r1.y;
            rg[4 * kGS] = r2.x; rg[5 * kGS] = r2.y; rg[6 * kGS] = r3.x; rg[7 * kGS] = r3.y;
        }
        // the output tile may leave through the async proxy (bulk copy)
        if (P.bulk_y) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive(bars + kDoneBar + 8 * b);
        const uint32_t q0 = it.q;
        tile_next(P, it);
        run += it.q != q0;
    }
}

// ================================================================ stage role
// Staging: unit u of a tile is two 16-byte loads (positions pa and pa + 8,
// eight channels) that become eight words of the transposed tile
// (stage_x_tile's layout); units are numbered so that a warp's stores are
// conflict-free, and thread st takes units st + kStageT * r.
// A stage thread's units, fixed for the whole launch: position pa of the low
// half (pb = pa + kGS), element offset of the loads in a tile of x, byte
// offset of the stores in a tile buffer (-1: no unit).
struct StageUnits {
    int pa[kStageU], src[kStageU], dst[kStageU];
};

__device__ __forceinline__ StageUnits stage_units(const PipeParams &P, int st) {
    StageUnits su;
    const int CC = P.C >> 3, per_q = 4 * ((CC + 7) & ~7), units = kGS * per_q;
#pragma unroll
    for (int r = 0; r < kStageU; ++r) {
        const int u = st + r * kStageT;
        int q, j, cc;
        stage_unit_coords(u, per_q, P.inv_perq, q, j, cc);
        const bool ok = u < units && cc < CC;
        su.pa[r] = ok ? q + 2 * kGS * j : kTP;
        su.src[r] = su.pa[r] * P.C + cc * 8;
        su.dst[r] = ok ? (cc * 8) * kRB + (((q ^ (cc & kFM)) << 4) | (j << 2)) : -1;
    }
    return su;
}

__device__ __forceinline__ void stage_load(const PipeParams &P, const TileRef &tr,
                                           const StageUnits &su, uint4 *v) {
    const uint16_t *xt = P.x + ((size_t)tr.n * P.HW + tr.p0) * P.C;
#pragma unroll
    for (int r = 0; r < kStageU; ++r) {
        v[2 * r] = su.pa[r] < tr.np ? __ldcs(reinterpret_cast<const uint4 *>(xt + su.src[r]))
                                    : make_uint4(0u, 0u, 0u, 0u);
        v[2 * r + 1] = su.pa[r] + kGS < tr.np
                           ? __ldcs(reinterpret_cast<const uint4 *>(xt + su.src[r] + kGS * P.C))
                           : make_uint4(0u, 0u, 0u, 0u);
    }
}

// Eight words of the transposed tile per unit (layout of stage_x_tile).
__device__ __forceinline__ void stage_store(unsigned char *xs, const StageUnits &su,
                                            const uint4 *v) {
#pragma unroll
    for (int r = 0; r < kStageU; ++r) {
        if (su.dst[r] < 0) continue;
        unsigned char *d = xs + su.dst[r];
        const uint4 va = v[2 * r], vb = v[2 * r + 1];
        *reinterpret_cast<uint32_t *>(d + 0 * kRB) = __byte_perm(va.x, vb.x, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 1 * kRB) = __byte_perm(va.x, vb.x, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 2 * kRB) = __byte_perm(va.y, vb.y, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 3 * kRB) = __byte_perm(va.y, vb.y, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 4 * kRB) = __byte_perm(va.z, vb.z, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 5 * kRB) = __byte_perm(va.z, vb.z, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 6 * kRB) = __byte_perm(va.w, vb.w, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 7 * kRB) = __byte_perm(va.w, vb.w, 0x7632);
    }
}

// ---------------------------------------------------------------- gate (stage role)
// At the start of a run the stage role reduces z[n] from the S tagged unit
// sums of example n (in unit order, one channel per thread) and evaluates the
// gate of every expert: u = z at the support in deployment order,
// h = ReLU(W1 u + b1), g = w2 . h + b2, tau (Eq. (tau)), a = softmax(L / tau)
// (Eq. (weights)). The weights go to the weight fields of one of kWTabs run
// tables (pslot layout; runs use them in turn, so the mix role may still read
// the kBufs previous runs' tables). Every CTA
// with a run of example n evaluates the same gate from the same z (identical
// results); the CTA with the example's first run also writes z and tau to the
// workspace.

// Group of K lanes per expert (k <= K, K = 16 or 32): lane j holds hidden unit
// j and support position j. u is broadcast within the group by shuffles; W1,
// b1 and w2 are zero-padded to K in shared memory, so positions k..K-1 add
// nothing.
template <int K>
__device__ __forceinline__ void gate_groups(const PipeParams &P, const unsigned char *sm,
                                            const float *zs, float *ws_w, int n, bool out) {
    constexpr int kE = 2;                  // experts per group at a time (independent chains)
    constexpr int kNG = kStageT / K;       // groups
    const int st = threadIdx.x - kMixT;
    const int k = P.k, kp = P.kp;
    const int j = st & (K - 1), gi = st / K;
    const float *W1p = reinterpret_cast<const float *>(sm + P.off_W1);
    const float *b1p = reinterpret_cast<const float *>(sm + P.off_b1);
    const float *w2p = reinterpret_cast<const float *>(sm + P.off_w2);
    const int32_t *pidx = P.gate_tabs ? reinterpret_cast<const int32_t *>(sm + P.off_pidx) : P.pidx;
    const float *plog = P.gate_tabs ? reinterpret_cast<const float *>(sm + P.off_plog) : P.plog;
    const float b2 = __ldg(P.b2);
    const bool pos = j < k;
    // lane j's row of W1 (hidden unit j), b1 and w2 stay in registers; row
    // element (i + j) mod K is read at step i, so the lanes hit different banks
    float wr[K];
#pragma unroll
    for (int i = 0; i < K; ++i) wr[i] = W1p[j * K + ((i + j) & (K - 1))];
    const float b1j = b1p[j], w2j = w2p[j];
    for (int e0 = 0; e0 < P.R; e0 += kE * kNG) {
        int e[kE];
        bool act[kE];
        float uj[kE], h[kE];
#pragma unroll
        for (int c = 0; c < kE; ++c) {
            e[c] = e0 + gi + c * kNG;
            act[c] = e[c] < P.R && pos;
            uj[c] = act[c] ? zs[pidx[(size_t)e[c] * k + j]] : 0.f;
            h[c] = b1j;
        }
#pragma unroll
        for (int i = 0; i < K; ++i) {
            const int src = (i + j) & (K - 1);
#pragma unroll
            for (int c = 0; c < kE; ++c)
                h[c] = fmaf(wr[i], __shfl_sync(0xffffffffu, uj[c], src, K), h[c]);
        }
        float gp[kE], L[kE];
#pragma unroll
        for (int c = 0; c < kE; ++c) {
            gp[c] = w2j * fmaxf(h[c], 0.f);
            L[c] = act[c] ? plog[(size_t)e[c] * k + j] : 0.f;
        }
#pragma unroll
        for (int o = K / 2; o > 0; o >>= 1)
#pragma unroll
            for (int c = 0; c < kE; ++c) gp[c] += __shfl_xor_sync(0xffffffffu, gp[c], o, K);
        float ex[kE], zsum[kE];
#pragma unroll
        for (int c = 0; c < kE; ++c) {
            const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-(gp[c] + b2)));
            const float L0 = __shfl_sync(0xffffffffu, L[c], 0, K);  // position 0: largest logit
            ex[c] = act[c] ? expf((L[c] - L0) / tau) : 0.f;
            zsum[c] = ex[c];
            if (out && act[c] && j == 0) P.tau[(size_t)n * P.R + e[c]] = tau;
        }
#pragma unroll
        for (int o = K / 2; o > 0; o >>= 1)
#pragma unroll
            for (int c = 0; c < kE; ++c) zsum[c] += __shfl_xor_sync(0xffffffffu, zsum[c], o, K);
#pragma unroll
        for (int c = 0; c < kE; ++c)
            if (act[c]) ws_w[4 * pslot(e[c], kp, j >> 1) + 2 + (j & 1)] = ex[c] / zsum[c];
    }
}

// Warp per expert for k > 32, a lane per hidden unit (W1 rows padded to ks).
__device__ void gate_warps(const PipeParams &P, unsigned char *sm, const float *zs, float *ws_w,
                           int n, bool out) {
    const int st = threadIdx.x - kMixT;
    const int warp = st >> 5, lane = threadIdx.x & 31;
    float *uw = reinterpret_cast<float *>(sm + P.off_uw) + warp * P.k;
    const float *W1s = reinterpret_cast<const float *>(sm + P.off_W1);
    const float *b1s = reinterpret_cast<const float *>(sm + P.off_b1);
    const float *w2s = reinterpret_cast<const float *>(sm + P.off_w2);
    const int32_t *pidx = P.gate_tabs ? reinterpret_cast<const int32_t *>(sm + P.off_pidx) : P.pidx;
    const float *plog = P.gate_tabs ? reinterpret_cast<const float *>(sm + P.off_plog) : P.plog;
    const int k = P.k, ks = P.ks, kp = P.kp;
    const float b2 = __ldg(P.b2);
    for (int e = warp; e < P.R; e += kStageT / 32) {
        const int32_t *ie = pidx + (size_t)e * k;
        const float *L = plog + (size_t)e * k;
        for (int i = lane; i < k; i += 32) uw[i] = zs[ie[i]];
        __syncwarp();
        float gp = 0.f;
        for (int j = lane; j < k; j += 32) {
            const float *wr = W1s + j * ks;
            float hj = b1s[j];
            for (int i = 0; i < k; ++i) hj = fmaf(wr[i], uw[i], hj);
            gp = fmaf(w2s[j], fmaxf(hj, 0.f), gp);
        }
        const float gv = warp_sum(gp) + b2;
        const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-gv));
        const float L0 = L[0];
        const float ex0 = lane < k ? expf((L[lane] - L0) / tau) : 0.f;
        const float ex1 = lane + 32 < k ? expf((L[lane + 32] - L0) / tau) : 0.f;
        const float zsum = warp_sum(ex0 + ex1);
        if (lane < k) ws_w[4 * pslot(e, kp, lane >> 1) + 2 + (lane & 1)] = ex0 / zsum;
        if (lane + 32 < k) ws_w[4 * pslot(e, kp, (lane + 32) >> 1) + 2 + (lane & 1)] = ex1 / zsum;
        if (out && lane == 0) P.tau[(size_t)n * P.R + e] = tau;
        __syncwarp();
    }
}

// Starts the copy of example n's unit sums ([S][C] tagged words, contiguous)
// into zbuf; the next stage_gate waits for it on zbar.
__device__ __forceinline__ void zsum_prefetch(const PipeParams &P, unsigned char *sm, int n) {
    const uint32_t bytes = (uint32_t)P.S * (uint32_t)P.C * 8u;
    const unsigned long long *src = P.part + (size_t)n * P.S * P.C;
    asm volatile(
        "mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t"
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%2], [%3], %1, [%0];"
        ::"r"(smem_u32(sm + P.off_bar) + kZBar), "r"(bytes), "r"(smem_u32(sm + P.off_zbuf)), "l"(src)
        : "memory");
}

// z and the weights of example n into shared memory (zs, ws_w), from the unit
// sums copied into zbuf (phase zph of zbar); a sum that was not yet written
// when it was copied is read again from the workspace. False when a wait gave
// up (the same on every stage thread).
__device__ bool stage_gate(const PipeParams &P, unsigned char *sm, int n, bool out, uint32_t ready,
                           uint32_t item, float *ws_w, uint32_t zph) {
    const int st = threadIdx.x - kMixT;
    float *zs = reinterpret_cast<float *>(sm + P.off_zs);
    const unsigned long long *zb = reinterpret_cast<const unsigned long long *>(sm + P.off_zbuf);
    bool ok = mbar_wait(smem_u32(sm + P.off_bar) + kZBar, zph, P.ctrl, item);
    for (int c = st; c < P.C && ok; c += kStageT) {
        const unsigned long long *pc = P.part + (size_t)n * P.S * P.C + c;
        unsigned long long v[kMaxUnits];
        bool fresh = true;
#pragma unroll
        for (int s = 0; s < kMaxUnits; ++s) {
            v[s] = s < P.S ? zb[s * P.C + c] : 0ull;
            fresh = fresh && (s >= P.S || tag_ok(v[s], ready));
        }
        // sums that were not written when they were copied are read again, all
        // of them at once, until they are (bounded)
        for (uint32_t it = 0; !fresh && ok; ++it) {
            if (it >= kSpinLimit) {
                report_timeout(P.ctrl, item);
                ok = false;
                break;
            }
            if (it > 0) {
                if (ld_relaxed(P.ctrl + kCtrlError) != 0u) { ok = false; break; }
                __nanosleep(128);
            }
            fresh = true;
#pragma unroll
            for (int s = 0; s < kMaxUnits; ++s)
                if (s < P.S && !tag_ok(v[s], ready)) v[s] = ld_tagged(pc + (size_t)s * P.C);
#pragma unroll
            for (int s = 0; s < kMaxUnits; ++s) fresh = fresh && (s >= P.S || tag_ok(v[s], ready));
        }
        float sum = 0.f;
#pragma unroll
        for (int s = 0; s < kMaxUnits; ++s)
            if (s < P.S) sum += tag_val(v[s]);
        const float zv = sum / (float)P.HW;
        zs[c] = zv;
        if (out) P.z[(size_t)n * P.C + c] = zv;
    }
    // zbuf was read through the generic proxy; the next copy into it is async
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (!bar_and(kBarStage, kStageT, ok)) return false;
    if (P.k <= 16) gate_groups<16>(P, sm, zs, ws_w, n, out);
    else if (P.k <= 32) gate_groups<32>(P, sm, zs, ws_w, n, out);
    else gate_warps(P, sm, zs, ws_w, n, out);
    bar_sync(kBarStage, kStageT);  // zs is free again and ws_w is complete
    return true;
}

// Residual column from the groups' partial sums, then the [np][E] output
// block (contiguous in y) with 16-byte streaming stores.
__device__ void copy_tile(const PipeParams &P, unsigned char *sm, int b, const TileRef &tr, int st) {
    const int R = P.R, E = R + 1, Es = P.Es;
    uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys[b]);
    const float *rp = reinterpret_cast<const float *>(sm + P.off_rp[b]);
    {
        // the residual column: four lanes per position add a quarter of the
        // groups' partial sums each
        static_assert(kStageT == 4 * kTP, "four stage lanes per position");
        const int px = st >> 2, part = st & 3;
        float s = 0.f;
        if (P.nU > 0) {
#pragma unroll
            for (int gg = part; gg < kGroups; gg += 4) s += rp[gg * kRPS + px];
            s += __shfl_xor_sync(0xffffffffu, s, 1);
            s += __shfl_xor_sync(0xffffffffu, s, 2);
            s = s / (float)P.nU;
        }
        if (part == 0 && px < tr.np) ys[px * Es + R] = f32_to_bf16(s);
    }
    const int cnt = tr.np * E;
    uint16_t *dst = P.y + ((size_t)tr.n * P.HW + tr.p0) * E;
    if (P.bulk_y) {
        // [np][E] is contiguous in shared memory and in y: one bulk copy
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        bar_sync(kBarStage, kStageT);
        if (st == 0) {
            asm volatile(
                "cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n\t"
                "cp.async.bulk.commit_group;" ::"l"(dst),
                "r"(smem_u32(ys)), "r"((uint32_t)cnt * 2u)
                : "memory");
        }
        return;
    }
    bar_sync(kBarStage, kStageT);
    const int head =
        min(cnt, (int)(((16u - ((uint32_t)reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u) >> 1));
    for (int o = st; o < head; o += kStageT) {
        const int p = fdiv(o, E, P.inv_E);
        __stcs(dst + o, ys[p * Es + (o - p * E)]);
    }
    const int nv = (cnt - head) >> 3;
    for (int v = st; v < nv; v += kStageT) {
        const int o = head + v * 8;
        int p = fdiv(o, E, P.inv_E), e = o - p * E;
        uint32_t w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t lo = ys[p * Es + e];
            if (++e == E) { e = 0; ++p; }
            const uint32_t hi = ys[p * Es + e];
            if (++e == E) { e = 0; ++p; }
            w[q] = lo | (hi << 16);
        }
        __stcs(reinterpret_cast<uint4 *>(dst + o), make_uint4(w[0], w[1], w[2], w[3]));
    }
    for (int o = head + nv * 8 + st; o < cnt; o += kStageT) {
        const int p = fdiv(o, E, P.inv_E);
        __stcs(dst + o, ys[p * Es + (o - p * E)]);
    }
}

__device__ void stage_role(const PipeParams &P, unsigned char *sm, uint32_t ready) {
    set_role_regs<kStageRegs, kLaunchRegs>();
    const int st = threadIdx.x - kMixT;
    const uint32_t bars = smem_u32(sm + P.off_bar);
    uint4 pre[2 * kStageU];
    const StageUnits su = stage_units(P, st);
    TileIter it{blockIdx.x, 0};
    TileRef prev[kBufs];  // tiles held by the buffers
    uint32_t t = 0, run = 0;
    uint32_t zissued = 0;  // unit-sum copies started (run r's copy is phase r of zbar)
    bool alive = true;
    if (it.q < P.runs) {
        const TileRef tr = tile_of(P, it);
        if (st == 0) zsum_prefetch(P, sm, tr.n);
        zissued = 1;
        alive = stage_gate(P, sm, tr.n, it.q % (uint32_t)P.RN == 0, ready, it.q,
                           reinterpret_cast<float *>(sm + P.off_tab[0]), 0u);
        // the unit sums of the next run's example arrive while this run is mixed
        if (alive && it.q + gridDim.x < P.runs) {
            if (st == 0) zsum_prefetch(P, sm, (int)((it.q + gridDim.x) / (uint32_t)P.RN));
            zissued = 2;
        }
        stage_load(P, tr, su, pre);
    }
    for (; alive && it.q < P.runs; ++t) {
        const int b = (int)(t % kBufs);
        const TileRef tr = tile_of(P, it);
        if (t >= kBufs) {
            // buffer b held tile t - kBufs: once mixed, write it out
            const bool ok =
                mbar_wait(bars + kDoneBar + 8 * b, ((t - kBufs) / kBufs) & 1u, P.ctrl, it.q);
            if (!bar_and(kBarStage, kStageT, ok)) { alive = false; break; }
            copy_tile(P, sm, b, prev[b], st);
        }
        prev[b] = tr;
        stage_store(sm + P.off_xs[b], su, pre);
        // the bulk copy of tile t - kBufs has read ys[b] before mix may overwrite it
        if (P.bulk_y && st == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        mbar_arrive(bars + kFullBar + 8 * b);
        const uint32_t q0 = it.q;
        tile_next(P, it);
        if (it.q < P.runs) {
            const TileRef nt = tile_of(P, it);
            // a new run: its gate first (no prefetched data live across it), into
            // a run table that none of the runs still in the buffers use
            if (it.q != q0) {
                ++run;
                if (!stage_gate(P, sm, nt.n, it.q % (uint32_t)P.RN == 0, ready, it.q,
                                reinterpret_cast<float *>(sm + P.off_tab[run % kWTabs]), run & 1u)) {
                    alive = false;
                    break;
                }
                if (it.q + gridDim.x < P.runs) {
                    if (st == 0) zsum_prefetch(P, sm, (int)((it.q + gridDim.x) / (uint32_t)P.RN));
                    zissued = run + 2;
                }
            }
            stage_load(P, nt, su, pre);
        }
    }
    if (alive) {
        // the last tiles
        for (uint32_t tt = t >= kBufs ? t - kBufs : 0; tt < t; ++tt) {
            const int b = (int)(tt % kBufs);
            const bool ok = mbar_wait(bars + kDoneBar + 8 * b, (tt / kBufs) & 1u, P.ctrl, blockIdx.x);
            if (!bar_and(kBarStage, kStageT, ok)) break;
            copy_tile(P, sm, b, prev[b], st);
        }
    }
    // bulk copies complete before the CTA exits: the output tiles, and a
    // unit-sum copy that an early exit left unread (phase zissued - 1)
    if (st == 0) {
        if (P.bulk_y) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
        if (!alive && zissued > 0) {
            const uint32_t zb = smem_u32(sm + P.off_bar) + kZBar;
            for (uint32_t i = 0; i < kSpinLimit && !mbar_test(zb, (zissued - 1) & 1u); ++i)
                __nanosleep(256);
        }
    }
}

// ================================================================ pool role
// Example n is pooled as S slices of consecutive positions (units u = n*S + s,
// CTA u mod G). Pool warp w owns 8-channel blocks [w*cpw, (w+1)*cpw); lane l
// reads block w*cpw + l % cpw of rows r, r + rpi, r + 2 rpi, ... of the unit,
// with r = l / cpw and rpi = 32 / cpw rows per warp load. A unit is read in
// blocks of kPoolWin steps (rows past its end read nothing) with every
// consumed load replaced at once by the one kPoolWin steps ahead; the last
// block of a unit prefetches the first rows of the next. The loops carry no
// branches, so the loads stay in flight. At the end of a unit the warp adds
// its rows together with shuffles and the lanes with r == 0 write the unit's
// channel sums as tagged words.
__device__ __forceinline__ int unit_begin(const PipeParams &P, int s) {
    return (int)(((long long)s * P.HW) / P.S);
}

struct PoolUnit {
    uint32_t u;
    int p, pe;             // this lane's first row, end of the unit
    const uint16_t *base;  // x of the unit's example at this lane's channel block
};

__device__ __forceinline__ PoolUnit pool_unit(const PipeParams &P, uint32_t u, int r, int blk) {
    PoolUnit c;
    c.u = u;
    c.p = 0;
    c.pe = 0;
    c.base = P.x;
    if (u < P.pool_items) {
        const int n = (int)(u / (uint32_t)P.S), s = (int)(u - (uint32_t)n * P.S);
        const int p0 = unit_begin(P, s);
        c.pe = unit_begin(P, s + 1);
        c.p = p0 + r;
        c.base = P.x + (size_t)n * P.HW * P.C + blk * 8;
    }
    return c;
}

// Loads of step block bi of unit c (rows past the end read nothing).
__device__ __forceinline__ void pool_block_load(const PipeParams &P, const PoolUnit &c, int bi,
                                                bool own, uint4 *v) {
    const int row0 = c.p + bi * kPoolWin * P.rpi;
#pragma unroll
    for (int d = 0; d < kPoolWin; ++d) {
        const int row = row0 + d * P.rpi;
        v[d] = (own && row < c.pe) ? ld_stream(c.base + (size_t)row * P.C) : make_uint4(0u, 0u, 0u, 0u);
    }
}

__device__ __forceinline__ void add8(float2 *acc, const uint4 v) {
    acc[0] = __fadd2_rn(acc[0], unpack2(v.x));
    acc[1] = __fadd2_rn(acc[1], unpack2(v.y));
    acc[2] = __fadd2_rn(acc[2], unpack2(v.z));
    acc[3] = __fadd2_rn(acc[3], unpack2(v.w));
}

// Consumes the window v and refills it from block bi of unit c.
__device__ __forceinline__ void pool_block(const PipeParams &P, const PoolUnit &c, int bi, bool own,
                                           uint4 *v, float2 *acc) {
    const int row0 = c.p + bi * kPoolWin * P.rpi;
#pragma unroll
    for (int d = 0; d < kPoolWin; ++d) {
        add8(acc, v[d]);
        const int row = row0 + d * P.rpi;
        v[d] = (own && row < c.pe) ? ld_stream(c.base + (size_t)row * P.C) : make_uint4(0u, 0u, 0u, 0u);
    }
}

// End of unit u for this warp: rows combined, channel sums written tagged.
__device__ __forceinline__ void unit_flush(const PipeParams &P, uint32_t u, float2 *acc, int lane,
                                          int blk, bool own, uint32_t ready, uint32_t drop) {
    float f[8] = {acc[0].x, acc[0].y, acc[1].x, acc[1].y, acc[2].x, acc[2].y, acc[3].x, acc[3].y};
    for (int o = P.cpw; o < 32; o <<= 1) {
#pragma unroll
        for (int q = 0; q < 8; ++q) f[q] += __shfl_xor_sync(0xffffffffu, f[q], o);
    }
    if (own && lane < P.cpw && u + 1u != drop) {
        const int n = (int)(u / (uint32_t)P.S), s = (int)(u - (uint32_t)n * P.S);
        unsigned long long *dst = P.part + ((size_t)n * P.S + s) * P.C + blk * 8;
#pragma unroll
        for (int q = 0; q < 8; ++q) st_tagged(dst + q, f[q], ready);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] = make_float2(0.f, 0.f);
}

__device__ void pool_role(const PipeParams &P, uint32_t ready, uint32_t drop) {
    set_role_regs<kPoolRegs, kLaunchRegs>();
    const int pw = (threadIdx.x - kMixT - kStageT) >> 5, lane = threadIdx.x & 31;
    const int blk = pw * P.cpw + (lane & (P.cpw - 1)), r = lane / P.cpw;
    const bool own = blk < (P.C >> 3);
    PoolUnit cur = pool_unit(P, blockIdx.x, r, blk);
    uint4 v[kPoolWin];
    pool_block_load(P, cur, 0, own, v);
    float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                     make_float2(0.f, 0.f)};
    while (cur.u < P.pool_items) {
        const PoolUnit nxt = pool_unit(P, cur.u + gridDim.x, r, blk);
        // blocks of kPoolWin steps of the unit (its rows start at cur.p - r)
        const int blocks = (cur.pe - (cur.p - r) + P.rpi * kPoolWin - 1) / (P.rpi * kPoolWin);
        for (int bi = 1; bi < blocks; ++bi) pool_block(P, cur, bi, own, v, acc);
        pool_block(P, nxt, 0, own, v, acc);  // the next unit's first block
        unit_flush(P, cur.u, acc, lane, blk, own, ready, drop);
        cur = nxt;
    }
}

// ================================================================ the kernel
__global__ void __launch_bounds__(kPipeT, 1) moce_pipe_kernel(const PipeParams P) {
    extern __shared__ __align__(128) unsigned char sm[];
    const uint32_t epoch = ld_relaxed(P.ctrl + kCtrlEpoch);
    const uint32_t ready = epoch + 1u;
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    if (threadIdx.x >= kMixT + kStageT) {
        // the pool role needs none of the shared data below: it starts at once
        pool_role(P, ready, drop);
    } else {
        // data that stays for the whole launch (mix and stage roles): U list,
        // gate parameters and support tables, the zero row of both x buffers,
        // the run tables' row offsets (weights start at zero)
        int32_t *s_resid = reinterpret_cast<int32_t *>(sm + P.off_U);
        for (int i = threadIdx.x; i < P.nU; i += kMixT + kStageT) s_resid[i] = __ldg(P.resid + i);
        float *W1s = reinterpret_cast<float *>(sm + P.off_W1);
        if (P.Kg) {
            // group gate: W1 as [Kg][Kg], b1 and w2 as [Kg], zero-padded
            for (int q = threadIdx.x; q < P.Kg * P.Kg; q += kMixT + kStageT) {
                const int j = q / P.Kg, i = q - j * P.Kg;
                W1s[q] = (j < P.k && i < P.k) ? __ldg(P.W1 + j * P.k + i) : 0.f;
            }
            for (int j = threadIdx.x; j < P.Kg; j += kMixT + kStageT) {
                reinterpret_cast<float *>(sm + P.off_b1)[j] = j < P.k ? __ldg(P.b1 + j) : 0.f;
                reinterpret_cast<float *>(sm + P.off_w2)[j] = j < P.k ? __ldg(P.w2 + j) : 0.f;
            }
        } else {
            // warp gate: W1 rows padded to ks
            for (int q = threadIdx.x; q < P.k * P.k; q += kMixT + kStageT) {
                const int j = q / P.k, i = q - j * P.k;
                W1s[j * P.ks + i] = __ldg(P.W1 + q);
            }
            for (int j = threadIdx.x; j < P.k; j += kMixT + kStageT) {
                reinterpret_cast<float *>(sm + P.off_b1)[j] = __ldg(P.b1 + j);
                reinterpret_cast<float *>(sm + P.off_w2)[j] = __ldg(P.w2 + j);
            }
        }
        if (P.gate_tabs) {
            for (int q = threadIdx.x; q < P.R * P.k; q += kMixT + kStageT) {
                reinterpret_cast<int32_t *>(sm + P.off_pidx)[q] = __ldg(P.pidx + q);
                reinterpret_cast<float *>(sm + P.off_plog)[q] = __ldg(P.plog + q);
            }
        }
        for (int q = threadIdx.x; q < kBufs * (kRB / 4); q += kMixT + kStageT) {
            const int b = q / (kRB / 4), w = q - b * (kRB / 4);
            reinterpret_cast<uint32_t *>(sm + P.off_xs[b] + (size_t)P.C * kRB)[w] = 0u;
        }
        for (int q = threadIdx.x; q < P.R * P.kp; q += kMixT + kStageT) {
            const int el = q / P.kp, i = q - el * P.kp;
            uint32_t off = (uint32_t)P.C * kRB;  // padding entries read the zero row
            if (i < P.k) {
                const uint32_t c = (uint32_t)__ldg(P.pidx + (size_t)el * P.k + i);
                off = (c * kRB) | (((c >> 3) & kFM) << 4);
            }
            for (int b = 0; b < kWTabs; ++b) {
                uint32_t *w = reinterpret_cast<uint32_t *>(
                    reinterpret_cast<uint4 *>(sm + P.off_tab[b]) + pslot(el, P.kp, i >> 1));
                w[i & 1] = off;
                w[2 + (i & 1)] = 0u;
            }
        }
        if (threadIdx.x == 0) {
            const uint32_t bars = smem_u32(sm + P.off_bar);
            for (int b = 0; b < kBufs; ++b) {
                mbar_init(bars + kFullBar + 8 * b, kStageT);
                mbar_init(bars + kDoneBar + 8 * b, kMixT);
            }
            mbar_init(bars + kZBar, 1);
            // zbar completes through the async proxy (bulk copies)
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        bar_sync(kBarPrologue, kMixT + kStageT);

        if (threadIdx.x < kMixT) mix_role(P, sm);
        else stage_role(P, sm, ready);
    }

    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t old = atomicAdd(P.ctrl + kCtrlExitCounter, 1u);
        if (old == gridDim.x - 1u) {
            P.ctrl[kCtrlExitCounter] = 0u;
            P.ctrl[kCtrlEpoch] = epoch + 1u;
            __threadfence();
        }
    }
}

// ---------------------------------------------------------------- host side
struct PipePlan {
    int kp = 0, Es = 0, ks = 0, Kg = 0;
    bool gate_tabs = false;
    size_t off_xs[kBufs] = {}, off_ys[kBufs] = {}, off_rp[kBufs] = {}, off_tab[kWTabs] = {};
    size_t off_zs = 0, off_zbuf = 0, off_uw = 0, off_W1 = 0, off_b1 = 0, off_w2 = 0;
    size_t off_pidx = 0, off_plog = 0, off_U = 0, off_bar = 0, smem = 0;
};

// Shared memory: kBufs x buffers of C + 1 rows (row C = zeros), kBufs output
// tiles and residual partial blocks, kWTabs run tables, the gate's z and unit-sum copy, the gate parameters, [support
// tables,] U, mbarriers.
bool pipe_plan(int C, int R, int k, PipePlan *plan) {
    // C <= 256: every staging unit of a tile has its thread (kStageU per thread)
    if (C % 8 != 0 || C < 8 || C > 256 || k < 1 || k > kGateMaxK || R < 1) return false;
    PipePlan p;
    p.kp = k + (k & 1);
    p.Es = (R + 1) + ((R + 1) & 1);
    p.ks = (k % 2 == 0) ? k + 1 : k;
    p.Kg = k <= 16 ? 16 : (k <= 32 ? 32 : 0);
    size_t off = 0;
    auto take = [&](size_t bytes, size_t al) {
        off = align_up(off, al);
        const size_t o = off;
        off += bytes;
        return o;
    };
    for (int b = 0; b < kBufs; ++b) p.off_xs[b] = take((size_t)(C + 1) * kRB, 128);
    for (int b = 0; b < kBufs; ++b) p.off_ys[b] = take((size_t)kTP * p.Es * 2, 16);
    for (int b = 0; b < kBufs; ++b) p.off_rp[b] = take((size_t)kGroups * kRPS * 4, 16);
    for (int b = 0; b < kWTabs; ++b) p.off_tab[b] = take((size_t)pslot_count(R, p.kp) * 16, 16);
    p.off_zs = take((size_t)C * 4, 16);
    p.off_zbuf = take((size_t)kMaxUnits * C * 8, 128);
    p.off_uw = take((size_t)(kStageT / 32) * k * 4, 16);
    const int kg = p.Kg ? p.Kg : k;
    p.off_W1 = take((size_t)(p.Kg ? p.Kg * p.Kg : k * p.ks) * 4, 16);
    p.off_b1 = take((size_t)kg * 4, 16);
    p.off_w2 = take((size_t)kg * 4, 16);
    p.gate_tabs = (size_t)R * k * 8 <= 16 * 1024;
    if (p.gate_tabs) {
        p.off_pidx = take((size_t)R * k * 4, 16);
        p.off_plog = take((size_t)R * k * 4, 16);
    }
    p.off_U = take((size_t)C * 4, 16);
    p.off_bar = take(16 * kBufs + 8, 8);
    p.smem = off;
    if (p.smem > 227 * 1024) return false;
    *plan = p;
    return true;
}

// Pooling units (slices) per example: about 3 x PP positions per unit, with
// N * S close to a whole number of rounds of the G CTAs; at most PT (the
// unit-sum region of the workspace holds PT per example, and z reads all S
// at once).
int pool_units_per_example(int N, int HW, int PP, int PT, int G) {
    const long long px = (long long)N * HW;
    const long long m0 = std::max(1LL, (px + (long long)G * 3 * PP - 1) / ((long long)G * 3 * PP));
    int best = 1;
    double best_eff = -1.0;
    for (long long m = m0; m <= 4 * m0; ++m) {
        const long long S = std::min<long long>(PT, (m * G + N - 1) / N);
        const long long units = (long long)N * S;
        const double eff = (double)units / (double)(((units + G - 1) / G) * G);
        if (eff > best_eff + 1e-9) {
            best_eff = eff;
            best = (int)S;
        }
        if (eff >= 0.97) break;
    }
    return best < 1 ? 1 : best;
}

}  // namespace

bool pipe_supported(int N, int HW, int C, int R, int k) {
    (void)N;
    (void)HW;
    PipePlan plan;
    return pipe_plan(C, R, k, &plan);
}

cudaError_t launch_pipe(const uint16_t *x, int N, int HW, int C, int R, int k,
                        const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                        const float *W1, const float *b1, const float *w2, const float *b2,
                        float tmin, float tmax, uint16_t *y, const WsLayout &L, unsigned char *ws,
                        cudaStream_t s) {
    PipePlan plan;
    if (!pipe_plan(C, R, k, &plan)) return cudaErrorNotSupported;
    PipeParams P;
    P.x = x;
    P.y = y;
    P.N = N;
    P.HW = HW;
    P.C = C;
    P.R = R;
    P.k = k;
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
    P.ctrl = reinterpret_cast<uint32_t *>(ws + L.ctrl);
    P.part = reinterpret_cast<unsigned long long *>(ws + L.partial);
    P.z = reinterpret_cast<float *>(ws + L.z);
    P.tau = reinterpret_cast<float *>(ws + L.tau);
    P.MT = (HW + kTP - 1) / kTP;
    P.RN = (P.MT + kRun - 1) / kRun;
    const unsigned long long runs = (unsigned long long)N * P.RN;
    if (runs >= 0xffff0000ull) return cudaErrorInvalidValue;
    P.runs = (uint32_t)runs;
    // pool: 8-channel blocks per warp (a power of two), rows per warp load
    {
        const int per = ((C >> 3) + kPoolWarps - 1) / kPoolWarps;
        int cpw = 1;
        while (cpw < per) cpw <<= 1;
        P.cpw = cpw;
        P.rpi = 32 / cpw;
    }
    P.kp = plan.kp;
    P.Es = plan.Es;
    P.ks = plan.ks;
    P.Kg = plan.Kg;
    // every output tile [np][R + 1] starts and ends on a 16-byte boundary of y
    // when HW * (R + 1) is a multiple of 8: it leaves by one bulk copy
    P.bulk_y = ((long long)HW * (R + 1)) % 8 == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0;
    if (P.bulk_y) P.Es = R + 1;
    P.gate_tabs = plan.gate_tabs ? 1 : 0;
    for (int b = 0; b < kBufs; ++b) {
        P.off_xs[b] = (uint32_t)plan.off_xs[b];
        P.off_ys[b] = (uint32_t)plan.off_ys[b];
        P.off_rp[b] = (uint32_t)plan.off_rp[b];
    }
    P.off_zs = (uint32_t)plan.off_zs;
    P.off_zbuf = (uint32_t)plan.off_zbuf;
    for (int b = 0; b < kWTabs; ++b) P.off_tab[b] = (uint32_t)plan.off_tab[b];
    P.off_uw = (uint32_t)plan.off_uw;
    P.off_W1 = (uint32_t)plan.off_W1;
    P.off_b1 = (uint32_t)plan.off_b1;
    P.off_w2 = (uint32_t)plan.off_w2;
    P.off_pidx = (uint32_t)plan.off_pidx;
    P.off_plog = (uint32_t)plan.off_plog;
    P.off_U = (uint32_t)plan.off_U;
    P.off_bar = (uint32_t)plan.off_bar;
    P.inv_perq = 1.0f / (float)(4 * (((C >> 3) + 7) & ~7));
    P.inv_E = 1.0f / (float)(R + 1);
    P.inv_kp = 1.0f / (float)plan.kp;

    cudaError_t err = cudaFuncSetAttribute(moce_pipe_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)plan.smem);
    if (err != cudaSuccess) return err;
    int dev = 0, sms = 0, per_sm = 0;
    if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
    if ((err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return err;
    if ((err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, moce_pipe_kernel, kPipeT,
                                                             plan.smem)) != cudaSuccess)
        return err;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const int G = sms * per_sm;
    P.S = pool_units_per_example(N, HW, 64, std::min(L.pool_tiles, kMaxUnits), G);
    const unsigned long long pool_items = (unsigned long long)N * P.S;
    if (pool_items >= 0xffff0000ull) return cudaErrorInvalidValue;
    P.pool_items = (uint32_t)pool_items;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)moce_pipe_kernel, dim3(G),
                                       dim3(kPipeT), args, plan.smem, s);
}

}  // namespace moce
