// Resident-tile persistent forward kernel of a MoCE layer (Sec. 3.3-3.4):
// pooling, gate, softmax weights, routed mixing and the residual expert in
// one launch that reads x from HBM once, for NHWC bf16 layers with
// C_in <= 256.
//
// Every expert's temperature depends on the whole-image average of its
// support (Sec. 3.3), so no position of an example can be mixed before all
// of the example has been pooled. The example is cut into tiles of 64
// positions: tile t of example n is work item n*T + t, and CTA b (one per SM,
// all resident: cooperative launch) takes items b, b + G, b + 2G, ... A tile
// stays in the CTA's shared memory, transposed to channel-major rows, from
// the moment it is read until it has been mixed: a ring of D slots holds the
// CTA's next tiles while the examples they belong to are being pooled by
// the other CTAs. Four warp roles:
//
//   load     (warps 12-27) reads tiles with 16-byte loads (two tiles ahead),
//            stores each transposed into a free slot and leaves its partial
//            channel sums in shared memory. It touches no other global
//            memory, so nothing it does waits for its loads in flight.
//   publish  (warp 8) adds the partial sums, publishes the tile's channel
//            sums (fp32 for the exact fallback, and as 64-bit fixed-point
//            integers added into the example's accumulator) and counts the
//            tile into the example's arrival counter.
//   fetch    (warp 9) waits until every tile of its item's example is
//            counted and reads z from the accumulator (integer sums do not
//            depend on the order of the additions: z is deterministic) into
//            one of two z buffers, one item ahead of the gate.
//   gate     (warps 10-11) evaluates the gate of every expert (Eq. (tau))
//            and the softmax weights (Eq. (weights)) straight into one of
//            two mixing tables.
//   mix      (warps 0-7) mixes a slot with its table: each group of 8 lanes
//            owns 8 positions per lane and an expert pair (Eq. (expert)) plus
//            a slice of the residual sum (Eq. (res)); it writes the tile of y
//            into one of two output buffers and sends it to HBM with one bulk
//            copy.
//
// The roles hand slots, sums and tables over through shared-memory
// mbarriers; in each role one thread waits and the others block at a
// barrier. Every wait is bounded: one that gives up records MOCE_ERR_TIMEOUT
// in the workspace and every other wait returns. The only wait between CTAs
// is the fetch role's wait for an arrival count; the publish role that
// counts waits only for its own CTA's loads, so the waits form no cycle.
//
// The accumulators and counters of a forward are zeroed by the forward
// before it (two sets, chosen by the parity of the forward's epoch), so no
// CTA has to wait for the others to finish reading them.
#include <algorithm>

#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kTP = kRingTile;        // positions per tile
constexpr int kGS = 8;                // lanes of a mixing group
constexpr int kGPW = 32 / kGS;        // mixing groups per warp
constexpr int kRB = 16 * kGS;         // bytes per staged channel row (kTP bf16)
constexpr int kFM = 7;                // chunk swizzle mask of the staged rows
constexpr int kMixT = 256;            // mix role: warps 0-7
constexpr int kPubT = 32;             // publish role: warp 8
constexpr int kFetchT = 32;           // fetch role: warp 9
constexpr int kGateT = 64;            // gate role: warps 10-11
constexpr int kLoadT = 512;           // load role: warps 12-27
constexpr int kRingT = kMixT + kPubT + kFetchT + kGateT + kLoadT;
constexpr int kGate0 = kMixT + kPubT + kFetchT;  // first gate thread
constexpr int kLoad0 = kGate0 + kGateT;          // first load thread
constexpr int kMixWarps = kMixT / 32;
constexpr int kGroups = kMixT / kGS;  // mixing groups per CTA
constexpr int kRPS = kTP + 8;         // row stride (floats) of the residual partial sums
constexpr int kNT = 2;                // mixing tables
constexpr int kYB = 2;                // output tile buffers
constexpr int kNB = 2;                // partial-sum blocks between load and publish
constexpr int kMaxD = 6;              // x slots at most
constexpr int kRedF = 1024;           // floats of a partial-sum block
constexpr int kGateMaxK = 64;
constexpr int kBarMix = 1, kBarGate = 2, kBarLoad = 3;
// Fixed-point scale of the pooled sums: 2^24. A tile sum of magnitude at
// most 2^38 / T keeps the example's integer sum within int64; a larger one
// marks the example for the exact fp32 reduction instead.
constexpr float kFixScale = 16777216.0f;
constexpr float kFixInv = 1.0f / 16777216.0f;
static_assert(kRingT * 72 <= 65536, "72 registers per thread at one CTA per SM");
static_assert(kMixT == 4 * kTP, "four mixing threads per position in the epilogue");
static_assert(kTP == 8 * kGS, "a group's lanes cover the tile");

// mbarriers (8 bytes each, one arrival each): full[s] (load -> mix),
// empty[s] (mix -> load), pooled[b] (load -> publish), rfree[b] (publish ->
// load), tready[b] (gate -> mix), tfree[b] (mix -> gate), zready[b] (fetch
// -> gate), zfree[b] (gate -> fetch).
constexpr int kMbFull = 0, kMbEmpty = kMaxD, kMbPooled = 2 * kMaxD, kMbRFree = 2 * kMaxD + kNB,
              kMbTReady = 2 * kMaxD + 2 * kNB, kMbTFree = 2 * kMaxD + 2 * kNB + kNT,
              kMbZReady = 2 * kMaxD + 2 * kNB + 2 * kNT,
              kMbZFree = 2 * kMaxD + 2 * kNB + 3 * kNT, kMbWords = 2 * kMaxD + 2 * kNB + 4 * kNT;

struct RingParams {
    const uint16_t *x;
    uint16_t *y;
    int N, HW, C, R, k, nU, T;
    uint32_t items;               // N * T tiles
    const int32_t *pidx;
    const float *plog;
    const int32_t *resid;
    const float *W1, *b1, *w2, *b2;
    float tmin, tmax;
    uint32_t *ctrl;
    float *part;                  // [N][T][C] tile channel sums (exact fallback)
    unsigned long long *zacc;     // [2][N][C] fixed-point channel sums of the examples
    uint32_t *count;              // [2][N] tiles of example n counted
    uint32_t *ovf;                // [2][N] a tile sum of example n was beyond the fixed-point range
    float *z, *tau;
    int D;                        // x slots
    int CG, nrow;                 // load role: 64-channel groups (1, 2, 4), partial-sum rows
    int kp, Es, ks, Kg;           // Kg: padded gate width (16, 32), 0: a warp per expert
    int RS;                       // entries per support position of a mixing table (tslot)
    int bulk_y;                   // output tiles leave by one bulk copy
    int gate_tabs;                // support tables of the gate in shared memory, [k][R]
    float fix_max;                // largest tile sum magnitude for the fixed-point path
    uint32_t off_xs, xs_bytes;
    uint32_t off_tab[kNT], off_ys[kYB];
    uint32_t off_rp, off_red, off_zs, off_uw, off_W1, off_b1, off_w2, off_pidx, off_plog, off_U,
        off_bar;
    float inv_E;
};

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_add_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
// Bounded wait until *p == want. False when this or another wait gave up.
__device__ bool wait_count(const uint32_t *p, uint32_t want, uint32_t *ctrl, uint32_t item) {
    for (uint32_t it = 0; it < kSpinLimit; ++it) {
        if (ld_acquire(p) == want) return true;
        if (ld_relaxed(ctrl + kCtrlError) != 0u) return false;
        __nanosleep(it < 64 ? 32 : 256);
    }
    report_timeout(ctrl, item);
    return false;
}

__device__ __forceinline__ uint32_t mbar(const RingParams &P, const unsigned char *sm, int word) {
    return smem_u32(sm + P.off_bar) + 8u * (uint32_t)word;
}

// Entry (uint4 units) of support positions (2 i2, 2 i2 + 1) of expert e in a
// mixing table {row offset, row offset, weight, weight}. Entries are grouped
// by position: a gate warp writing one position of 32 experts touches
// consecutive entries, and the block of 16 experts shifts the entries by
// one, so the four lane groups of a mixing warp (experts 16 apart) read
// different banks.
__device__ __host__ __forceinline__ int tslot(int RS, int e, int i2) { return i2 * RS + e + (e >> 4); }
__host__ inline int tslot_rows(int R) { return R + (R >> 4) + 1; }

// Support table element (e, i): [k][R] in shared memory or [R][k] in global.
struct SupTab {
    const int32_t *idx;
    const float *lg;
    int se, si;
    __device__ __forceinline__ int at(int e, int i) const { return e * se + i * si; }
};

// ================================================================ gate role
// Gate of every expert of one example (Eq. (tau)): u = z at the expert's
// support in deployment order, h = ReLU(W1 u + b1), g = w2 . h + b2,
// tau = tau_min + (tau_max - tau_min) sigma(g); weights a = softmax(L / tau)
// (Eq. (weights)), written into a mixing table. A thread per expert (k <= K):
// u in registers, W1 transposed in shared memory ([K][K], zero-padded), the
// hidden units in blocks of 8.
template <int K>
__device__ void gate_threads(const RingParams &P, unsigned char *sm, const float *zs,
                             const SupTab &S, unsigned char *tab, float *tau_out) {
    const int gt = threadIdx.x - kGate0;
    const int k = P.k, kp = P.kp;
    const float *W1t = reinterpret_cast<const float *>(sm + P.off_W1);
    const float *b1p = reinterpret_cast<const float *>(sm + P.off_b1);
    const float *w2p = reinterpret_cast<const float *>(sm + P.off_w2);
    const float b2 = __ldg(P.b2);
    for (int e = gt; e < P.R; e += kGateT) {
        float u[K];
#pragma unroll
        for (int i = 0; i < K; ++i) u[i] = i < k ? zs[S.idx[S.at(e, i)]] : 0.f;
        float g = 0.f;
#pragma unroll
        for (int jc = 0; jc < K; jc += 8) {
            float h[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) h[jj] = b1p[jc + jj];
#pragma unroll
            for (int i = 0; i < K; ++i) {
                const float4 wa = *reinterpret_cast<const float4 *>(W1t + i * K + jc);
                const float4 wb = *reinterpret_cast<const float4 *>(W1t + i * K + jc + 4);
                h[0] = fmaf(wa.x, u[i], h[0]);
                h[1] = fmaf(wa.y, u[i], h[1]);
                h[2] = fmaf(wa.z, u[i], h[2]);
                h[3] = fmaf(wa.w, u[i], h[3]);
                h[4] = fmaf(wb.x, u[i], h[4]);
                h[5] = fmaf(wb.y, u[i], h[5]);
                h[6] = fmaf(wb.z, u[i], h[6]);
                h[7] = fmaf(wb.w, u[i], h[7]);
            }
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) g = fmaf(w2p[jc + jj], fmaxf(h[jj], 0.f), g);
        }
        const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-(g + b2)));
        const float rt = 1.f / tau;
        const float L0 = S.lg[S.at(e, 0)];  // position 0 holds the largest logit
        float ex[K], s = 0.f;
#pragma unroll
        for (int i = 0; i < K; ++i) {
            ex[i] = i < k ? expf((S.lg[S.at(e, i)] - L0) * rt) : 0.f;
            s += ex[i];
        }
        const float inv = 1.f / s;
        uint4 *te = reinterpret_cast<uint4 *>(tab);
#pragma unroll
        for (int i = 0; i < K; i += 2)  // the odd-k pad gets 0
            if (i < kp)
                *reinterpret_cast<float2 *>(reinterpret_cast<float *>(te + tslot(P.RS, e, i >> 1)) + 2) =
                    make_float2(ex[i] * inv, ex[i + 1] * inv);
        if (tau_out) tau_out[e] = tau;
    }
}

// A warp per expert for 32 < k <= 64, a lane per hidden unit (W1 rows
// padded to ks in shared memory).
__device__ void gate_warps(const RingParams &P, unsigned char *sm, const float *zs,
                           const SupTab &S, unsigned char *tab, float *tau_out) {
    const int gt = threadIdx.x - kGate0;
    const int warp = gt >> 5, lane = threadIdx.x & 31;
    float *uw = reinterpret_cast<float *>(sm + P.off_uw) + warp * P.k;
    const float *W1s = reinterpret_cast<const float *>(sm + P.off_W1);
    const float *b1s = reinterpret_cast<const float *>(sm + P.off_b1);
    const float *w2s = reinterpret_cast<const float *>(sm + P.off_w2);
    const int k = P.k, ks = P.ks, kp = P.kp;
    const float b2 = __ldg(P.b2);
    for (int e = warp; e < P.R; e += kGateT / 32) {
        for (int i = lane; i < k; i += 32) uw[i] = zs[S.idx[S.at(e, i)]];
        __syncwarp();
        float gp = 0.f;
        for (int jj = lane; jj < k; jj += 32) {
            const float *wr = W1s + jj * ks;
            float hj = b1s[jj];
            for (int i = 0; i < k; ++i) hj = fmaf(wr[i], uw[i], hj);
            gp = fmaf(w2s[jj], fmaxf(hj, 0.f), gp);
        }
        const float gv = warp_sum(gp) + b2;
        const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-gv));
        const float L0 = S.lg[S.at(e, 0)];
        const float ex0 = lane < k ? expf((S.lg[S.at(e, lane)] - L0) / tau) : 0.f;
        const float ex1 = lane + 32 < k ? expf((S.lg[S.at(e, lane + 32)] - L0) / tau) : 0.f;
        const float zsum = warp_sum(ex0 + ex1);
        float *tw = reinterpret_cast<float *>(tab);
        if (lane < kp) tw[4 * tslot(P.RS, e, lane >> 1) + 2 + (lane & 1)] = lane < k ? ex0 / zsum : 0.f;
        if (lane + 32 < kp)
            tw[4 * tslot(P.RS, e, (lane + 32) >> 1) + 2 + (lane & 1)] = lane + 32 < k ? ex1 / zsum : 0.f;
        if (lane == 0 && tau_out) tau_out[e] = tau;
        __syncwarp();
    }
}

// z of item r's example into z buffer r mod 2 (Sec. 3.3, GAP): wait until
// every tile of the example is counted, then the example's fixed-point
// accumulator (or, past the fixed-point range, the fp32 tile sums in tile
// order). Lane l owns channels 8 l .. 8 l + 7. The CTA with the example's
// first tile also writes z to the workspace.
__device__ void fetch_role(const RingParams &P, unsigned char *sm, uint32_t par) {
    const int lane = threadIdx.x & 31;
    const int c0 = 8 * lane;
    const bool own = c0 < P.C;
    const uint32_t *count = P.count + (size_t)par * P.N;
    const uint32_t *ovf = P.ovf + (size_t)par * P.N;
    const unsigned long long *zacc = P.zacc + (size_t)par * P.N * P.C;
    const float inv_hw = 1.0f / (float)P.HW;
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t zb = r & 1u;
        const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
        bool ok = true;
        if (lane == 0) {
            ok = r < 2u || mbar_wait(mbar(P, sm, kMbZFree + zb), ((r >> 1) - 1u) & 1u, P.ctrl, it);
            ok = ok && wait_count(count + n, (uint32_t)P.T, P.ctrl, it);
        }
        if (!__all_sync(0xffffffffu, ok)) break;
        __syncwarp();
        float z[8];
        if (own) {
            const ulonglong2 *za = reinterpret_cast<const ulonglong2 *>(zacc + (size_t)n * P.C + c0);
            const ulonglong2 q0 = __ldcg(za), q1 = __ldcg(za + 1), q2 = __ldcg(za + 2),
                             q3 = __ldcg(za + 3);
            const unsigned long long q[8] = {q0.x, q0.y, q1.x, q1.y, q2.x, q2.y, q3.x, q3.y};
#pragma unroll
            for (int m = 0; m < 8; ++m) z[m] = __ll2float_rn((long long)q[m]) * kFixInv * inv_hw;
        }
        if (__ldcg(ovf + n) != 0u && own) {
            // a tile sum was beyond the fixed-point range: the fp32 tile sums
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const float *pc = P.part + (size_t)n * P.T * P.C + c0 + m;
                float s = 0.f;
                for (int tt = 0; tt < P.T; ++tt) s += __ldcg(pc + (size_t)tt * P.C);
                z[m] = s / (float)P.HW;
            }
        }
        if (own) {
            float4 *zs = reinterpret_cast<float4 *>(reinterpret_cast<float *>(sm + P.off_zs) +
                                                    zb * P.C + c0);
            zs[0] = make_float4(z[0], z[1], z[2], z[3]);
            zs[1] = make_float4(z[4], z[5], z[6], z[7]);
            if (t == 0) {
                float4 *zo = reinterpret_cast<float4 *>(P.z + (size_t)n * P.C + c0);
                zo[0] = zs[0];
                zo[1] = zs[1];
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(mbar(P, sm, kMbZReady + zb));
    }
}

// The gate of item r from z buffer r mod 2 into table r mod kNT. The CTA
// with the example's first tile also writes tau to the workspace.
__device__ void gate_role(const RingParams &P, unsigned char *sm) {
    const int gt = threadIdx.x - kGate0;
    SupTab S;
    if (P.gate_tabs) {
        S.idx = reinterpret_cast<const int32_t *>(sm + P.off_pidx);
        S.lg = reinterpret_cast<const float *>(sm + P.off_plog);
        S.se = 1;
        S.si = P.R;
    } else {
        S.idx = P.pidx;
        S.lg = P.plog;
        S.se = P.k;
        S.si = 1;
    }
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t tb = r % kNT, zb = r & 1u;
        const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
        bool ok = true;
        if (gt == 0) {
            // table tb is free once the mix role is done with item r - kNT
            ok = r < kNT ||
                 mbar_wait(mbar(P, sm, kMbTFree + tb), ((r / kNT) - 1u) & 1u, P.ctrl, it);
            ok = ok && mbar_wait(mbar(P, sm, kMbZReady + zb), (r >> 1) & 1u, P.ctrl, it);
        }
        if (!bar_and(kBarGate, kGateT, ok)) break;
        const float *zs = reinterpret_cast<const float *>(sm + P.off_zs) + zb * P.C;
        unsigned char *tab = sm + P.off_tab[tb];
        float *tau_out = t == 0 ? P.tau + (size_t)n * P.R : nullptr;
        if (P.Kg == 16) gate_threads<16>(P, sm, zs, S, tab, tau_out);
        else if (P.Kg == 32) gate_threads<32>(P, sm, zs, S, tab, tau_out);
        else gate_warps(P, sm, zs, S, tab, tau_out);
        bar_sync(kBarGate, kGateT);  // the table is complete; the z buffer is free again
        if (gt == 0) {
            mbar_arrive(mbar(P, sm, kMbTReady + tb));
            mbar_arrive(mbar(P, sm, kMbZFree + zb));
        }
    }
}

// Publishes the channel sums of item r's tile (partial sums of block r mod
// kNB) and counts the tile into its example: lane l owns channels 8 l ..
// 8 l + 7.
__device__ void publish_role(const RingParams &P, unsigned char *sm, uint32_t par,
                             uint32_t drop) {
    const int lane = threadIdx.x & 31;
    const int c0 = 8 * lane;
    const bool own = c0 < P.C;
    uint32_t *count = P.count + (size_t)par * P.N;
    uint32_t *ovf = P.ovf + (size_t)par * P.N;
    unsigned long long *zacc = P.zacc + (size_t)par * P.N * P.C;
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t b = r % kNB;
        const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
        bool ok = true;
        if (lane == 0) ok = mbar_wait(mbar(P, sm, kMbPooled + b), (r / kNB) & 1u, P.ctrl, it);
        if (!__all_sync(0xffffffffu, ok)) break;
        __syncwarp();  // lane 0's wait orders the partial sums before every lane's reads
        if (own) {
            const float *red = reinterpret_cast<const float *>(sm + P.off_red) + b * kRedF;
            float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            for (int q = 0; q < P.nrow; ++q) {
                const float4 a = *reinterpret_cast<const float4 *>(red + q * P.C + c0);
                const float4 c = *reinterpret_cast<const float4 *>(red + q * P.C + c0 + 4);
                v[0] += a.x; v[1] += a.y; v[2] += a.z; v[3] += a.w;
                v[4] += c.x; v[5] += c.y; v[6] += c.z; v[7] += c.w;
            }
            float4 *pt = reinterpret_cast<float4 *>(P.part + ((size_t)n * P.T + t) * P.C + c0);
            pt[0] = make_float4(v[0], v[1], v[2], v[3]);
            pt[1] = make_float4(v[4], v[5], v[6], v[7]);
            bool big = false;
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                if (fabsf(v[m]) <= P.fix_max)
                    red_add_u64(zacc + (size_t)n * P.C + c0 + m,
                                (unsigned long long)__float2ll_rn(v[m] * kFixScale));
                else
                    big = true;  // also NaN
            }
            if (big) atomicOr(ovf + n, 1u);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(mbar(P, sm, kMbRFree + b));  // block b is read
        __threadfence();
        __syncwarp();
        if (lane == 0 && it + 1u != drop)  // fault injection: this tile is never counted
            atomicAdd(count + n, 1u);
    }
}

// ================================================================ load role
// Staging unit (q, j, cc) of a tile: positions pa = q + 16 j and pa + 8,
// channels 8 cc .. 8 cc + 7 (two 16-byte loads), stored as eight words of
// pixel pairs into rows 8 cc .. 8 cc + 7, word j of chunk q ^ (cc & 7). A
// mixing lane that reads chunk q of a row gets positions q + 8 m, m = 0..7.
// Lane l of load warp w: cc = 8 (w mod CG) + (l mod 8), j = l / 8, units
// q = (w + 16 i) / CG for i = 0, 1 while w + 16 i < 8 CG; a warp's loads
// read 128 contiguous bytes per position and its stores hit 32 banks.
struct LoadUnits {
    int nu;          // units per tile (0..2)
    int cc;          // 8-channel block
    bool own;        // cc < C / 8
    int row;         // row of the partial-sum block
    int pa[2];       // low position of each unit (the high one is pa + 8)
    int src[2];      // element offset of the low position's load in a tile of x
    int dst[2];      // byte offset of the unit's first word in a slot
};

__device__ __forceinline__ LoadUnits load_units(const RingParams &P, int lt) {
    LoadUnits u;
    const int w = lt >> 5, lane = lt & 31;
    const int j = lane >> 3;
    u.cc = 8 * (w & (P.CG - 1)) + (lane & 7);
    u.own = u.cc < (P.C >> 3);
    u.nu = (w < 8 * P.CG) + (w + 16 < 8 * P.CG);
    u.row = w / P.CG;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int q = (w + 16 * i) / P.CG;
        u.pa[i] = q + 16 * j;
        u.src[i] = u.pa[i] * P.C + u.cc * 8;
        u.dst[i] = (u.cc * 8) * kRB + (((q ^ (u.cc & kFM)) << 4) | (j << 2));
    }
    return u;
}

// The loads of item it (none past the last item; positions past the end of
// the example read nothing).
__device__ __forceinline__ void tile_loads(const RingParams &P, const LoadUnits &u, uint32_t it,
                                           uint4 *v) {
    const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
    if (it >= P.items) {
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = zero;
        return;
    }
    const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
    const int p0 = t * kTP, np = min(kTP, P.HW - p0);
    const uint16_t *xt = P.x + ((size_t)n * P.HW + p0) * P.C;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool on = i < u.nu && u.own;
        v[2 * i] = (on && u.pa[i] < np) ? ld_stream(xt + u.src[i]) : zero;
        v[2 * i + 1] = (on && u.pa[i] + 8 < np) ? ld_stream(xt + u.src[i] + 8 * P.C) : zero;
    }
}

// One item of the load role: store the tile held in v into slot r mod D,
// refill v with the loads of the item two ahead, leave the tile's partial
// channel sums (one row per warp row) in block r mod kNB. False when a wait
// gave up.
__device__ __forceinline__ bool load_item(const RingParams &P, unsigned char *sm,
                                          const LoadUnits &u, uint32_t it, uint32_t r, uint4 *v) {
    const int lt = threadIdx.x - kLoad0;
    const int lane = lt & 31;
    const uint32_t s = r % (uint32_t)P.D, b = r % kNB;
    // slot s is free once the mix role is done with item r - D, block b once
    // the publish role is done with item r - kNB
    bool ok = true;
    if (lt == 0) {
        if (r >= (uint32_t)P.D)
            ok = mbar_wait(mbar(P, sm, kMbEmpty + s), ((r / P.D) - 1u) & 1u, P.ctrl, it);
        if (ok && r >= (uint32_t)kNB)
            ok = mbar_wait(mbar(P, sm, kMbRFree + b), ((r / kNB) - 1u) & 1u, P.ctrl, it);
    }
    if (!bar_and(kBarLoad, kLoadT, ok)) return false;
    unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
    float acc[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) acc[m] = 0.f;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        if (i >= u.nu || !u.own) continue;
        unsigned char *d = xs + u.dst[i];
        const uint4 va = v[2 * i], vb = v[2 * i + 1];
        uint32_t w[8];
        w[0] = __byte_perm(va.x, vb.x, 0x5410); w[1] = __byte_perm(va.x, vb.x, 0x7632);
        w[2] = __byte_perm(va.y, vb.y, 0x5410); w[3] = __byte_perm(va.y, vb.y, 0x7632);
        w[4] = __byte_perm(va.z, vb.z, 0x5410); w[5] = __byte_perm(va.z, vb.z, 0x7632);
        w[6] = __byte_perm(va.w, vb.w, 0x5410); w[7] = __byte_perm(va.w, vb.w, 0x7632);
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            *reinterpret_cast<uint32_t *>(d + m * kRB) = w[m];
            acc[m] += bf16lo(w[m]) + bf16hi(w[m]);
        }
    }
    // the item two ahead is in flight while this one is reduced and the
    // next one is stored
    tile_loads(P, u, it + 2u * gridDim.x, v);
    // partial channel sums: lanes with the same cc (j = 0..3) by shuffles;
    // the publish role adds the rows
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], 8);
        acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], 16);
    }
    if (lane < 8 && u.nu > 0 && u.own) {
        float *red = reinterpret_cast<float *>(sm + P.off_red) + b * kRedF;
        float4 *rr = reinterpret_cast<float4 *>(red + u.row * P.C + u.cc * 8);
        rr[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
        rr[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    }
    bar_sync(kBarLoad, kLoadT);
    if (lt == 0) {
        mbar_arrive(mbar(P, sm, kMbFull + s));
        mbar_arrive(mbar(P, sm, kMbPooled + b));
    }
    return true;
}

// Items alternate between the two register sets (unrolled by two, so each
// set stays in registers).
__device__ void load_role(const RingParams &P, unsigned char *sm, const LoadUnits &u, uint4 *va,
                          uint4 *vb) {
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items;) {
        if (!load_item(P, sm, u, it, r, va)) break;
        it += gridDim.x;
        ++r;
        if (it >= P.items) break;
        if (!load_item(P, sm, u, it, r, vb)) break;
        it += gridDim.x;
        ++r;
    }
}

// ================================================================ mix role
// Weighted sums of two experts for the lane's 8 positions, over their table
// entries (RS apart); the experts are interleaved for instruction-level
// parallelism. An entry is {row offset, row offset, weight, weight} of two
// support positions.
__device__ __forceinline__ void mix_pairs(const unsigned char *xs, const uint4 *ta, const uint4 *tb,
                                          int RS, int npairs, uint32_t lx, float2 &a0, float2 &a1,
                                          float2 &a2, float2 &a3, float2 &b0, float2 &b1,
                                          float2 &b2, float2 &b3) {
#pragma unroll 2
    for (int i2 = 0; i2 < npairs; ++i2) {
        const uint4 ea = ta[i2 * RS];
        const uint4 eb = tb[i2 * RS];
        const uint4 va0 = lds128(xs + (ea.x ^ lx));
        const uint4 va1 = lds128(xs + (ea.y ^ lx));
        const uint4 vb0 = lds128(xs + (eb.x ^ lx));
        const uint4 vb1 = lds128(xs + (eb.y ^ lx));
        const float2 wa0 = make_float2(__uint_as_float(ea.z), __uint_as_float(ea.z));
        const float2 wa1 = make_float2(__uint_as_float(ea.w), __uint_as_float(ea.w));
        const float2 wb0 = make_float2(__uint_as_float(eb.z), __uint_as_float(eb.z));
        const float2 wb1 = make_float2(__uint_as_float(eb.w), __uint_as_float(eb.w));
        a0 = __ffma2_rn(wa0, unpack2(va0.x), a0);
        a1 = __ffma2_rn(wa0, unpack2(va0.y), a1);
        a2 = __ffma2_rn(wa0, unpack2(va0.z), a2);
        a3 = __ffma2_rn(wa0, unpack2(va0.w), a3);
        b0 = __ffma2_rn(wb0, unpack2(vb0.x), b0);
        b1 = __ffma2_rn(wb0, unpack2(vb0.y), b1);
        b2 = __ffma2_rn(wb0, unpack2(vb0.z), b2);
        b3 = __ffma2_rn(wb0, unpack2(vb0.w), b3);
        a0 = __ffma2_rn(wa1, unpack2(va1.x), a0);
        a1 = __ffma2_rn(wa1, unpack2(va1.y), a1);
        a2 = __ffma2_rn(wa1, unpack2(va1.z), a2);
        a3 = __ffma2_rn(wa1, unpack2(va1.w), a3);
        b0 = __ffma2_rn(wb1, unpack2(vb1.x), b0);
        b1 = __ffma2_rn(wb1, unpack2(vb1.y), b1);
        b2 = __ffma2_rn(wb1, unpack2(vb1.z), b2);
        b3 = __ffma2_rn(wb1, unpack2(vb1.w), b3);
    }
}

__device__ void mix_role(const RingParams &P, unsigned char *sm) {
    const int st = threadIdx.x;
    const int warp = st >> 5, lane = st & 31;
    const int h = lane / kGS, lig = lane % kGS;
    const uint32_t lx = (uint32_t)lig << 4;
    const int g = warp * kGPW + h;
    const int R = P.R, E = R + 1, kp = P.kp, NP = (R + 1) >> 1, Es = P.Es;
    const int32_t *s_resid = reinterpret_cast<const int32_t *>(sm + P.off_U);
    float *rp = reinterpret_cast<float *>(sm + P.off_rp);
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t s = r % (uint32_t)P.D, tb = r % kNT, yb = r % kYB;
        // one thread waits for the slot and the table, the others at the
        // barrier; thread 0 has also seen the bulk copy of item r - kYB
        // finish reading ys
        bool ok = true;
        if (st == 0) {
            ok = mbar_wait(mbar(P, sm, kMbFull + s), (r / P.D) & 1u, P.ctrl, it) &&
                 mbar_wait(mbar(P, sm, kMbTReady + tb), (r / kNT) & 1u, P.ctrl, it);
        }
        if (!bar_and(kBarMix, kMixT, ok)) break;
        const unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys[yb]);
        const uint4 *tab = reinterpret_cast<const uint4 *>(sm + P.off_tab[tb]);
        // expert pairs: warp w's groups take pairs w + 8h of each block of 32
        for (int blk = 0; blk < NP; blk += kMixWarps * kGPW) {
            const int pr = blk + warp + kMixWarps * h;
            if (pr >= NP) continue;
            const int ea = 2 * pr, eb = ea + 1;
            float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
            float2 b0 = a0, b1 = a0, b2 = a0, b3 = a0;
            // an odd last expert pairs with itself; its twin's result is dropped
            const int ebb = eb < R ? eb : ea;
            mix_pairs(xs, tab + tslot(P.RS, ea, 0), tab + tslot(P.RS, ebb, 0), P.RS, kp >> 1, lx,
                      a0, a1, a2, a3, b0, b1, b2, b3);
            // lane lig's positions are lig + 8 m
            if (P.bulk_y) {
                // rows of odd length: 16-bit stores
                uint16_t *yh = ys + lig * Es + ea;
                const int stp = kGS * Es;
                const float av[8] = {a0.x, a0.y, a1.x, a1.y, a2.x, a2.y, a3.x, a3.y};
                const float bv[8] = {b0.x, b0.y, b1.x, b1.y, b2.x, b2.y, b3.x, b3.y};
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    yh[q * stp] = f32_to_bf16(av[q]);
                    if (eb < R) yh[q * stp + 1] = f32_to_bf16(bv[q]);
                }
            } else {
                uint32_t *yw = reinterpret_cast<uint32_t *>(ys + lig * Es + ea);
                const int stp = (kGS * Es) >> 1;
                yw[0 * stp] = pack_bf16x2(a0.x, b0.x);
                yw[1 * stp] = pack_bf16x2(a0.y, b0.y);
                yw[2 * stp] = pack_bf16x2(a1.x, b1.x);
                yw[3 * stp] = pack_bf16x2(a1.y, b1.y);
                yw[4 * stp] = pack_bf16x2(a2.x, b2.x);
                yw[5 * stp] = pack_bf16x2(a2.y, b2.y);
                yw[6 * stp] = pack_bf16x2(a3.x, b3.x);
                yw[7 * stp] = pack_bf16x2(a3.y, b3.y);
            }
        }
        // residual: group g sums U entries g, g + kGroups, ... for its positions
        if (P.nU > 0) {
            float2 r0 = make_float2(0.f, 0.f), r1 = r0, r2 = r0, r3 = r0;
            for (int uu = g; uu < P.nU; uu += kGroups) {
                const uint32_t c = (uint32_t)s_resid[uu];
                const uint4 vv = lds128(xs + (((c * kRB) | (((c >> 3) & kFM) << 4)) ^ lx));
                r0 = __fadd2_rn(r0, unpack2(vv.x));
                r1 = __fadd2_rn(r1, unpack2(vv.y));
                r2 = __fadd2_rn(r2, unpack2(vv.z));
                r3 = __fadd2_rn(r3, unpack2(vv.w));
            }
            float *rg = rp + g * kRPS + lig;
            rg[0 * kGS] = r0.x; rg[1 * kGS] = r0.y; rg[2 * kGS] = r1.x; rg[3 * kGS] = r1.y;
            rg[4 * kGS] = r2.x; rg[5 * kGS] = r2.y; rg[6 * kGS] = r3.x; rg[7 * kGS] = r3.y;
        }
        bar_sync(kBarMix, kMixT);
        // the slot and the table are no longer read
        if (st == 0) {
            mbar_arrive(mbar(P, sm, kMbEmpty + s));
            mbar_arrive(mbar(P, sm, kMbTFree + tb));
        }
        const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
        const int p0 = t * kTP, np = min(kTP, P.HW - p0);
        {
            // the residual column: four threads per position add a quarter of
            // the groups' partial sums each
            const int px = st >> 2, part = st & 3;
            float sum = 0.f;
            if (P.nU > 0) {
#pragma unroll
                for (int gg = part; gg < kGroups; gg += 4) sum += rp[gg * kRPS + px];
                sum += __shfl_xor_sync(0xffffffffu, sum, 1);
                sum += __shfl_xor_sync(0xffffffffu, sum, 2);
                sum = sum / (float)P.nU;
            }
            if (part == 0 && px < np) ys[px * Es + R] = f32_to_bf16(sum);
        }
        const int cnt = np * E;
        uint16_t *dst = P.y + ((size_t)n * P.HW + p0) * E;
        if (P.bulk_y) {
            // [np][E] is contiguous in shared memory and in y: one bulk copy
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            bar_sync(kBarMix, kMixT);
            if (st == 0) {
                asm volatile(
                    "cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n\t"
                    "cp.async.bulk.commit_group;\n\t"
                    "cp.async.bulk.wait_group.read 1;" ::"l"(dst),
                    "r"(smem_u32(ys)), "r"((uint32_t)cnt * 2u)
                    : "memory");
            }
            continue;
        }
        bar_sync(kBarMix, kMixT);
        // rows of y not 16-byte aligned: 16-byte streaming stores between a
        // 16-bit head and tail
        const int head = min(
            cnt, (int)(((16u - ((uint32_t)reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u) >> 1));
        for (int o = st; o < head; o += kMixT) {
            const int p = fdiv(o, E, P.inv_E);
            __stcs(dst + o, ys[p * Es + (o - p * E)]);
        }
        const int nv = (cnt - head) >> 3;
        for (int vi = st; vi < nv; vi += kMixT) {
            const int o = head + vi * 8;
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
        for (int o = head + nv * 8 + st; o < cnt; o += kMixT) {
            const int p = fdiv(o, E, P.inv_E);
            __stcs(dst + o, ys[p * Es + (o - p * E)]);
        }
    }
    // bulk copies complete before the CTA exits
    if (st == 0 && P.bulk_y) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ================================================================ the kernel
__global__ void __launch_bounds__(kRingT, 1) moce_ring_kernel(const RingParams P) {
    extern __shared__ __align__(128) unsigned char sm[];
    const uint32_t epoch = ld_relaxed(P.ctrl + kCtrlEpoch);
    const uint32_t par = epoch & 1u;
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    const int tid = threadIdx.x;
    const bool loader = tid >= kLoad0;
    // the load role's first two tiles are in flight during the set-up
    LoadUnits lu;
    uint4 va[4], vb[4];
    if (loader) {
        lu = load_units(P, tid - kLoad0);
        tile_loads(P, lu, blockIdx.x, va);
        tile_loads(P, lu, blockIdx.x + gridDim.x, vb);
    }
    // the next forward's accumulators and counters (the other parity) start
    // from zero; nothing in this forward uses them
    {
        const uint32_t np = par ^ 1u;
        const size_t gid = (size_t)blockIdx.x * kRingT + tid, gs = (size_t)gridDim.x * kRingT;
        unsigned long long *za = P.zacc + (size_t)np * P.N * P.C;
        for (size_t i = gid; i < (size_t)P.N * P.C; i += gs) za[i] = 0ull;
        for (size_t i = gid; i < (size_t)P.N; i += gs) {
            P.count[np * P.N + i] = 0u;
            P.ovf[np * P.N + i] = 0u;
        }
    }
    // set-up: U list, gate parameters and support tables, the mixing tables'
    // row offsets (weights 0), the zero row of every slot, mbarriers
    int32_t *s_resid = reinterpret_cast<int32_t *>(sm + P.off_U);
    for (int i = tid; i < P.nU; i += kRingT) s_resid[i] = __ldg(P.resid + i);
    float *W1s = reinterpret_cast<float *>(sm + P.off_W1);
    float *b1s = reinterpret_cast<float *>(sm + P.off_b1);
    float *w2s = reinterpret_cast<float *>(sm + P.off_w2);
    if (P.Kg) {
        // W1 transposed: W1s[i * Kg + j] = W1[j][i], zero-padded
        for (int q = tid; q < P.Kg * P.Kg; q += kRingT) {
            const int i = q / P.Kg, j = q - i * P.Kg;
            W1s[q] = (j < P.k && i < P.k) ? __ldg(P.W1 + j * P.k + i) : 0.f;
        }
        for (int j = tid; j < P.Kg; j += kRingT) {
            b1s[j] = j < P.k ? __ldg(P.b1 + j) : 0.f;
            w2s[j] = j < P.k ? __ldg(P.w2 + j) : 0.f;
        }
    } else {
        for (int q = tid; q < P.k * P.k; q += kRingT) {
            const int j = q / P.k, i = q - j * P.k;
            W1s[j * P.ks + i] = __ldg(P.W1 + q);
        }
        for (int j = tid; j < P.k; j += kRingT) {
            b1s[j] = __ldg(P.b1 + j);
            w2s[j] = __ldg(P.w2 + j);
        }
    }
    if (P.gate_tabs) {
        // [k][R]: a gate warp's threads (experts) read consecutive words
        for (int q = tid; q < P.R * P.k; q += kRingT) {
            const int e = q / P.k, i = q - e * P.k;
            reinterpret_cast<int32_t *>(sm + P.off_pidx)[i * P.R + e] = __ldg(P.pidx + q);
            reinterpret_cast<float *>(sm + P.off_plog)[i * P.R + e] = __ldg(P.plog + q);
        }
    }
    for (int q = tid; q < P.D * (kRB / 4); q += kRingT) {
        const int d = q / (kRB / 4), w = q - d * (kRB / 4);
        reinterpret_cast<uint32_t *>(sm + P.off_xs + d * P.xs_bytes + (size_t)P.C * kRB)[w] = 0u;
    }
    for (int q = tid; q < P.R * P.kp; q += kRingT) {
        const int el = q / P.kp, i = q - el * P.kp;
        uint32_t off = (uint32_t)P.C * kRB;  // padding entries read the zero row
        if (i < P.k) {
            const uint32_t c = (uint32_t)__ldg(P.pidx + (size_t)el * P.k + i);
            off = (c * kRB) | (((c >> 3) & kFM) << 4);
        }
        for (int b = 0; b < kNT; ++b) {
            uint32_t *w = reinterpret_cast<uint32_t *>(
                reinterpret_cast<uint4 *>(sm + P.off_tab[b]) + tslot(P.RS, el, i >> 1));
            w[i & 1] = off;
            w[2 + (i & 1)] = 0u;
        }
    }
    if (tid == 0) {
        for (int d = 0; d < P.D; ++d) {
            mbar_init(mbar(P, sm, kMbFull + d), 1);
            mbar_init(mbar(P, sm, kMbEmpty + d), 1);
        }
        for (int b = 0; b < kNB; ++b) {
            mbar_init(mbar(P, sm, kMbPooled + b), 1);
            mbar_init(mbar(P, sm, kMbRFree + b), 1);
        }
        for (int b = 0; b < kNT; ++b) {
            mbar_init(mbar(P, sm, kMbTReady + b), 1);
            mbar_init(mbar(P, sm, kMbTFree + b), 1);
            mbar_init(mbar(P, sm, kMbZReady + b), 1);
            mbar_init(mbar(P, sm, kMbZFree + b), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (tid < kMixT) mix_role(P, sm);
    else if (tid < kMixT + kPubT) publish_role(P, sm, par, drop);
    else if (tid < kGate0) fetch_role(P, sm, par);
    else if (!loader) gate_role(P, sm);
    else load_role(P, sm, lu, va, vb);

    __syncthreads();
    if (tid == 0) {
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
struct RingPlan {
    int D = 0, CG = 0, nrow = 0, kp = 0, Es = 0, ks = 0, Kg = 0, WE = 0, RS = 0;
    size_t xs_bytes = 0, off_xs = 0, off_tab[kNT] = {}, off_ys[kYB] = {};
    size_t off_rp = 0, off_red = 0, off_zs = 0, off_uw = 0, off_W1 = 0, off_b1 = 0;
    size_t off_w2 = 0, off_pidx = 0, off_plog = 0, off_U = 0, off_bar = 0, smem = 0;
    bool gate_tabs = false;
};

int sm_count() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms;
}

// Shared memory: D slots of C + 1 staged rows (row C = zeros), kNT mixing
// tables, kYB output tiles, the residual partial sums, the pooling reduction
// block, z, the gate's parameters and scratch, U, the mailbox, mbarriers. D
// is the largest count (at most kMaxD) that fits.
bool ring_plan(int N, int HW, int C, int R, int k, int G, bool bulk_y, RingPlan *plan) {
    (void)N;
    if (C % 8 != 0 || C < 8 || C > 256 || k < 1 || k > kGateMaxK || R < 1 || HW < 1 || G < 1)
        return false;
    const int T = (HW + kTP - 1) / kTP;
    if (T > G) return false;  // an example's tiles on distinct CTAs: at most two rounds apart
    RingPlan p;
    const int cgs = ((C >> 3) + 7) / 8;
    p.CG = cgs <= 1 ? 1 : (cgs <= 2 ? 2 : 4);
    p.nrow = std::min(8, 16 / p.CG);
    p.kp = k + (k & 1);
    p.Es = bulk_y ? R + 1 : (R + 1) + ((R + 1) & 1);
    p.ks = (k % 2 == 0) ? k + 1 : k;
    p.Kg = k <= 16 ? 16 : (k <= 32 ? 32 : 0);
    p.RS = tslot_rows(R);
    p.WE = (p.kp >> 1) * p.RS;
    p.xs_bytes = align_up((size_t)(C + 1) * kRB, 128);
    size_t off = 0;
    auto take = [&](size_t bytes, size_t al) {
        off = align_up(off, al);
        const size_t o = off;
        off += bytes;
        return o;
    };
    for (int b = 0; b < kNT; ++b) p.off_tab[b] = take((size_t)p.WE * 16, 16);
    for (int b = 0; b < kYB; ++b) p.off_ys[b] = take((size_t)kTP * p.Es * 2, 16);
    p.off_rp = take((size_t)kGroups * kRPS * 4, 16);
    p.off_red = take((size_t)kNB * kRedF * 4, 16);
    p.off_zs = take((size_t)2 * C * 4, 16);
    p.off_uw = take((size_t)(kGateT / 32) * k * 4, 16);
    const int kg = p.Kg ? p.Kg : k;
    p.off_W1 = take((size_t)(p.Kg ? p.Kg * p.Kg : k * p.ks) * 4, 16);
    p.off_b1 = take((size_t)kg * 4, 16);
    p.off_w2 = take((size_t)kg * 4, 16);
    p.gate_tabs = (size_t)R * k * 8 <= 8 * 1024;
    if (p.gate_tabs) {
        p.off_pidx = take((size_t)R * k * 4, 16);
        p.off_plog = take((size_t)R * k * 4, 16);
    }
    p.off_U = take((size_t)C * 4, 16);
    p.off_bar = take((size_t)kMbWords * 8, 8);
    const size_t fixed = align_up(off, 128);
    const size_t budget = 227 * 1024;
    if (fixed + 2 * p.xs_bytes > budget) return false;
    p.D = (int)std::min<size_t>(kMaxD, (budget - fixed) / p.xs_bytes);
    p.off_xs = fixed;
    p.smem = fixed + (size_t)p.D * p.xs_bytes;
    *plan = p;
    return true;
}

}  // namespace

bool ring_supported(int N, int HW, int C, int R, int k) {
    RingPlan plan;
    return ring_plan(N, HW, C, R, k, sm_count(), false, &plan);
}

cudaError_t launch_ring(const uint16_t *x, int N, int HW, int C, int R, int k,
                        const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                        const float *W1, const float *b1, const float *w2, const float *b2,
                        float tmin, float tmax, uint16_t *y, const WsLayout &L, unsigned char *ws,
                        cudaStream_t s) {
    const int G = sm_count();
    // every output tile [np][R + 1] starts and ends on a 16-byte boundary of y
    // when HW * (R + 1) is a multiple of 8: it leaves by one bulk copy
    const bool bulk_y =
        ((long long)HW * (R + 1)) % 8 == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0;
    RingPlan plan;
    if (!ring_plan(N, HW, C, R, k, G, bulk_y, &plan)) return cudaErrorNotSupported;
    RingParams P;
    P.x = x;
    P.y = y;
    P.N = N;
    P.HW = HW;
    P.C = C;
    P.R = R;
    P.k = k;
    P.nU = nU;
    P.T = (HW + kTP - 1) / kTP;
    const unsigned long long items = (unsigned long long)N * P.T;
    if (items >= 0xffff0000ull) return cudaErrorInvalidValue;
    P.items = (uint32_t)items;
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
    P.part = reinterpret_cast<float *>(ws + L.partial);
    P.zacc = reinterpret_cast<unsigned long long *>(ws + L.zacc);
    P.count = reinterpret_cast<uint32_t *>(ws + L.sync);
    P.ovf = P.count + 2 * (size_t)N;
    P.gate_tabs = plan.gate_tabs ? 1 : 0;
    P.fix_max = 274877906944.0f / (float)P.T;  // 2^38 / T
    P.z = reinterpret_cast<float *>(ws + L.z);
    P.tau = reinterpret_cast<float *>(ws + L.tau);
    P.D = plan.D;
    P.CG = plan.CG;
    P.nrow = plan.nrow;
    P.kp = plan.kp;
    P.Es = plan.Es;
    P.ks = plan.ks;
    P.Kg = plan.Kg;
    P.RS = plan.RS;
    P.bulk_y = bulk_y ? 1 : 0;
    P.off_xs = (uint32_t)plan.off_xs;
    P.xs_bytes = (uint32_t)plan.xs_bytes;
    for (int b = 0; b < kNT; ++b) P.off_tab[b] = (uint32_t)plan.off_tab[b];
    for (int b = 0; b < kYB; ++b) P.off_ys[b] = (uint32_t)plan.off_ys[b];
    P.off_rp = (uint32_t)plan.off_rp;
    P.off_red = (uint32_t)plan.off_red;
    P.off_zs = (uint32_t)plan.off_zs;
    P.off_pidx = (uint32_t)plan.off_pidx;
    P.off_plog = (uint32_t)plan.off_plog;
    P.off_uw = (uint32_t)plan.off_uw;
    P.off_W1 = (uint32_t)plan.off_W1;
    P.off_b1 = (uint32_t)plan.off_b1;
    P.off_w2 = (uint32_t)plan.off_w2;
    P.off_U = (uint32_t)plan.off_U;
    P.off_bar = (uint32_t)plan.off_bar;
    P.inv_E = 1.0f / (float)(R + 1);

    cudaError_t err = cudaFuncSetAttribute(moce_ring_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)plan.smem);
    if (err != cudaSuccess) return err;
    int per_sm = 0;
    if ((err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, moce_ring_kernel, kRingT,
                                                             plan.smem)) != cudaSuccess)
        return err;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)moce_ring_kernel, dim3(G), dim3(kRingT), args,
                                       plan.smem, s);
}

}  // namespace moce
