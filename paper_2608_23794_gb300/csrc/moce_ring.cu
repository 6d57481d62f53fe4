// Two-pass and single-pass ring forwards of a MoCE layer (Sec. 3.3-3.4) for
// NHWC bf16 layers with C_in <= 256, C_out <= 64 and k <= 16.
//
// Every expert's temperature depends on the whole-image average of its
// support (Sec. 3.3), so no position of an example can be mixed before all
// of the example has been pooled. The examples are cut into tiles of 64
// positions (tile t of example n is item n*T + t).
//
// Pass 1, moce_poolgate_kernel, streams x once: each CTA reduces a run of
// tiles to its channel sums and adds them, as 64-bit fixed-point
// integers, into accumulator words of the example (integer sums do not
// depend on the order of the additions, so z is deterministic; a sum beyond
// the fixed-point range is kept as an epoch-tagged fp32 word instead). The
// CTA that counts an example's last run reads z, evaluates the gate of
// every expert (Eq. (tau)) and the softmax weights (Eq. (weights)) and
// writes them in mixing-table order; it also clears the example's
// accumulators for the next forward.
//
// Mixing table: for expert pair p (experts 2p, 2p + 1) and support positions
// (2 i2, 2 i2 + 1), one float4 {w(2p, 2i2), w(2p, 2i2+1), w(2p+1, 2i2),
// w(2p+1, 2i2+1)} at entry [i2][4 (p mod 8) + p / 8] of an [8][32] block: a
// mixing lane reads its pair's entries 512 bytes apart from one base, and the
// four lane groups of a mixing warp (pairs 8 apart) read different banks.
//
// Pass 2, moce_ring_kernel, reads x again and mixes it: one CTA per SM takes
// items b, b + G, ...; its copy warp (19) brings each tile (64 positions x C
// channels, contiguous in NHWC) into a ring of D shared-memory slots by one
// bulk copy as soon as a slot is free, so several tiles are in flight; the
// load warps (8-15) transpose a landed tile in place to channel-major rows;
// the table warps (16-18) bring the weights of the item two ahead into one of
// six mixing tables by a bulk copy and sum the tile's unselected channels for
// the residual expert (Eq. (res)); the mix warps (0-7) mix two items per
// round, each slot with its table: each group of 8 lanes owns one expert pair
// for the whole launch and reads one 16-byte row chunk (8 positions) per lane
// and support, with the pair's row offsets in a shared table (Eq. (expert)); each tile
// of y, residual column included, leaves by one bulk copy. The roles hand
// slots and tables over through shared-memory mbarriers; every wait is
// bounded and none crosses CTAs. No role holds global loads in registers
// across a barrier: x and the weights arrive by bulk copies, so the barriers
// never wait for HBM.
//
// The single-pass mode (moce_ring_kernel<true>, one cooperative launch) runs
// pass 1's work inside the same CTAs: each CTA pools its own tiles kLead
// rounds before it mixes them (Seq), the load warps reduce a pooled tile and
// the CTA that counts an example's last tile runs its gate (pool_tile,
// gate_if_last), and the table warps wait, bounded, for the example's tag
// before they bring its weights.
#include <algorithm>

#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kTP = kRingTile;        // positions per tile
constexpr int kGS = 8;                // lanes of a mixing group
constexpr int kRB = 16 * kGS;         // bytes per staged channel row (kTP bf16)
constexpr int kFM = 7;                // chunk swizzle mask of the staged rows
constexpr int kMixT = 256;            // pass 2: mix warps 0-7
constexpr int kLoadT = 256;           // pass 2: load warps 8-15
constexpr int kTabT = 96;             // pass 2: table warps 16-18
constexpr int kProdT = 32;            // pass 2: the copy warp 19
constexpr int kLoadW = kLoadT / 32;
constexpr int kLU = 32 / kLoadW;      // staging units per load thread and tile (at C = 256)
constexpr int kRingT = kMixT + kLoadT + kTabT + kProdT;
constexpr int kLoad0 = kMixT;                    // first load thread
constexpr int kTab0 = kMixT + kLoadT;            // first table thread
constexpr int kProd0 = kTab0 + kTabT;            // the copy warp's first thread
constexpr int kResParts = kTabT / 8;             // residual: U entries split kResParts ways
constexpr int kPairWarps = 8;         // mix warp w takes expert pairs w + 8 h
// Mixing tables: the weights of item r + 2 go into table (r + 2) mod kNT as
// the table role starts item r, which must then wait only for items the mix
// role has finished (r - 3 and before: a mixing round takes two items), so
// kNT >= 2 + 3.
constexpr int kNT = 6;
constexpr int kYB = 4;                // output tile buffers (two items per mixing round)
constexpr int kRS = 4;                // residual columns (the table role runs ahead)
constexpr int kMaxD = 6;              // x slots at most
constexpr int kLead = 10;             // single pass: rounds a CTA pools ahead of mixing
constexpr int kGateMaxK = 16;          // support positions a mixing lane keeps in registers
constexpr int kMaxPairs = 32;          // expert pairs: one per mixing group
constexpr int kWBlock = kMaxPairs * 8; // float4 entries of a weight block
constexpr int kBarMix = 1, kBarLoad = 2, kBarTab = 3;
// Registers per thread: 96 for every role (kRingT * 96 <= 65536).
constexpr int kLaunchRegs = 96, kMixRegs = 96, kLoadRegs = 96, kTabRegs = 96;
static_assert(kMixT * kMixRegs + kLoadT * kLoadRegs + (kTabT + kProdT) * kTabRegs <=
                  kRingT * kLaunchRegs,
              "register split exceeds the launch allocation");
static_assert(kMixT % 128 == 0 && kLoadT % 128 == 0 && (kTabT + kProdT) % 128 == 0,
              "whole warpgroups (the copy warp shares the table warps' register count)");
constexpr int kPoolT = 256;           // pass 1 threads per CTA
constexpr int kPoolCTAs = 8;          // pass 1 CTAs per SM
constexpr int kAccG = 4;              // accumulator words per (example, channel)
static_assert(kRingT * kLaunchRegs <= 65536, "launch registers at one CTA per SM");
static_assert(kMixT == kPairWarps * 32, "one mix warp per set of expert pairs");
static_assert(kTP == 8 * kGS, "a group's lanes cover the tile");
static_assert(kPoolT == 4 * kTP, "pass 1: 32 channel blocks x 8 rows of positions");

// Accumulator word of one (example, channel, group): bits 56-63 count the
// runs added so far, bits 48-55 the runs published as fp32 instead, bits
// 0-47 hold the sum of kFixBias + round(s * 2^20) over the fixed-point runs
// (s = the run's channel sum, |s| < 2^19, so every term is in (0, 2^40) and
// any count of runs below 256 fits). The gate reads a word only once its run
// count is complete, so the adders need no fence before they count.
constexpr float kFixScale = 1048576.0f;  // 2^20
constexpr float kFixInv = 1.0f / 1048576.0f;
constexpr float kFixMax = 524288.0f;     // 2^19
constexpr unsigned long long kFixBias = 1ull << 39;
constexpr unsigned long long kWideOne = 1ull << 48;
constexpr unsigned long long kRunOne = 1ull << 56;

// mbarriers of pass 2 (8 bytes each): raw[s] (the bulk copy of a tile into
// slot s has landed: copy warp's arrival + transaction bytes), full[s]
// (load -> mix, table), empty[s] (mix and table -> copy warp: two
// arrivals), tready[b] (table -> mix), tfree[b] (mix -> table), rdone[c]
// (table -> mix: residual column c), rfree[c] (mix -> table).
constexpr int kMbFull = 0, kMbEmpty = kMaxD, kMbTReady = 2 * kMaxD, kMbTFree = 2 * kMaxD + kNT,
              kMbRDone = 2 * kMaxD + 2 * kNT, kMbRFree = 2 * kMaxD + 2 * kNT + kRS,
              kMbRaw = 2 * kMaxD + 2 * kNT + 2 * kRS, kMbWords = 3 * kMaxD + 2 * kNT + 2 * kRS;

// float4 entry of expert pair p, support positions (2 i2, 2 i2 + 1), in a
// weight block.
__device__ __forceinline__ int wslot(int p, int i2) { return i2 * 32 + 4 * (p & 7) + (p >> 3); }

struct PoolParams {
    const uint16_t *x;
    int N, HW, C, R, k, T;
    int RL, RPE;                  // tiles per run, runs per example
    uint32_t runs;                // N * RPE
    const int32_t *pidx;
    const float *plog;
    const float *W1, *b1, *w2, *b2;
    float tmin, tmax;
    uint32_t *ctrl;
    unsigned long long *part;     // [N][RPE][C] tagged fp32 run sums beyond the fixed-point range
    unsigned long long *zacc;     // [N][kAccG][C] accumulator words
    uint32_t *count;              // [N] runs of example n counted in this forward
    uint32_t *made;               // [N] tag of the forward whose pass 1 wrote example n's weights
    float4 *wts;                  // [N][kWBlock] softmax weights in mixing-table order
    float *z, *tau;
    int kp, Kg;
};

struct RingParams {
    const uint16_t *x;
    uint16_t *y;
    int N, HW, C, R, k, nU, T;
    uint32_t items;               // N * T tiles
    int Gn, Gt;                   // the grid size G = Gn * T + Gt (items a CTA steps over)
    const int32_t *pidx;
    const int32_t *resid;
    uint32_t *ctrl;
    const float4 *wts;            // [N][kWBlock] from pass 1
    const uint32_t *made;         // [N] tags written with them
    int D;                        // x slots
    int CG;                       // load role: 64-channel groups (1, 2, 4)
    int kp, Es;
    int bulk_y;                   // output tiles leave by one bulk copy
    uint32_t off_xs, xs_bytes;
    uint32_t off_tab[kNT], off_ys[kYB];
    uint32_t off_res, off_rred, off_U, off_offs, off_bar;
    float inv_nU;                 // 1 / |U| (0 when U is empty)
    float inv_E;
    int lead;                     // single pass: rounds a CTA pools ahead of mixing
    uint32_t off_pool;            // single pass: the load role's pooling scratch
    PoolParams pool;              // single pass: pooling and gate parameters
};

__device__ __forceinline__ void red_add_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Bounded wait for an mbarrier phase; the waiting thread sleeps between
// polls, so its warp leaves the issue slots to the warps that work.
__device__ bool ring_wait(uint32_t a, uint32_t parity, uint32_t *ctrl, uint32_t item) {
    for (uint32_t it = 0; it < kSpinLimit; ++it) {
        if (mbar_try(a, parity)) return true;
        if ((it & 15u) == 15u && ld_relaxed(ctrl + kCtrlError) != 0u) return false;
        __nanosleep(64);
    }
    report_timeout(ctrl, item);
    return false;
}

__device__ __forceinline__ uint32_t mbar(const RingParams &P, const unsigned char *sm, int word) {
    return smem_u32(sm + P.off_bar) + 8u * (uint32_t)word;
}

// Support table element (e, i): [R][k] in global memory.
struct SupTab {
    const int32_t *idx;
    const float *lg;
    int se, si;
    __device__ __forceinline__ int at(int e, int i) const { return e * se + i * si; }
};

// ================================================================ pass 1
// Gate of every expert of one example (Eq. (tau)): u = z at the expert's
// support in deployment order, h = ReLU(W1 u + b1), g = w2 . h + b2,
// tau = tau_min + (tau_max - tau_min) sigma(g); weights a = softmax(L / tau)
// (Eq. (weights)), written into the mixing table. Run by the mix role:
// K / 4 threads per expert (k <= K), thread q of an expert owns hidden units
// and support positions 4 q .. 4 q + 3. W1 is transposed in shared memory
// ([K][K], zero-padded, b2 after w2); the softmax uses powers of two,
// exp((L_i - L_0) / tau) = 2^((L_i - L_0) log2(e) / tau).
// Not inlined: its registers do not add to those of the mixing loop.
template <int K>
__device__ __noinline__ void gate_experts(const PoolParams &P, const float *W1t, const float *b1p,
                                          const float *w2p, const float *zs, const SupTab &S,
                                          float4 *wts, float *tau_out, int st) {
    constexpr int TPE = K / 4;             // threads per expert
    constexpr int EPP = kPoolT / TPE;      // experts per pass
    const int q = st % TPE, el = st / TPE;
    const int k = P.k, kp = P.kp;
    const float b2 = w2p[K];
    const float4 bq = *reinterpret_cast<const float4 *>(b1p + 4 * q);
    const float4 wq = *reinterpret_cast<const float4 *>(w2p + 4 * q);
    for (int e0 = 0; e0 < P.R; e0 += EPP) {
        const int e = e0 + el;
        const bool act = e < P.R;
        float2 h0 = make_float2(bq.x, bq.y), h1 = make_float2(bq.z, bq.w);
        // the inputs in blocks of 16
#pragma unroll
        for (int i0 = 0; i0 < K; i0 += 16) {
            float u[16];
#pragma unroll
            for (int i = 0; i < 16; ++i)
                u[i] = (act && i0 + i < k) ? zs[S.idx[S.at(e, i0 + i)]] : 0.f;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float4 w = *reinterpret_cast<const float4 *>(W1t + (i0 + i) * K + 4 * q);
                const float2 uu = make_float2(u[i], u[i]);
                h0 = __ffma2_rn(make_float2(w.x, w.y), uu, h0);
                h1 = __ffma2_rn(make_float2(w.z, w.w), uu, h1);
            }
        }
        float g = wq.x * fmaxf(h0.x, 0.f);
        g = fmaf(wq.y, fmaxf(h0.y, 0.f), g);
        g = fmaf(wq.z, fmaxf(h1.x, 0.f), g);
        g = fmaf(wq.w, fmaxf(h1.y, 0.f), g);
#pragma unroll
        for (int o = 1; o < TPE; o <<= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
        const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-(g + b2)));
        const float rt = 1.4426950408889634f / tau;  // log2(e) / tau
        float ex[4], s = 0.f;
        if (act) {
            const float L0 = S.lg[S.at(e, 0)];  // position 0 holds the largest logit
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const int i = 4 * q + m;
                ex[m] = i < k ? exp2f((S.lg[S.at(e, i)] - L0) * rt) : 0.f;
                s += ex[m];
            }
        } else {
#pragma unroll
            for (int m = 0; m < 4; ++m) ex[m] = 0.f;
        }
#pragma unroll
        for (int o = 1; o < TPE; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (act) {
            const float inv = 1.f / s;
            // positions 4q .. 4q+3 are entries 2q and 2q+1 (the odd-k pad gets 0)
            float *wf = reinterpret_cast<float *>(wts);
            const int pr = e >> 1, half = 2 * (e & 1);
            if (4 * q < kp)
                *reinterpret_cast<float2 *>(wf + 4 * wslot(pr, 2 * q) + half) =
                    make_float2(ex[0] * inv, ex[1] * inv);
            if (4 * q + 2 < kp)
                *reinterpret_cast<float2 *>(wf + 4 * wslot(pr, 2 * q + 1) + half) =
                    make_float2(ex[2] * inv, ex[3] * inv);
            if (tau_out && q == 0) tau_out[e] = tau;
        }
    }
}


// Shared memory of pass 1: partial sums [8][C], z [C], W1 transposed [Kg][Kg],
// b1 [Kg], w2 [Kg] + b2, the last-CTA flag.
struct PoolSmem {
    float red[8 * 256];
    float zs[256];
    float W1t[32 * 32];
    float b1[32];
    float w2[33];
    uint32_t last;
    uint32_t cmd;  // single pass: the load role's next step while it waits for a slot
};

// The example's gate, by the kPoolT threads (tid = 0 .. kPoolT - 1, meeting at
// bar()) of the CTA that counted its last run: z from the accumulator words
// (and the tagged fp32 run sums, in run order), then every expert's
// temperature and weights; the accumulators and the counter are cleared for
// the next forward, and made[n] = tag is published after everything else.
template <typename Bar>
__device__ void finish_example(const PoolParams &P, PoolSmem &S, int n, uint32_t tag, int tid,
                               Bar bar) {
    const unsigned long long T = (unsigned long long)P.RPE;  // runs of the example
    unsigned long long *za = P.zacc + (size_t)n * kAccG * P.C;
    for (int c = tid; c < P.C; c += kPoolT) {
        long long fx = 0;
        bool wide = false;
#pragma unroll
        for (int g = 0; g < kAccG; ++g) {
            const unsigned long long Tg = (T - (unsigned long long)g + kAccG - 1) / kAccG;
            // every run of the group has landed in the word (bounded)
            unsigned long long w = ld_relaxed64(za + (size_t)g * P.C + c);
            for (uint32_t i = 0; (w >> 56) != Tg && i < kSpinLimit; ++i) {
                if ((i & 15u) == 15u && ld_relaxed(P.ctrl + kCtrlError) != 0u) break;
                __nanosleep(64);
                w = ld_relaxed64(za + (size_t)g * P.C + c);
            }
            if ((w >> 56) != Tg) report_timeout(P.ctrl, (uint32_t)n);
            const unsigned long long wg = (w >> 48) & 0xffull;
            fx += (long long)(w & ((1ull << 48) - 1ull)) - (long long)((Tg - wg) * kFixBias);
            wide = wide || wg != 0ull;
        }
        float s = __ll2float_rn(fx) * kFixInv;
        if (wide) {
            const unsigned long long *pc = P.part + (size_t)n * P.RPE * P.C + c;
            for (int t = 0; t < P.RPE; ++t) {
                const unsigned long long wv = __ldcg(pc + (size_t)t * P.C);
                if ((uint32_t)(wv >> 32) == tag) s += __uint_as_float((uint32_t)wv);
            }
        }
        const float zv = s / (float)P.HW;
        S.zs[c] = zv;
        P.z[(size_t)n * P.C + c] = zv;
#pragma unroll
        for (int g = 0; g < kAccG; ++g) za[(size_t)g * P.C + c] = 0ull;
    }
    // W1 transposed (W1t[i * Kg + j] = W1[j][i]), zero-padded; b2 after w2
    for (int q = tid; q < P.Kg * P.Kg; q += kPoolT) {
        const int i = q / P.Kg, j = q - i * P.Kg;
        S.W1t[q] = (j < P.k && i < P.k) ? __ldg(P.W1 + j * P.k + i) : 0.f;
    }
    for (int j = tid; j < P.Kg; j += kPoolT) {
        S.b1[j] = j < P.k ? __ldg(P.b1 + j) : 0.f;
        S.w2[j] = j < P.k ? __ldg(P.w2 + j) : 0.f;
    }
    if (tid == 0) {
        S.w2[P.Kg] = __ldg(P.b2);
        P.count[n] = 0u;
    }
    bar();
    SupTab sup;
    sup.idx = P.pidx;
    sup.lg = P.plog;
    sup.se = P.k;
    sup.si = 1;
    float4 *wts = P.wts + (size_t)n * kWBlock;
    // entries no expert writes (padding positions, the twin of an odd last
    // expert) stay 0
    for (int q = tid; q < kWBlock; q += kPoolT) wts[q] = make_float4(0.f, 0.f, 0.f, 0.f);
    bar();
    float *tau = P.tau + (size_t)n * P.R;
    if (P.Kg == 16) gate_experts<16>(P, S.W1t, S.b1, S.w2, S.zs, sup, wts, tau, tid);
    else gate_experts<32>(P, S.W1t, S.b1, S.w2, S.zs, sup, wts, tau, tid);
    // the weights, z and tau are visible before the tag: mixing CTAs of the
    // same launch read it with acquire
    __threadfence();
    bar();
    if (tid == 0) st_release(P.made + n, tag);
}

// A CTA pools one run of up to RL consecutive tiles of one example: thread
// (row = tid / 32, cb = tid mod 32) adds positions row, row + 8, ... of
// channels 8 cb .. 8 cb + 7 over the run (eight 16-byte loads in flight per
// tile), the eight rows are added in order through shared memory, and thread
// c publishes channel c of the run. The CTA that counts an example's last
// run finishes the example.
__global__ void __launch_bounds__(kPoolT) moce_poolgate_kernel(const PoolParams P) {
    __shared__ __align__(16) PoolSmem S;
    const int tid = threadIdx.x;
    const int row = tid >> 5, cb = tid & 31;
    const bool own = 8 * cb < P.C;
    const uint32_t tag = ld_relaxed(P.ctrl + kCtrlEpoch) + 1u;
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    // the mixing pass may launch now: it reads pass 1's results only after
    // griddepcontrol.wait, and the epoch only at its end
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    for (uint32_t ru = blockIdx.x; ru < P.runs; ru += gridDim.x) {
        const int n = (int)(ru / (uint32_t)P.RPE), j = (int)(ru - (uint32_t)n * P.RPE);
        const int t0 = j * P.RL, t1 = min(P.T, t0 + P.RL);
        const uint16_t *xe = P.x + (size_t)n * P.HW * P.C + 8 * cb;
        float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int t = t0; t < t1; ++t) {
            const int p0 = t * kTP, np = min(kTP, P.HW - p0);
            uint4 v[8];
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const int p = row + 8 * m;
                v[m] = (own && p < np) ? ld_stream(xe + (size_t)(p0 + p) * P.C)
                                       : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                a[0] += bf16lo(v[m].x); a[1] += bf16hi(v[m].x);
                a[2] += bf16lo(v[m].y); a[3] += bf16hi(v[m].y);
                a[4] += bf16lo(v[m].z); a[5] += bf16hi(v[m].z);
                a[6] += bf16lo(v[m].w); a[7] += bf16hi(v[m].w);
            }
        }
        if (own) {
            float4 *rr = reinterpret_cast<float4 *>(S.red + row * P.C + 8 * cb);
            rr[0] = make_float4(a[0], a[1], a[2], a[3]);
            rr[1] = make_float4(a[4], a[5], a[6], a[7]);
        }
        __syncthreads();
        if (tid < P.C && ru + 1u != drop) {  // fault injection: this run is never counted
            float s = 0.f;
#pragma unroll
            for (int q = 0; q < 8; ++q) s += S.red[q * P.C + tid];
            unsigned long long add;
            if (fabsf(s) < kFixMax) {
                add = kRunOne + kFixBias + (unsigned long long)__float2ll_rn(s * kFixScale);
            } else {  // beyond the fixed-point range (or NaN): a tagged fp32 word
                P.part[((size_t)n * P.RPE + j) * P.C + tid] =
                    ((unsigned long long)tag << 32) | __float_as_uint(s);
                add = kRunOne + kWideOne;
            }
            red_add_u64(P.zacc + ((size_t)n * kAccG + (j % kAccG)) * P.C + tid, add);
            __threadfence();
        }
        __syncthreads();  // every channel of the run is added; red is free again
        if (tid == 0) {
            uint32_t last = 0u;
            if (ru + 1u != drop) {
                const uint32_t old = atomicAdd(P.count + n, 1u);
                if (old == (uint32_t)P.RPE - 1u) {
                    __threadfence();
                    last = 1u;
                }
            }
            S.last = last;
        }
        __syncthreads();
        if (S.last) {
            finish_example(P, S, n, tag, tid, [] { __syncthreads(); });
            __syncthreads();
        }
    }
}

// ================================================================ pass 2
// Staging unit (q, j, cc) of a tile: positions pa = q + 16 j and pa + 8,
// channels 8 cc .. 8 cc + 7 (two 16-byte loads), stored as eight words of
// pixel pairs into rows 8 cc .. 8 cc + 7, word j of chunk q ^ (cc & 7). A
// mixing lane that reads chunk q of a row gets positions q + 8 m, m = 0..7.
// Lane l of load warp w: cc = 8 (w mod CG) + (l mod 8), j = l / 8, units
// q = (w + 8 i) / CG for i = 0 .. kLU - 1 while w + 8 i < 8 CG; a warp's
// reads take 128 contiguous bytes per position and its stores hit 32 banks.
struct LoadUnits {
    int nu;          // units per tile (0..kLU)
    int cc;          // 8-channel block
    bool own;        // cc < C / 8
    int pa[kLU];     // low position of each unit (the high one is pa + 8)
    int src[kLU];    // element offset of the low position in a tile of x
    int dst[kLU];    // byte offset of the unit's first word in a slot
};

__device__ __forceinline__ LoadUnits load_units(const RingParams &P, int lt) {
    LoadUnits u;
    const int w = lt >> 5, lane = lt & 31;
    const int j = lane >> 3;
    u.cc = 8 * (w & (P.CG - 1)) + (lane & 7);
    u.own = u.cc < (P.C >> 3);
    u.nu = 0;
#pragma unroll
    for (int i = 0; i < kLU; ++i) u.nu += (w + kLoadW * i < 8 * P.CG);
#pragma unroll
    for (int i = 0; i < kLU; ++i) {
        const int q = (w + kLoadW * i) / P.CG;
        u.pa[i] = q + 16 * j;
        u.src[i] = u.pa[i] * P.C + u.cc * 8;
        u.dst[i] = (u.cc * 8) * kRB + (((q ^ (u.cc & kFM)) << 4) | (j << 2));
    }
    return u;
}

// A CTA's items are b, b + G, ... (rounds r = 0 .. nb - 1); ItemPos follows
// one of them (item it: example n, tile t) without divisions.
struct ItemPos {
    uint32_t r, it;
    int n, t;
    __device__ __forceinline__ explicit ItemPos(const RingParams &P) : r(0), it(blockIdx.x) {
        n = (int)(blockIdx.x / (uint32_t)P.T);
        t = (int)blockIdx.x - n * P.T;
    }
    __device__ __forceinline__ void next(const RingParams &P) {
        ++r;
        it += gridDim.x;
        n += P.Gn;
        t += P.Gt;
        if (t >= P.T) {
            t -= P.T;
            ++n;
        }
    }
    __device__ __forceinline__ int p0() const { return t * kTP; }
    __device__ __forceinline__ int np(const RingParams &P) const { return min(kTP, P.HW - t * kTP); }
};

// The CTA's slot sequence: every position j takes slot j mod D (phase bit
// (j / D) mod 2 of the slot's raw and empty mbarriers) for one tile; full[s]
// completes only for mixing positions, so the roles that wait on it keep one
// phase bit per slot (FullPhase). A two-pass launch only
// mixes: position r holds item r. A single-pass launch also pools its own
// items L = lead rounds ahead: positions pool(0 .. L - 1), then per round r
// pool(r + L) (while there is one) and mix(r). Every role walks the same
// sequence. F: a single-pass launch.
template <bool F>
struct Seq {
    ItemPos pool, mix;  // next pool item, next mix item
    uint32_t j, s, ph;  // position, slot, phase bit
    uint32_t nb;        // items of this CTA
    bool is_pool;       // the position pools (else it mixes mix)
    __device__ __forceinline__ explicit Seq(const RingParams &P)
        : pool(P), mix(P), j(0), s(0), ph(0) {
        nb = (P.items - blockIdx.x + gridDim.x - 1) / gridDim.x;
        decide(P);
    }
    __device__ __forceinline__ void decide(const RingParams &P) {
        is_pool = F && pool.r < nb && pool.r < mix.r + (uint32_t)P.lead;
    }
    __device__ __forceinline__ bool live() const { return mix.r < nb; }
    __device__ __forceinline__ const ItemPos &item() const { return is_pool ? pool : mix; }
    __device__ __forceinline__ void next(const RingParams &P) {
        if (is_pool) pool.next(P);
        else mix.next(P);
        ++j;
        if (++s == (uint32_t)P.D) {
            s = 0;
            ph ^= 1u;
        }
        decide(P);
    }
    // the next mixing position
    __device__ __forceinline__ void next_mix(const RingParams &P) {
        do next(P);
        while (live() && is_pool);
    }
};

// Example n's tag: with acquire in a single-pass launch (the gate ran in
// another CTA of it), else relaxed (pass 1 has finished).
template <bool F>
__device__ __forceinline__ uint32_t read_tag(const RingParams &P, int n) {
    return F ? ld_acquire(P.made + n) : ld_relaxed(P.made + n);
}

// Waits until example n's gate has run in this forward (made[n] == tag,
// read with acquire; v is a value already read). A two-pass launch starts
// after pass 1 has finished, so there a stale tag is reported at once; a
// single-pass launch waits (bounded) for the CTA that pools the example's
// last tile. False when the wait gave up or another wait did.
template <bool F>
__device__ bool made_wait(const RingParams &P, int n, uint32_t tag, uint32_t v, uint32_t it) {
    for (uint32_t i = 1; v != tag; ++i) {
        if (!F || i >= kSpinLimit) {
            report_timeout(P.ctrl, it);
            return false;
        }
        if ((i & 15u) == 0u && ld_relaxed(P.ctrl + kCtrlError) != 0u) return false;
        __nanosleep(64);
        v = read_tag<F>(P, n);
    }
    return true;
}

// Slot of mixing item m (round m of the CTA, nb items): its position is m
// in a two-pass launch; in a single-pass launch with L = min(lead, nb) pooled
// positions first it is L + 2 m while pooled positions still follow, then
// nb + m.
template <bool F>
__device__ __forceinline__ uint32_t mix_slot(const RingParams &P, uint32_t m, uint32_t nb) {
    uint32_t pos = m;
    if (F) {
        const uint32_t L = min((uint32_t)P.lead, nb);
        pos = m < nb - L ? L + 2u * m : nb + m;
    }
    return pos % (uint32_t)P.D;
}
__device__ __forceinline__ uint32_t cta_items(const RingParams &P) {
    return (P.items - blockIdx.x + gridDim.x - 1) / gridDim.x;
}

// Phase bits of the full mbarriers, one per slot: a role that waits for
// every mixing use of every slot in order flips slot s's bit after each wait.
struct FullPhase {
    uint32_t bits = 0;
    __device__ __forceinline__ uint32_t take(uint32_t s) {
        const uint32_t b = (bits >> s) & 1u;
        bits ^= 1u << s;
        return b;
    }
};

// One bulk copy of the weight block of mix item q's example into table
// q.r mod kNT; tready of that table completes when the 4 KB have landed.
__device__ __forceinline__ void weights_copy(const RingParams &P, unsigned char *sm,
                                             const ItemPos &q) {
    const uint32_t tb = q.r % kNT;
    const uint32_t bar = mbar(P, sm, kMbTReady + tb);
    // the weights were written by generic stores (of this launch, read
    // with acquire, or of pass 1); the mix role's reads of the table's
    // previous contents come first
    asm volatile(
        "fence.proxy.async.global;\n\t"
        "fence.proxy.async.shared::cta;\n\t"
        "mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t"
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%2], [%3], %1, "
        "[%0];" ::"r"(bar),
        "r"((uint32_t)(kWBlock * 16)), "r"(smem_u32(sm + P.off_tab[tb])),
        "l"(P.wts + (size_t)q.n * kWBlock)
        : "memory");
}

// The copy warp walks the slot sequence: per position, once the slot is
// released (empty[s]: the mix and table roles, or the load role for a
// pooled tile), one bulk copy of the tile's np * C contiguous bf16 (NHWC);
// raw[s] completes when the bytes have landed. On a wait that gave up, the
// copies still in flight land before the warp returns.
template <bool F>
__device__ void copy_role(const RingParams &P, unsigned char *sm) {
    set_role_regs<kTabRegs, kLaunchRegs>();
    if ((threadIdx.x & 31) == 0) {
        Seq<F> q(P);
        bool ok = true;
        for (; q.live(); q.next(P)) {
            if (q.j >= (uint32_t)P.D &&
                !ring_wait(mbar(P, sm, kMbEmpty + q.s), q.ph ^ 1u, P.ctrl, q.item().it)) {
                ok = false;
                break;
            }
            const ItemPos &w = q.item();
            const uint32_t bytes = (uint32_t)w.np(P) * (uint32_t)P.C * 2u;
            const uint16_t *src = P.x + ((size_t)w.n * P.HW + w.p0()) * P.C;
            const uint32_t bar = mbar(P, sm, kMbRaw + q.s);
            // the slot's earlier generic-proxy reads and writes come before the copy
            asm volatile(
                "fence.proxy.async.shared::cta;\n\t"
                "mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t"
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%2], [%3], %1, "
                "[%0];" ::"r"(bar),
                "r"(bytes), "r"(smem_u32(sm + P.off_xs + q.s * P.xs_bytes)), "l"(src)
                : "memory");
        }
        if (!ok) {
            const uint32_t j1 = q.j, d = (uint32_t)P.D;
            for (uint32_t j = j1 > d ? j1 - d : 0u; j < j1; ++j) {
                const uint32_t bar = mbar(P, sm, kMbRaw + j % d);
                for (uint32_t i = 0; i < kSpinLimit && !mbar_test(bar, (j / d) & 1u); ++i)
                    __nanosleep(256);
            }
        }
    }
    __syncwarp();
}

// A pooled position (single-pass launches), by the load role: thread
// (row = lt / 32, cb = lt mod 32) adds positions row, row + 8, ... of
// channels 8 cb .. 8 cb + 7 of the raw tile, the eight rows are added in
// order through shared memory, the slot is released, and thread c adds the
// tile's channel sum c to the example's accumulator words (group t mod kAccG)
// as in pass 1 (run count included). After the role's barrier thread 0
// counts the tile; the count it gets back is looked at two positions later
// (gate_if_last), so the role does not wait for it.
__device__ __forceinline__ void pool_tile(const RingParams &P, unsigned char *sm,
                                          const unsigned char *xs, const ItemPos &w, uint32_t s,
                                          uint32_t tag, uint32_t drop, uint32_t &old) {
    const int lt = threadIdx.x - kLoad0;
    const int row = lt >> 5, cb = lt & 31;
    PoolSmem &S = *reinterpret_cast<PoolSmem *>(sm + P.off_pool);
    const int np = w.np(P);
    float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (8 * cb < P.C) {
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const int p = row + 8 * m;
            if (p < np) {
                const uint4 v = lds128(xs + 2 * (p * P.C + 8 * cb));
                a[0] += bf16lo(v.x); a[1] += bf16hi(v.x);
                a[2] += bf16lo(v.y); a[3] += bf16hi(v.y);
                a[4] += bf16lo(v.z); a[5] += bf16hi(v.z);
                a[6] += bf16lo(v.w); a[7] += bf16hi(v.w);
            }
        }
        float4 *rr = reinterpret_cast<float4 *>(S.red + row * P.C + 8 * cb);
        rr[0] = make_float4(a[0], a[1], a[2], a[3]);
        rr[1] = make_float4(a[4], a[5], a[6], a[7]);
    }
    bar_sync(kBarLoad, kLoadT);  // the raw tile is read; the row sums are complete
    if (lt == 0) {
        // the slot is free (two arrivals, as the mix and table roles give it)
        mbar_arrive(mbar(P, sm, kMbEmpty + s));
        mbar_arrive(mbar(P, sm, kMbEmpty + s));
    }
    const PoolParams &Q = P.pool;
    const bool counted = w.it + 1u != drop;  // fault injection: this tile is never counted
    if (lt < P.C && counted) {
        float sum = 0.f;
#pragma unroll
        for (int qq = 0; qq < 8; ++qq) sum += S.red[qq * P.C + lt];
        unsigned long long add;
        if (fabsf(sum) < kFixMax) {
            add = kRunOne + kFixBias + (unsigned long long)__float2ll_rn(sum * kFixScale);
        } else {  // beyond the fixed-point range (or NaN): a tagged fp32 word
            Q.part[((size_t)w.n * P.T + w.t) * P.C + lt] =
                ((unsigned long long)tag << 32) | __float_as_uint(sum);
            __threadfence();  // the word is visible before the run is counted in it
            add = kRunOne + kWideOne;
        }
        red_add_u64(Q.zacc + ((size_t)w.n * kAccG + (w.t % kAccG)) * P.C + lt, add);
    }
    bar_sync(kBarLoad, kLoadT);  // every channel of the tile is added; red is free again
    if (lt == 0 && counted) old = atomicAdd(Q.count + w.n, 1u);
}

// The count of a pooled tile (thread 0's old), looked at one position later:
// the CTA that counted the example's last tile runs its gate with the load
// role's threads.
__device__ __forceinline__ void gate_if_last(const RingParams &P, unsigned char *sm, int n,
                                             uint32_t old, uint32_t tag) {
    const int lt = threadIdx.x - kLoad0;
    PoolSmem &S = *reinterpret_cast<PoolSmem *>(sm + P.off_pool);
    if (lt == 0) {
        const uint32_t last = old == (uint32_t)P.T - 1u ? 1u : 0u;
        S.last = last;
    }
    bar_sync(kBarLoad, kLoadT);
    if (S.last) {
        finish_example(P.pool, S, n, tag, lt, [] { bar_sync(kBarLoad, kLoadT); });
        bar_sync(kBarLoad, kLoadT);
    }
}

// The load role walks the slot sequence: once raw[s] completes, a pooled
// position is reduced (pool_tile); a mixing position is read unit by unit
// (positions past np read as 0), the role meets at a barrier, and the units
// are written back in place as channel-major rows of pixel pairs (the raw
// tile, np * C * 2 bytes, lies within rows 0 .. C - 1, so row C stays zero);
// full[s] then tells the mix and table roles.
template <bool F>
__device__ void load_role(const RingParams &P, unsigned char *sm, const LoadUnits &u,
                          uint32_t tag) {
    set_role_regs<kLoadRegs, kLaunchRegs>();
    const int lt = threadIdx.x - kLoad0;
    const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    // the last two pooled tiles whose counts have not been looked at:
    // example (-1: none) and, in thread 0, the count it got back
    int pend0 = -1, pend1 = -1;
    uint32_t old0 = 0xffffffffu, old1 = 0xffffffffu;
    Seq<F> q(P);
    for (; q.live(); q.next(P)) {
        const uint32_t s = q.s;
        if constexpr (F) {
            // pending counts are looked at before and while the role waits
            // for the slot: an example's gate must not wait for this CTA's
            // slots (mixing positions of other CTAs may need the example)
            if (pend0 >= 0) gate_if_last(P, sm, pend0, old0, tag);
            pend0 = pend1;
            old0 = old1;
            pend1 = -1;
            PoolSmem &S = *reinterpret_cast<PoolSmem *>(sm + P.off_pool);
            for (uint32_t polls = 1;; ++polls) {
                if (lt == 0) {
                    uint32_t cmd = 0;  // 0: wait on, 1: landed, 2: gate pend0 now, 3: give up
                    if (mbar_try(mbar(P, sm, kMbRaw + s), q.ph)) {
                        cmd = 1;
                    } else if (polls >= kSpinLimit) {
                        report_timeout(P.ctrl, q.item().it);
                        cmd = 3;
                    } else if ((polls & 15u) == 0u && ld_relaxed(P.ctrl + kCtrlError) != 0u) {
                        cmd = 3;
                    } else if (pend0 >= 0 && polls >= 2) {
                        cmd = 2;
                    }
                    S.cmd = cmd;
                }
                bar_sync(kBarLoad, kLoadT);
                const uint32_t cmd = S.cmd;
                bar_sync(kBarLoad, kLoadT);  // the command word is free again
                if (cmd == 1) break;
                if (cmd == 3) return;
                if (cmd == 2) {
                    gate_if_last(P, sm, pend0, old0, tag);
                    pend0 = -1;
                }
            }
        } else {
            bool ok = true;
            if (lt == 0) ok = ring_wait(mbar(P, sm, kMbRaw + s), q.ph, P.ctrl, q.item().it);
            if (!bar_and(kBarLoad, kLoadT, ok)) return;
        }
        unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
        if constexpr (F) {
            if (q.is_pool) {
                old1 = 0xffffffffu;
                pool_tile(P, sm, xs, q.pool, s, tag, drop, old1);
                pend1 = q.pool.n;
                continue;
            }
        }
        const int np = q.mix.np(P);
        uint4 v[2 * kLU];
#pragma unroll
        for (int i = 0; i < kLU; ++i) {
            const bool on = i < u.nu && u.own;
            v[2 * i] = (on && u.pa[i] < np) ? lds128(xs + 2 * u.src[i]) : zero;
            v[2 * i + 1] = (on && u.pa[i] + 8 < np) ? lds128(xs + 2 * (u.src[i] + 8 * P.C)) : zero;
        }
        bar_sync(kBarLoad, kLoadT);  // the raw tile is read
#pragma unroll
        for (int i = 0; i < kLU; ++i) {
            if (i >= u.nu || !u.own) continue;
            unsigned char *d = xs + u.dst[i];
            const uint4 va = v[2 * i], vb = v[2 * i + 1];
            *reinterpret_cast<uint32_t *>(d + 0 * kRB) = __byte_perm(va.x, vb.x, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 1 * kRB) = __byte_perm(va.x, vb.x, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 2 * kRB) = __byte_perm(va.y, vb.y, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 3 * kRB) = __byte_perm(va.y, vb.y, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 4 * kRB) = __byte_perm(va.z, vb.z, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 5 * kRB) = __byte_perm(va.z, vb.z, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 6 * kRB) = __byte_perm(va.w, vb.w, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 7 * kRB) = __byte_perm(va.w, vb.w, 0x7632);
        }
        bar_sync(kBarLoad, kLoadT);
        if (lt == 0) mbar_arrive(mbar(P, sm, kMbFull + s));
    }
    if constexpr (F) {
        if (pend0 >= 0) gate_if_last(P, sm, pend0, old0, tag);
        if (pend1 >= 0) gate_if_last(P, sm, pend1, old1, tag);
    }
}

// The table role walks the mixing positions. Its thread 0 brings the weights
// of the item two ahead: once table (r + 2) mod kNT is released (the mix role
// finished item r + 2 - kNT) and the example's gate has run in this forward
// (made_wait), one bulk copy into the table. Then, once the tile is staged,
// the residual expert (Eq. (res)): thread (q = chunk, part) adds U entries
// part, part + kResParts, ... for the chunk's 8 positions, the parts are added
// in order, and res[r mod kRS][p] = sum / |U| (0 if U is empty).
template <bool F>
__device__ void table_role(const RingParams &P, unsigned char *sm, uint32_t tag) {
    set_role_regs<kTabRegs, kLaunchRegs>();
    const int tt = threadIdx.x - kTab0;
    const int q = tt & 7, part = tt >> 3;
    const uint32_t lx = (uint32_t)q << 4;
    const int32_t *s_resid = reinterpret_cast<const int32_t *>(sm + P.off_U);
    float *rred = reinterpret_cast<float *>(sm + P.off_rred);
    const uint32_t nb = cta_items(P);
    FullPhase fph;
    // thread 0: the next item whose weights to bring, and the copies made
    ItemPos wq(P);
    uint32_t wcopies = 0;
    bool wok = true;
    if (tt == 0) {
        // a two-pass launch may start before pass 1 has finished; the
        // weights and tags are read after it has
        if (!F) asm volatile("griddepcontrol.wait;" ::: "memory");
        for (int i = 0; i < 2 && wok && wq.r < nb; ++i) {
            wok = made_wait<F>(P, wq.n, tag, read_tag<F>(P, wq.n), wq.it);
            if (wok) weights_copy(P, sm, wq), ++wcopies, wq.next(P);
        }
    }
    for (ItemPos mi(P); mi.r < nb; mi.next(P)) {
        const uint32_t r = mi.r, it = mi.it, s = mix_slot<F>(P, r, nb);
        const uint32_t rc = r % kRS;
        const uint32_t fp = fph.take(s);
        bool ok = wok;
        if (tt == 0 && ok && wq.r < nb) {
            const uint32_t tb = wq.r % kNT;
            if (wq.r >= (uint32_t)kNT)
                ok = ring_wait(mbar(P, sm, kMbTFree + tb), ((wq.r / kNT) - 1u) & 1u, P.ctrl, it);
            if (ok) ok = made_wait<F>(P, wq.n, tag, read_tag<F>(P, wq.n), wq.it);
            if (ok) weights_copy(P, sm, wq), ++wcopies, wq.next(P);
            wok = ok;
        }
        if (tt == 0) {
            if (ok) ok = ring_wait(mbar(P, sm, kMbFull + s), fp, P.ctrl, it);
            if (ok && r >= (uint32_t)kRS)
                ok = ring_wait(mbar(P, sm, kMbRFree + rc), ((r / kRS) - 1u) & 1u, P.ctrl, it);
        }
        if (!bar_and(kBarTab, kTabT, ok)) break;
        const unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
        float2 r0 = make_float2(0.f, 0.f), r1 = r0, r2 = r0, r3 = r0;
        for (int u = part; u < P.nU; u += kResParts) {
            const uint32_t c = (uint32_t)s_resid[u];
            const uint4 vv = lds128(xs + (((c * kRB) | (((c >> 3) & kFM) << 4)) ^ lx));
            r0 = __fadd2_rn(r0, unpack2(vv.x));
            r1 = __fadd2_rn(r1, unpack2(vv.y));
            r2 = __fadd2_rn(r2, unpack2(vv.z));
            r3 = __fadd2_rn(r3, unpack2(vv.w));
        }
        // chunk q's positions are q + 8 m
        float *rg = rred + part * kTP + q;
        rg[0 * 8] = r0.x; rg[1 * 8] = r0.y; rg[2 * 8] = r1.x; rg[3 * 8] = r1.y;
        rg[4 * 8] = r2.x; rg[5 * 8] = r2.y; rg[6 * 8] = r3.x; rg[7 * 8] = r3.y;
        bar_sync(kBarTab, kTabT);
        if (tt == 0) mbar_arrive(mbar(P, sm, kMbEmpty + s));  // the slot is read
        if (tt < kTP) {
            float sum = 0.f;
#pragma unroll
            for (int pp = 0; pp < kResParts; ++pp) sum += rred[pp * kTP + tt];
            reinterpret_cast<float *>(sm + P.off_res)[rc * kTP + tt] = sum * P.inv_nU;
        }
        bar_sync(kBarTab, kTabT);  // rred is free again; the residual column is complete
        if (tt == 0) mbar_arrive(mbar(P, sm, kMbRDone + rc));
    }
    // after a wait gave up, weight copies still in flight land before the
    // CTA exits (after a normal end the mix role has waited for all of them)
    if (tt == 0) {
        for (uint32_t m = wcopies > (uint32_t)kNT ? wcopies - (uint32_t)kNT : 0u; m < wcopies; ++m) {
            const uint32_t bar = mbar(P, sm, kMbTReady + m % kNT);
            for (uint32_t i = 0; i < kSpinLimit && !mbar_test(bar, (m / kNT) & 1u); ++i)
                __nanosleep(256);
        }
    }
}

// ================================================================ mix role
// Row offset (bytes in a slot) of channel c for the lane whose chunk mask is
// lx: row c, chunk ((c >> 3) & 7) ^ lane; channel C is the zero row.
__device__ __forceinline__ uint32_t row_off(uint32_t c, uint32_t lx) {
    return ((c * kRB) | (((c >> 3) & kFM) << 4)) ^ lx;
}

// Shared-memory loads at 32-bit shared-window addresses.
__device__ __forceinline__ uint2 lds64(uint32_t a) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
    return v;
}
__device__ __forceinline__ float4 lds128f(uint32_t a) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(a));
    return v;
}

// bf16 pair -> two fp32: the low half by an integer multiply (FMA pipe),
// the high half by a mask (ALU pipe), so the two pipes share the unpacking.
__device__ __forceinline__ float2 unpack2_split(uint32_t w) {
    uint32_t lo;
    asm("mul.lo.u32 %0, %1, 65536;" : "=r"(lo) : "r"(w));
    return make_float2(__uint_as_float(lo), __uint_as_float(w & 0xffff0000u));
}


// Weighted sums of the lane's expert pair for its 8 positions (the 16-byte
// chunk of each row): entry i2 is one float4 of weights (at wa + 512 i2) and
// four row chunks at xa + the 16-bit offsets of the pair's offset word (at
// oa + 256 i2, XORed with the lane's chunk, lxx); acc[j] (expert a) and
// acc[4 + j] (expert b) hold word j's positions lig + 16 j and lig + 16 j + 8.
// Entry i2 + 1's reads are issued before entry i2 is added.
__device__ __forceinline__ uint4 lds128u(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(a));
    return v;
}
struct MixEntry8 {
    float4 w;
    uint4 a0, a1, b0, b1;
};
__device__ __forceinline__ MixEntry8 mix_load8(uint32_t xa, uint32_t wa, uint2 o, uint32_t lxx,
                                               int i2) {
    MixEntry8 m;
    const uint32_t oa = o.x ^ lxx, ob = o.y ^ lxx;
    m.w = lds128f(wa + 512u * i2);
    m.a0 = lds128u(xa + (oa & 0xffffu));
    m.a1 = lds128u(xa + (oa >> 16));
    m.b0 = lds128u(xa + (ob & 0xffffu));
    m.b1 = lds128u(xa + (ob >> 16));
    return m;
}
__device__ __forceinline__ void mix_add4(float2 *acc, float w, const uint4 &v) {
    const float2 ww = make_float2(w, w);
    acc[0] = __ffma2_rn(ww, unpack2_split(v.x), acc[0]);
    acc[1] = __ffma2_rn(ww, unpack2_split(v.y), acc[1]);
    acc[2] = __ffma2_rn(ww, unpack2_split(v.z), acc[2]);
    acc[3] = __ffma2_rn(ww, unpack2_split(v.w), acc[3]);
}
__device__ __forceinline__ void mix_pair_full(uint32_t xa, uint32_t wa, uint32_t oa, uint32_t lxx,
                                              int npairs, float2 *acc) {
    uint2 on = lds64(oa + 256u);
    MixEntry8 cur = mix_load8(xa, wa, lds64(oa), lxx, 0);
#pragma unroll
    for (int i2 = 0; i2 < kGateMaxK / 2; ++i2) {
        if (i2 >= npairs) break;
        MixEntry8 nxt = cur;
        if (i2 + 1 < kGateMaxK / 2 && i2 + 1 < npairs) {
            nxt = mix_load8(xa, wa, on, lxx, i2 + 1);
            if (i2 + 2 < kGateMaxK / 2 && i2 + 2 < npairs) on = lds64(oa + 256u * (i2 + 2));
        }
        mix_add4(acc, cur.w.x, cur.a0);
        mix_add4(acc + 4, cur.w.z, cur.b0);
        mix_add4(acc, cur.w.y, cur.a1);
        mix_add4(acc + 4, cur.w.w, cur.b1);
        cur = nxt;
    }
}

template <bool F>
__device__ void mix_role(const RingParams &P, unsigned char *sm) {
    set_role_regs<kMixRegs, kLaunchRegs>();
    const int st = threadIdx.x;
    const int warp = st >> 5, lane = st & 31;
    const int h = lane / kGS, lig = lane % kGS;
    const uint32_t lx = (uint32_t)lig << 4;
    const int R = P.R, E = R + 1, kp = P.kp, NP = (R + 1) >> 1, Es = P.Es;
    const float *res = reinterpret_cast<const float *>(sm + P.off_res);
    // this group's expert pair (warp w's groups take pairs w + 8 h); padding
    // positions and the twin of an odd last expert read the zero row (their
    // weights are 0)
    const int pr = warp + kPairWarps * h;
    const int ea = 2 * pr, eb = ea + 1;
    const bool pair_on = pr < NP;
    // the offset table: entry (pair p, i2) at wslot(p, i2), two words of
    // row offsets without the lane's chunk (thread (p, i2) writes it)
    const uint32_t sm_a = smem_u32(sm);
    if (st < kWBlock) {
        const int p = st >> 3, i2 = st & 7;
        uint32_t o[4];
#pragma unroll
        for (int m = 0; m < 4; ++m) {
            const int e = 2 * p + (m >> 1), pos = 2 * i2 + (m & 1);
            const uint32_t c = (2 * p < R + 1 && e < R && pos < P.k)
                                   ? (uint32_t)__ldg(P.pidx + (size_t)e * P.k + pos)
                                   : (uint32_t)P.C;
            o[m] = row_off(c, 0u);
        }
        uint2 *ot = reinterpret_cast<uint2 *>(sm + P.off_offs);
        ot[wslot(p, i2)] = make_uint2(o[0] | (o[1] << 16), o[2] | (o[3] << 16));
    }
    bar_sync(kBarMix, kMixT);
    const uint32_t lxx = lx * 0x10001u;
    const uint32_t wlane = 16u * (uint32_t)(4 * (pr & 7) + (pr >> 3));  // wslot(pr, 0) * 16
    const uint32_t olane = sm_a + P.off_offs + 8u * (uint32_t)(4 * (pr & 7) + (pr >> 3));
    // item q: mix the slot with its table into ys[q.r mod kYB] and add the
    // residual column
    auto mix_item = [&](const ItemPos &q, uint32_t s) {
        const uint32_t r = q.r;
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys[r % kYB]);
        if (pair_on) {
            float2 acc[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] = make_float2(0.f, 0.f);
            mix_pair_full(sm_a + P.off_xs + s * P.xs_bytes, sm_a + P.off_tab[r % kNT] + wlane,
                          olane, lxx, kp >> 1, acc);
            // lane lig's positions are lig + 8 m: acc[m / 2], half m mod 2
            uint16_t *yh = ys + lig * Es + ea;
            const int stp = kGS * Es;
            if (P.bulk_y || eb == R) {
                // rows of odd length (or, for odd R, the twin's column is the
                // residual column, written below by another thread): 16-bit
                // stores
#pragma unroll
                for (int m = 0; m < 8; ++m) {
                    const float va = (m & 1) ? acc[m >> 1].y : acc[m >> 1].x;
                    const float vb = (m & 1) ? acc[4 + (m >> 1)].y : acc[4 + (m >> 1)].x;
                    yh[m * stp] = f32_to_bf16(va);
                    if (eb < R) yh[m * stp + 1] = f32_to_bf16(vb);
                }
            } else {
                uint32_t *yw = reinterpret_cast<uint32_t *>(yh);
                const int sw = stp >> 1;
#pragma unroll
                for (int m = 0; m < 8; ++m) {
                    const float va = (m & 1) ? acc[m >> 1].y : acc[m >> 1].x;
                    const float vb = (m & 1) ? acc[4 + (m >> 1)].y : acc[4 + (m >> 1)].x;
                    yw[m * sw] = pack_bf16x2(va, vb);
                }
            }
        }
        // the residual column (table role)
        if (st < q.np(P)) ys[st * Es + R] = f32_to_bf16(res[(r % kRS) * kTP + st]);
    };
    // item q's slot, table and residual column are read
    auto release = [&](const ItemPos &q, uint32_t s) {
        mbar_arrive(mbar(P, sm, kMbEmpty + s));
        mbar_arrive(mbar(P, sm, kMbTFree + q.r % kNT));
        mbar_arrive(mbar(P, sm, kMbRFree + q.r % kRS));
    };
    // rows of y not 16-byte aligned: 16-byte streaming stores between a
    // 16-bit head and tail
    auto store_item = [&](const ItemPos &q) {
        const uint16_t *ys = reinterpret_cast<const uint16_t *>(sm + P.off_ys[q.r % kYB]);
        const int cnt = q.np(P) * E;
        uint16_t *dst = P.y + ((size_t)q.n * P.HW + q.p0()) * E;
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
            for (int m = 0; m < 4; ++m) {
                const uint32_t lo = ys[p * Es + e];
                if (++e == E) { e = 0; ++p; }
                const uint32_t hi = ys[p * Es + e];
                if (++e == E) { e = 0; ++p; }
                w[m] = lo | (hi << 16);
            }
            __stcs(reinterpret_cast<uint4 *>(dst + o), make_uint4(w[0], w[1], w[2], w[3]));
        }
        for (int o = head + nv * 8 + st; o < cnt; o += kMixT) {
            const int p = fdiv(o, E, P.inv_E);
            __stcs(dst + o, ys[p * Es + (o - p * E)]);
        }
    };
    // rounds of two consecutive items (the last may have one)
    const uint32_t nb = cta_items(P);
    FullPhase fph;
    ItemPos q(P);
    while (q.r < nb) {
        ItemPos q2 = q;
        q2.next(P);
        const bool two = q2.r < nb;
        const uint32_t s1 = mix_slot<F>(P, q.r, nb), s2 = two ? mix_slot<F>(P, q2.r, nb) : 0u;
        const uint32_t fp1 = fph.take(s1), fp2 = two ? fph.take(s2) : 0u;
        // six threads wait for the two slots, tables and residual columns at
        // once, the others at the barrier; thread 0 has also seen the bulk
        // copies of the previous round finish reading their ys buffers
        bool ok = true;
        const int wi = st >> 5;
        if ((st & 31) == 0 && wi < (two ? 6 : 3)) {
            const ItemPos &w = wi < 3 ? q : q2;
            const uint32_t wr = w.r, wit = w.it;
            const int kind = wi % 3;
            if (kind == 0)
                ok = ring_wait(mbar(P, sm, kMbFull + (wi < 3 ? s1 : s2)), wi < 3 ? fp1 : fp2, P.ctrl,
                               wit);
            else if (kind == 1)
                ok = ring_wait(mbar(P, sm, kMbTReady + wr % kNT), (wr / kNT) & 1u, P.ctrl, wit);
            else
                ok = ring_wait(mbar(P, sm, kMbRDone + wr % kRS), (wr / kRS) & 1u, P.ctrl, wit);
        }
        if (!bar_and(kBarMix, kMixT, ok)) break;
        mix_item(q, s1);
        if (two) mix_item(q2, s2);
        if (P.bulk_y) {
            // [np][E] is contiguous in shared memory and in y: one bulk copy
            // per item, one group per round
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            bar_sync(kBarMix, kMixT);
            if (st == 0) {
                release(q, s1);
                if (two) release(q2, s2);
                for (int i = 0; i < (two ? 2 : 1); ++i) {
                    const ItemPos &w = i == 0 ? q : q2;
                    uint16_t *dst = P.y + ((size_t)w.n * P.HW + w.p0()) * E;
                    asm volatile(
                        "cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                        "r"(smem_u32(sm + P.off_ys[w.r % kYB])),
                        "r"((uint32_t)(w.np(P) * E) * 2u)
                        : "memory");
                }
                asm volatile(
                    "cp.async.bulk.commit_group;\n\t"
                    "cp.async.bulk.wait_group.read 1;" ::: "memory");
            }
        } else {
            bar_sync(kBarMix, kMixT);
            if (st == 0) {
                release(q, s1);
                if (two) release(q2, s2);
            }
            store_item(q);
            if (two) store_item(q2);
        }
        q = q2;
        if (two) q.next(P);
    }
    // bulk copies complete before the CTA exits
    if (st == 0 && P.bulk_y) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ================================================================ the mix kernel
template <bool F>
__global__ void __launch_bounds__(kRingT, 1) moce_ring_kernel(const RingParams P) {
    extern __shared__ __align__(128) unsigned char sm[];
    const int tid = threadIdx.x;
    const uint32_t epoch = ld_relaxed(P.ctrl + kCtrlEpoch);
    const uint32_t tag = epoch + 1u;
    const bool loader = tid >= kLoad0 && tid < kTab0;
    // set-up: U list, the zero row of every slot, mbarriers
    int32_t *s_resid = reinterpret_cast<int32_t *>(sm + P.off_U);
    for (int i = tid; i < P.nU; i += kRingT) s_resid[i] = __ldg(P.resid + i);
    for (int q = tid; q < P.D * (kRB / 4); q += kRingT) {
        const int d = q / (kRB / 4), w = q - d * (kRB / 4);
        reinterpret_cast<uint32_t *>(sm + P.off_xs + d * P.xs_bytes + (size_t)P.C * kRB)[w] = 0u;
    }
    if (tid == 0) {
        for (int d = 0; d < P.D; ++d) {
            mbar_init(mbar(P, sm, kMbRaw + d), 1);
            mbar_init(mbar(P, sm, kMbFull + d), 1);
            mbar_init(mbar(P, sm, kMbEmpty + d), 2);
        }
        for (int b = 0; b < kNT; ++b) {
            mbar_init(mbar(P, sm, kMbTReady + b), 1);
            mbar_init(mbar(P, sm, kMbTFree + b), 1);
        }
        for (int b = 0; b < kRS; ++b) {
            mbar_init(mbar(P, sm, kMbRDone + b), 1);
            mbar_init(mbar(P, sm, kMbRFree + b), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (tid < kMixT) mix_role<F>(P, sm);
    else if (loader) load_role<F>(P, sm, load_units(P, tid - kLoad0), tag);
    else if (tid < kProd0) table_role<F>(P, sm, tag);
    else copy_role<F>(P, sm);

    // the last CTA advances the epoch (the tag of the next forward)
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
    int D = 0, CG = 0, kp = 0, Es = 0, Kg = 0;
    size_t xs_bytes = 0, off_xs = 0, off_tab[kNT] = {}, off_ys[kYB] = {};
    size_t off_res = 0, off_rred = 0, off_U = 0, off_offs = 0, off_pool = 0, off_bar = 0;
    size_t smem = 0;
};

int sm_count() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms;
}

// Shared memory of pass 2: D slots of C + 1 staged rows (row C = zeros), kNT
// mixing tables, kYB output tiles, the residual partial sums, U, mbarriers.
// D is the largest count (at most kMaxD) that fits.
bool ring_plan(int C, int R, int k, bool bulk_y, bool fused, RingPlan *plan) {
    if (C % 8 != 0 || C < 8 || C > 256 || k < 1 || k > kGateMaxK || R < 1 || R > 2 * kMaxPairs)
        return false;
    RingPlan p;
    const int cgs = ((C >> 3) + 7) / 8;
    p.CG = cgs <= 1 ? 1 : (cgs <= 2 ? 2 : 4);
    p.kp = k + (k & 1);
    p.Es = bulk_y ? R + 1 : (R + 1) + ((R + 1) & 1);
    p.Kg = 16;
    p.xs_bytes = align_up((size_t)(C + 1) * kRB, 128);
    size_t off = 0;
    auto take = [&](size_t bytes, size_t al) {
        off = align_up(off, al);
        const size_t o = off;
        off += bytes;
        return o;
    };
    for (int b = 0; b < kNT; ++b) p.off_tab[b] = take((size_t)kWBlock * 16, 16);
    for (int b = 0; b < kYB; ++b) p.off_ys[b] = take((size_t)kTP * p.Es * 2, 16);
    p.off_res = take((size_t)kRS * kTP * 4, 16);
    p.off_rred = take((size_t)kResParts * kTP * 4, 16);
    p.off_U = take((size_t)C * 4, 16);
    p.off_offs = take((size_t)kWBlock * 8, 16);
    if (fused) p.off_pool = take(sizeof(PoolSmem), 16);
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

bool ring_supported(int N, int HW, int C, int R, int k, bool fused) {
    (void)N;
    RingPlan plan;
    return HW >= 1 && ring_plan(C, R, k, false, fused, &plan);
}

cudaError_t launch_ring(const uint16_t *x, int N, int HW, int C, int R, int k,
                        const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                        const float *W1, const float *b1, const float *w2, const float *b2,
                        float tmin, float tmax, uint16_t *y, const WsLayout &L, unsigned char *ws,
                        bool fused, cudaStream_t s) {
    const int G = sm_count();
    if (G < 1) return cudaErrorInvalidDevice;
    // every output tile [np][R + 1] starts and ends on a 16-byte boundary of y
    // when HW * (R + 1) is a multiple of 8: it leaves by one bulk copy
    const bool bulk_y =
        ((long long)HW * (R + 1)) % 8 == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0;
    RingPlan plan;
    if (!ring_plan(C, R, k, bulk_y, fused, &plan)) return cudaErrorNotSupported;
    const int T = (HW + kTP - 1) / kTP;
    const unsigned long long items = (unsigned long long)N * T;
    if (items >= 0xffff0000ull) return cudaErrorInvalidValue;

    // pass 1: pooling and gate
    PoolParams Q;
    Q.x = x;
    Q.N = N;
    Q.HW = HW;
    Q.C = C;
    Q.R = R;
    Q.k = k;
    Q.T = T;
    Q.pidx = pidx;
    Q.plog = plog;
    Q.W1 = W1;
    Q.b1 = b1;
    Q.w2 = w2;
    Q.b2 = b2;
    Q.tmin = tmin;
    Q.tmax = tmax;
    Q.ctrl = reinterpret_cast<uint32_t *>(ws + L.ctrl);
    Q.part = reinterpret_cast<unsigned long long *>(ws + L.partial);
    Q.zacc = reinterpret_cast<unsigned long long *>(ws + L.zacc);
    Q.count = reinterpret_cast<uint32_t *>(ws + L.sync);
    Q.made = Q.count + N;
    Q.wts = reinterpret_cast<float4 *>(ws + L.a);
    Q.z = reinterpret_cast<float *>(ws + L.z);
    Q.tau = reinterpret_cast<float *>(ws + L.tau);
    Q.kp = plan.kp;
    Q.Kg = plan.Kg;
    cudaError_t err = cudaSuccess;
    if (fused) {
        // single pass: every tile is its own run
        Q.RL = 1;
        Q.RPE = T;
        Q.runs = (uint32_t)items;
    } else {
    int per_sm = 0;
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, moce_poolgate_kernel, kPoolT, 0);
    if (err != cudaSuccess) return err;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // runs of RL tiles: about one resident wave of CTAs, at most 255 runs per
    // example (8-bit run counts in the accumulator words)
    {
        const long long slots = (long long)G * std::min(per_sm, kPoolCTAs);
        long long rpe = std::max<long long>(1, slots / std::max(1, N));  // runs fit one wave
        rpe = std::min<long long>(rpe, std::min<long long>(T, 255));
        Q.RL = (int)((T + rpe - 1) / rpe);
        Q.RPE = (T + Q.RL - 1) / Q.RL;
        Q.runs = (uint32_t)((unsigned long long)N * Q.RPE);
    }
    const unsigned long long g1 =
        std::min<unsigned long long>(Q.runs, (unsigned long long)G * std::min(per_sm, kPoolCTAs));
    moce_poolgate_kernel<<<(unsigned)g1, kPoolT, 0, s>>>(Q);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    }

    // pass 2 (or the single pass): mixing
    RingParams P;
    P.x = x;
    P.y = y;
    P.N = N;
    P.HW = HW;
    P.C = C;
    P.R = R;
    P.k = k;
    P.nU = nU;
    P.T = T;
    P.items = (uint32_t)items;
    P.pidx = pidx;
    P.resid = resid;
    P.ctrl = Q.ctrl;
    P.wts = Q.wts;
    P.made = Q.made;
    P.D = plan.D;
    P.CG = plan.CG;
    P.kp = plan.kp;
    P.Es = plan.Es;
    P.bulk_y = bulk_y ? 1 : 0;
    P.off_xs = (uint32_t)plan.off_xs;
    P.xs_bytes = (uint32_t)plan.xs_bytes;
    for (int b = 0; b < kNT; ++b) P.off_tab[b] = (uint32_t)plan.off_tab[b];
    for (int b = 0; b < kYB; ++b) P.off_ys[b] = (uint32_t)plan.off_ys[b];
    P.off_res = (uint32_t)plan.off_res;
    P.off_rred = (uint32_t)plan.off_rred;
    P.inv_nU = nU > 0 ? 1.0f / (float)nU : 0.0f;
    P.off_U = (uint32_t)plan.off_U;
    P.off_offs = (uint32_t)plan.off_offs;
    P.off_bar = (uint32_t)plan.off_bar;
    P.inv_E = 1.0f / (float)(R + 1);
    const void *kern = fused ? reinterpret_cast<const void *>(moce_ring_kernel<true>)
                             : reinterpret_cast<const void *>(moce_ring_kernel<false>);
    if ((err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)plan.smem)) != cudaSuccess)
        return err;
    const unsigned g2 = (unsigned)std::min<unsigned long long>(items, (unsigned long long)G);
    P.Gn = (int)(g2 / (unsigned)T);
    P.Gt = (int)(g2 % (unsigned)T);
    P.lead = kLead;
    P.off_pool = (uint32_t)plan.off_pool;
    P.pool = Q;
    if (!fused) {
        // programmatic dependent launch: the CTAs start on SMs that pass 1
        // has left and stage x while pass 1 finishes
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(g2);
        cfg.blockDim = dim3(kRingT);
        cfg.dynamicSmemBytes = plan.smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, moce_ring_kernel<false>, P);
    }
    // CTAs wait for gates that other CTAs of the launch run: all of them
    // must be resident (one per SM), which a cooperative launch guarantees
    int per_sm = 0;
    if ((err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, moce_ring_kernel<true>, kRingT,
                                                             plan.smem)) != cudaSuccess)
        return err;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel(kern, dim3(g2),
                                       dim3(kRingT), args, plan.smem, s);
}

}  // namespace moce
