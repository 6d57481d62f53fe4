// Two-pass forward of a MoCE layer (Sec. 3.3-3.4) for NHWC bf16 layers with
// C_in <= 256, C_out <= 64 and k <= 16.
//
// Every expert's temperature depends on the whole-image average of its
// support (Sec. 3.3), so no position of an example can be mixed before all
// of the example has been pooled. The examples are cut into tiles of 64
// positions (tile t of example n is item n*T + t).
//
// Pass 1, moce_poolgate_kernel, streams x once at full bandwidth: each CTA
// reduces a tile to its channel sums and adds them, as 64-bit fixed-point
// integers, into accumulator words of the example (integer sums do not
// depend on the order of the additions, so z is deterministic; a sum beyond
// the fixed-point range is kept as an epoch-tagged fp32 word instead). The
// CTA that counts an example's last tile reads z, evaluates the gate of
// every expert (Eq. (tau)) and the softmax weights (Eq. (weights)) and
// writes them in mixing-table order; it also clears the example's
// accumulators for the next forward.
//
// Mixing table: for expert pair p (experts 2p, 2p + 1) and support positions
// (2 i2, 2 i2 + 1), one float4 {w(2p, 2i2), w(2p, 2i2+1), w(2p+1, 2i2),
// w(2p+1, 2i2+1)} at entry [p][i2 ^ ((p >> 3) & 3)] of a [32][8] block: the
// four lane groups of a mixing warp (pairs 8 apart) read different banks.
//
// Pass 2, moce_ring_kernel, reads x again and mixes it: one CTA per SM takes
// items b, b + G, ...; its load warps (8-23) stage each tile, transposed to
// channel-major rows, into a ring of D shared-memory slots two tiles ahead;
// the table warps (24-27) copy the item's weights into one of three mixing
// tables and sum the tile's unselected channels for the residual expert
// (Eq. (res)); the mix warps (0-7) mix a slot with its table: each group of 8
// lanes owns 8 positions per lane and one expert pair for the whole launch,
// whose row offsets it keeps in registers (Eq. (expert)); the tile of y,
// residual column included, leaves by one bulk copy. The
// roles hand slots and tables over through shared-memory mbarriers (one
// thread waits, the others block at a barrier); every wait is bounded and
// none crosses CTAs.
#include <algorithm>

#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kTP = kRingTile;        // positions per tile
constexpr int kGS = 8;                // lanes of a mixing group
constexpr int kRB = 16 * kGS;         // bytes per staged channel row (kTP bf16)
constexpr int kFM = 7;                // chunk swizzle mask of the staged rows
constexpr int kMixT = 256;            // pass 2: mix warps 0-7
constexpr int kLoadT = 512;           // pass 2: load warps 8-23
constexpr int kTabT = 128;            // pass 2: table warps 24-27
constexpr int kRingT = kMixT + kLoadT + kTabT;
constexpr int kLoad0 = kMixT;                    // first load thread
constexpr int kTab0 = kMixT + kLoadT;            // first table thread
constexpr int kResParts = kTabT / 8;             // residual: U entries split kResParts ways
constexpr int kMixWarps = kMixT / 32;
constexpr int kNT = 3;                // mixing tables
constexpr int kYB = 2;                // output tile buffers
constexpr int kRS = 4;                // residual columns (the table role runs ahead)
constexpr int kMaxD = 6;              // x slots at most
constexpr int kGateMaxK = 16;          // support positions a mixing lane keeps in registers
constexpr int kMaxPairs = 32;          // expert pairs: one per mixing group
constexpr int kWBlock = kMaxPairs * 8; // float4 entries of a weight block
constexpr int kBarMix = 1, kBarLoad = 2, kBarTab = 3;
// Registers per thread: the launch gives every thread 72 (kRingT * 72 <=
// 65536); the roles then trade them with setmaxnreg within that total (the
// mixing loop keeps its row offsets in registers).
constexpr int kLaunchRegs = 72, kMixRegs = 96, kLoadRegs = 64, kTabRegs = 56;
static_assert(kMixT * kMixRegs + kLoadT * kLoadRegs + kTabT * kTabRegs <= kRingT * kLaunchRegs,
              "register split exceeds the launch allocation");
static_assert(kMixT % 128 == 0 && kLoadT % 128 == 0 && kTabT % 128 == 0, "whole warpgroups");
constexpr int kPoolT = 256;           // pass 1 threads per CTA
constexpr int kPoolCTAs = 8;          // pass 1 CTAs per SM
constexpr int kAccG = 4;              // accumulator words per (example, channel)
static_assert(kRingT * kLaunchRegs <= 65536, "launch registers at one CTA per SM");
static_assert(kMixT == 4 * kTP, "four mixing threads per position in the epilogue");
static_assert(kTP == 8 * kGS, "a group's lanes cover the tile");
static_assert(kPoolT == 4 * kTP, "pass 1: 32 channel blocks x 8 rows of positions");

// Accumulator word of one (example, channel, group): bits 48-55 count the
// runs published as fp32 instead, bits 0-47 hold the sum of
// kFixBias + round(s * 2^20) over the fixed-point runs (s = the run's
// channel sum, |s| < 2^19, so every term is in (0, 2^40) and any count of
// runs below 256 fits).
constexpr float kFixScale = 1048576.0f;  // 2^20
constexpr float kFixInv = 1.0f / 1048576.0f;
constexpr float kFixMax = 524288.0f;     // 2^19
constexpr unsigned long long kFixBias = 1ull << 39;
constexpr unsigned long long kWideOne = 1ull << 48;

// mbarriers of pass 2 (8 bytes each): full[s] (load -> mix, table), empty[s]
// (mix and table -> load: two arrivals), tready[b] (table -> mix), tfree[b]
// (mix -> table), rdone[c] (table -> mix: residual column c), rfree[c]
// (mix -> table).
constexpr int kMbFull = 0, kMbEmpty = kMaxD, kMbTReady = 2 * kMaxD, kMbTFree = 2 * kMaxD + kNT,
              kMbRDone = 2 * kMaxD + 2 * kNT, kMbRFree = 2 * kMaxD + 2 * kNT + kRS,
              kMbWords = 2 * kMaxD + 2 * kNT + 2 * kRS;

// float4 entry of expert pair p, support positions (2 i2, 2 i2 + 1), in a
// weight block.
__device__ __forceinline__ int wslot(int p, int i2) { return p * 8 + (i2 ^ ((p >> 3) & 3)); }

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
    uint32_t off_res, off_rred, off_U, off_bar;
    float inv_nU;                 // 1 / |U| (0 when U is empty)
    float inv_E;
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
                                          float4 *wts, float *tau_out) {
    constexpr int TPE = K / 4;             // threads per expert
    constexpr int EPP = kPoolT / TPE;      // experts per pass
    const int st = threadIdx.x;
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
};

// The example's gate, by its last pooling CTA: z from the accumulator words
// (and the tagged fp32 run sums, in run order), then every expert's
// temperature and weights; the accumulators and the counter are cleared for
// the next forward.
__device__ void finish_example(const PoolParams &P, PoolSmem &S, int n, uint32_t tag) {
    const int tid = threadIdx.x;
    const unsigned long long T = (unsigned long long)P.RPE;  // runs of the example
    unsigned long long *za = P.zacc + (size_t)n * kAccG * P.C;
    for (int c = tid; c < P.C; c += kPoolT) {
        long long fx = 0;
        bool wide = false;
#pragma unroll
        for (int g = 0; g < kAccG; ++g) {
            const unsigned long long Tg = (T - (unsigned long long)g + kAccG - 1) / kAccG;
            const unsigned long long w = __ldcg(za + (size_t)g * P.C + c);
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
    __syncthreads();
    SupTab sup;
    sup.idx = P.pidx;
    sup.lg = P.plog;
    sup.se = P.k;
    sup.si = 1;
    float4 *wts = P.wts + (size_t)n * kWBlock;
    // entries no expert writes (padding positions, the twin of an odd last
    // expert) stay 0
    for (int q = tid; q < kWBlock; q += kPoolT) wts[q] = make_float4(0.f, 0.f, 0.f, 0.f);
    __syncthreads();
    float *tau = P.tau + (size_t)n * P.R;
    if (P.Kg == 16) gate_experts<16>(P, S.W1t, S.b1, S.w2, S.zs, sup, wts, tau);
    else gate_experts<32>(P, S.W1t, S.b1, S.w2, S.zs, sup, wts, tau);
    if (tid == 0) P.made[n] = tag;  // read by pass 2 after this kernel ends
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
                add = kFixBias + (unsigned long long)__float2ll_rn(s * kFixScale);
            } else {  // beyond the fixed-point range (or NaN): a tagged fp32 word
                P.part[((size_t)n * P.RPE + j) * P.C + tid] =
                    ((unsigned long long)tag << 32) | __float_as_uint(s);
                add = kWideOne;
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
            finish_example(P, S, n, tag);
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
// q = (w + 16 i) / CG for i = 0, 1 while w + 16 i < 8 CG; a warp's loads
// read 128 contiguous bytes per position and its stores hit 32 banks.
struct LoadUnits {
    int nu;          // units per tile (0..2)
    int cc;          // 8-channel block
    bool own;        // cc < C / 8
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

// One item of the load role: store the tile held in v into slot r mod D and
// refill v with the loads of the item two ahead. False when a wait gave up.
__device__ __forceinline__ bool load_item(const RingParams &P, unsigned char *sm,
                                          const LoadUnits &u, uint32_t it, uint32_t r, uint4 *v) {
    const int lt = threadIdx.x - kLoad0;
    const uint32_t s = r % (uint32_t)P.D;
    // slot s is free once the mix role is done with item r - D
    bool ok = true;
    if (lt == 0 && r >= (uint32_t)P.D)
        ok = ring_wait(mbar(P, sm, kMbEmpty + s), ((r / P.D) - 1u) & 1u, P.ctrl, it);
    if (!bar_and(kBarLoad, kLoadT, ok)) return false;
    unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
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
    // the item two ahead is in flight while the next one is stored
    tile_loads(P, u, it + 2u * gridDim.x, v);
    bar_sync(kBarLoad, kLoadT);
    if (lt == 0) mbar_arrive(mbar(P, sm, kMbFull + s));
    return true;
}

// Items alternate between the two register sets (unrolled by two, so each
// set stays in registers).
__device__ void load_role(const RingParams &P, unsigned char *sm, const LoadUnits &u, uint4 *va,
                          uint4 *vb) {
    set_role_regs<kLoadRegs, kLaunchRegs>();
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

// The table role, per item r: copies the weights of the item's example
// (pass 1) into table r mod kNT (an example whose weights pass 1 of this
// forward did not produce, because a tile was never counted, is reported as
// MOCE_ERR_TIMEOUT); then, once the tile is staged, the residual expert
// (Eq. (res)): thread (q = chunk, part) adds U entries part, part +
// kResParts, ... for the chunk's 8 positions, the parts are added in order,
// and res[r mod kYB][p] = sum / |U| (0 if U is empty).
__device__ void table_role(const RingParams &P, unsigned char *sm, uint32_t tag) {
    set_role_regs<kTabRegs, kLaunchRegs>();
    const int tt = threadIdx.x - kTab0;
    const int q = tt & 7, part = tt >> 3;
    const uint32_t lx = (uint32_t)q << 4;
    const int32_t *s_resid = reinterpret_cast<const int32_t *>(sm + P.off_U);
    float *rred = reinterpret_cast<float *>(sm + P.off_rred);
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t tb = r % kNT, s = r % (uint32_t)P.D, rc = r % kRS;
        const int n = (int)(it / (uint32_t)P.T);
        bool ok = true;
        if (tt == 0 && r >= (uint32_t)kNT)
            ok = ring_wait(mbar(P, sm, kMbTFree + tb), ((r / kNT) - 1u) & 1u, P.ctrl, it);
        if (!bar_and(kBarTab, kTabT, ok)) break;
        if (tt == 0 && __ldg(P.made + n) != tag) report_timeout(P.ctrl, it);
        {
            const float4 *wn = P.wts + (size_t)n * kWBlock;
            float4 *tab = reinterpret_cast<float4 *>(sm + P.off_tab[tb]);
            float4 w[kWBlock / kTabT];
#pragma unroll
            for (int j = 0; j < kWBlock / kTabT; ++j) w[j] = __ldg(wn + tt + kTabT * j);
#pragma unroll
            for (int j = 0; j < kWBlock / kTabT; ++j) tab[tt + kTabT * j] = w[j];
        }
        bar_sync(kBarTab, kTabT);
        if (tt == 0) {
            mbar_arrive(mbar(P, sm, kMbTReady + tb));
            ok = ring_wait(mbar(P, sm, kMbFull + s), (r / P.D) & 1u, P.ctrl, it);
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
}

// ================================================================ mix role
// Row offset (bytes in a slot) of channel c for the lane whose chunk mask is
// lx: row c, chunk ((c >> 3) & 7) ^ lane; channel C is the zero row.
__device__ __forceinline__ uint32_t row_off(uint32_t c, uint32_t lx) {
    return ((c * kRB) | (((c >> 3) & kFM) << 4)) ^ lx;
}

// Weighted sums of the lane's expert pair for its 8 positions: per entry i2,
// one float4 of weights and four 16-byte row chunks whose offsets the lane
// holds in registers (offs[2 i2]: expert a, positions 2 i2 and 2 i2 + 1, low
// and high half; offs[2 i2 + 1]: expert b).
__device__ __forceinline__ void mix_pair_regs(const unsigned char *xs, const float4 *wt, int pr,
                                              int npairs, const uint32_t *offs, float2 &a0,
                                              float2 &a1, float2 &a2, float2 &a3, float2 &b0,
                                              float2 &b1, float2 &b2, float2 &b3) {
#pragma unroll
    for (int i2 = 0; i2 < kGateMaxK / 2; ++i2) {
        if (i2 >= npairs) break;
        const float4 w = wt[wslot(pr, i2)];
        const uint32_t oa = offs[2 * i2], ob = offs[2 * i2 + 1];
        const uint4 va0 = lds128(xs + (oa & 0xffffu));
        const uint4 va1 = lds128(xs + (oa >> 16));
        const uint4 vb0 = lds128(xs + (ob & 0xffffu));
        const uint4 vb1 = lds128(xs + (ob >> 16));
        const float2 wa0 = make_float2(w.x, w.x), wa1 = make_float2(w.y, w.y);
        const float2 wb0 = make_float2(w.z, w.z), wb1 = make_float2(w.w, w.w);
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
    set_role_regs<kMixRegs, kLaunchRegs>();
    const int st = threadIdx.x;
    const int warp = st >> 5, lane = st & 31;
    const int h = lane / kGS, lig = lane % kGS;
    const uint32_t lx = (uint32_t)lig << 4;
    const int R = P.R, E = R + 1, kp = P.kp, NP = (R + 1) >> 1, Es = P.Es;
    const float *res = reinterpret_cast<const float *>(sm + P.off_res);
    // this group's expert pair (warp w's groups take pairs w + 8h) and its
    // row offsets, fixed for the whole launch; padding positions and the twin
    // of an odd last expert read the zero row (their weights are 0)
    const int pr = warp + kMixWarps * h;
    const int ea = 2 * pr, eb = ea + 1;
    const bool pair_on = pr < NP;
    uint32_t offs[kGateMaxK];
#pragma unroll
    for (int i = 0; i < kGateMaxK; i += 2) {
        uint32_t o[4];
#pragma unroll
        for (int m = 0; m < 4; ++m) {
            const int e = m < 2 ? ea : eb, pos = i + (m & 1);
            const uint32_t c = (pair_on && e < R && pos < P.k)
                                   ? (uint32_t)__ldg(P.pidx + (size_t)e * P.k + pos)
                                   : (uint32_t)P.C;
            o[m] = row_off(c, lx);
        }
        offs[i] = o[0] | (o[1] << 16);
        offs[i + 1] = o[2] | (o[3] << 16);
    }
    uint32_t r = 0;
    for (uint32_t it = blockIdx.x; it < P.items; it += gridDim.x, ++r) {
        const uint32_t s = r % (uint32_t)P.D, tb = r % kNT, yb = r % kYB, rc = r % kRS;
        const int n = (int)(it / (uint32_t)P.T), t = (int)(it - (uint32_t)n * P.T);
        // one thread waits for the slot and the table, the others at the
        // barrier; thread 0 has also seen the bulk copy of item r - kYB
        // finish reading ys
        bool ok = true;
        if (st == 0) {
            ok = ring_wait(mbar(P, sm, kMbFull + s), (r / P.D) & 1u, P.ctrl, it) &&
                 ring_wait(mbar(P, sm, kMbTReady + tb), (r / kNT) & 1u, P.ctrl, it) &&
                 ring_wait(mbar(P, sm, kMbRDone + rc), (r / kRS) & 1u, P.ctrl, it);
        }
        if (!bar_and(kBarMix, kMixT, ok)) break;
        const unsigned char *xs = sm + P.off_xs + s * P.xs_bytes;
        uint16_t *ys = reinterpret_cast<uint16_t *>(sm + P.off_ys[yb]);
        const float4 *wt = reinterpret_cast<const float4 *>(sm + P.off_tab[tb]);
        if (pair_on) {
            float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
            float2 b0 = a0, b1 = a0, b2 = a0, b3 = a0;
            mix_pair_regs(xs, wt, pr, kp >> 1, offs, a0, a1, a2, a3, b0, b1, b2, b3);
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
            } else if (eb == R) {
                // odd R: the twin's column is the residual column, written
                // below by another thread
                uint16_t *yh = ys + lig * Es + ea;
                const int stp = kGS * Es;
                const float av[8] = {a0.x, a0.y, a1.x, a1.y, a2.x, a2.y, a3.x, a3.y};
#pragma unroll
                for (int q = 0; q < 8; ++q) yh[q * stp] = f32_to_bf16(av[q]);
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
        // the residual column (table role)
        const int p0 = t * kTP, np = min(kTP, P.HW - p0);
        if (st < np) ys[st * Es + R] = f32_to_bf16(res[rc * kTP + st]);
        const int cnt = np * E;
        uint16_t *dst = P.y + ((size_t)n * P.HW + p0) * E;
        if (P.bulk_y) {
            // [np][E] is contiguous in shared memory and in y: one bulk copy
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            bar_sync(kBarMix, kMixT);
            if (st == 0) {
                // the slot, the table and the residual column are read
                mbar_arrive(mbar(P, sm, kMbEmpty + s));
                mbar_arrive(mbar(P, sm, kMbTFree + tb));
                mbar_arrive(mbar(P, sm, kMbRFree + rc));
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
        if (st == 0) {
            // the slot, the table and the residual column are read
            mbar_arrive(mbar(P, sm, kMbEmpty + s));
            mbar_arrive(mbar(P, sm, kMbTFree + tb));
            mbar_arrive(mbar(P, sm, kMbRFree + rc));
        }
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

// ================================================================ the mix kernel
__global__ void __launch_bounds__(kRingT, 1) moce_ring_kernel(const RingParams P) {
    extern __shared__ __align__(128) unsigned char sm[];
    const int tid = threadIdx.x;
    const uint32_t epoch = ld_relaxed(P.ctrl + kCtrlEpoch);
    const uint32_t tag = epoch + 1u;
    const bool loader = tid >= kLoad0 && tid < kTab0;
    // the load role's first two tiles are in flight during the set-up
    LoadUnits lu;
    uint4 va[4], vb[4];
    if (loader) {
        lu = load_units(P, tid - kLoad0);
        tile_loads(P, lu, blockIdx.x, va);
        tile_loads(P, lu, blockIdx.x + gridDim.x, vb);
    }
    // set-up: U list, the zero row of every slot, mbarriers
    int32_t *s_resid = reinterpret_cast<int32_t *>(sm + P.off_U);
    for (int i = tid; i < P.nU; i += kRingT) s_resid[i] = __ldg(P.resid + i);
    for (int q = tid; q < P.D * (kRB / 4); q += kRingT) {
        const int d = q / (kRB / 4), w = q - d * (kRB / 4);
        reinterpret_cast<uint32_t *>(sm + P.off_xs + d * P.xs_bytes + (size_t)P.C * kRB)[w] = 0u;
    }
    if (tid == 0) {
        for (int d = 0; d < P.D; ++d) {
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

    if (tid < kMixT) mix_role(P, sm);
    else if (loader) load_role(P, sm, lu, va, vb);
    else table_role(P, sm, tag);

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
    size_t off_res = 0, off_rred = 0, off_U = 0, off_bar = 0, smem = 0;
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
bool ring_plan(int C, int R, int k, bool bulk_y, RingPlan *plan) {
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
    (void)N;
    RingPlan plan;
    return HW >= 1 && ring_plan(C, R, k, false, &plan);
}

cudaError_t launch_ring(const uint16_t *x, int N, int HW, int C, int R, int k,
                        const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                        const float *W1, const float *b1, const float *w2, const float *b2,
                        float tmin, float tmax, uint16_t *y, const WsLayout &L, unsigned char *ws,
                        cudaStream_t s) {
    const int G = sm_count();
    if (G < 1) return cudaErrorInvalidDevice;
    // every output tile [np][R + 1] starts and ends on a 16-byte boundary of y
    // when HW * (R + 1) is a multiple of 8: it leaves by one bulk copy
    const bool bulk_y =
        ((long long)HW * (R + 1)) % 8 == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0;
    RingPlan plan;
    if (!ring_plan(C, R, k, bulk_y, &plan)) return cudaErrorNotSupported;
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
    int per_sm = 0;
    cudaError_t err =
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, moce_poolgate_kernel, kPoolT, 0);
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

    // pass 2: mixing
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
    P.off_bar = (uint32_t)plan.off_bar;
    P.inv_E = 1.0f / (float)(R + 1);
    if ((err = cudaFuncSetAttribute(moce_ring_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)plan.smem)) != cudaSuccess)
        return err;
    const unsigned g2 = (unsigned)std::min<unsigned long long>(items, (unsigned long long)G);
    moce_ring_kernel<<<g2, kRingT, plan.smem, s>>>(P);
    return cudaGetLastError();
}

}  // namespace moce
