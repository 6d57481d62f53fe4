// Fused persistent forward kernel: pooling, gate, softmax weights, routed
// mixing and the residual expert of a MoCE layer (Sec. 3.3-3.4) in one
// launch, for NHWC bf16 inputs with gate width k <= 64.
//
// The temperature of every expert depends on the whole-image average of its
// support (Sec. 3.3), so an example can only be mixed after all of it has
// been pooled and x is needed twice. This kernel reads x from HBM once and
// keeps both passes busy on every SM at the same time, with two warp groups
// per CTA (one CTA per SM, cooperative launch so that all are resident):
//
//   pool group (4 warps)  streams pooling tiles of x from HBM through
//       registers and writes per-tile channel sums. It never waits, so it
//       runs ahead of the mix group.
//   mix group (8 warps)   runs, in order, GATE(n, b) and MIX(n, t) items:
//       GATE reduces the tile sums of example n to z[n] in tile order,
//       evaluates the gate of expert block b (Eq. (tau)) and writes the
//       softmax weights (Eq. (weights)). MIX stages a tile of x[n] - re-read
//       from L2, the pool group read it shortly before - transposed in shared
//       memory, and computes the routed mix (Eq. (expert)) and the residual
//       (Eq. (res)).
//
// Values passed between CTAs (tile sums, weights) are 64-bit words holding
// the fp32 value and a tag, epoch + 1, written with one single-copy-atomic
// store (epoch = completed forwards on this workspace; the last CTA to exit
// bumps it). A reader knows a value is current from its own tag, so no
// separate ready flags or acquire/release chains are needed, and the weights
// of the next MIX item are loaded together with its x tile while the current
// item computes.
//
// The mix group's list holds GATE(s) and MIX(s - lag) at stage s, and CTA b
// processes items b, b + G, ... of each list in order. MIX only waits for
// GATE items earlier in the same list, GATE only for pooling tiles, and the
// pool group never waits, so the unfinished item with the smallest index can
// always run and every wait ends. Each wait is nevertheless bounded
// (kSpinLimit polls); one that gives up records MOCE_ERR_TIMEOUT in the
// workspace and makes every other wait return, so the kernel always exits.
#include "moce_device.cuh"

namespace moce {
namespace {

constexpr int kMixThreads = kThreads;                  // mix group: warps 0-7
constexpr int kPoolThreads = 128;                      // pool group: warps 8-11
constexpr int kFusedThreads = kMixThreads + kPoolThreads;
constexpr int kBarMix = 1, kBarPool = 2;               // named barriers of the groups
constexpr int kPref = 16;                              // 16-byte prefetch registers, mix thread
constexpr int kPoolPref = 32;                          // 16-byte prefetch registers, pool thread
constexpr int kWPref = 4;                              // prefetched table weights per mix thread
constexpr int kGateMaxK = 64;                          // gate width of the one-warp-per-expert gate
constexpr int kMixWarps = kMixThreads / 32;

enum : int { kNone = 0, kGate = 1, kMix = 2 };

struct FusedParams {
    const uint16_t *x;
    uint16_t *y;
    int N, HW, C, R, k, nU;
    const int32_t *pidx;
    const float *plog;
    const int32_t *resid;
    const float *W1, *b1, *w2, *b2;
    float tmin, tmax;
    uint32_t *ctrl;
    unsigned long long *partial;  // tagged tile sums [N][PT][C]
    unsigned long long *a;        // tagged weights [N][R][k]
    float *z, *tau;
    int PP, PT;        // pooling tile positions, pooling tiles per example
    int MT;            // mixing tiles per example
    int GB;            // gate blocks per example
    int lag;           // stages between GATE(n) and MIX(n) in the mix list
    uint32_t pool_items, mix_items;
    MixGeom geom;
    int Es;            // row stride (elements) of the staged output tile, even
    int static_off;    // table offsets written once per CTA (every expert in one chunk)
    int wpref;         // table weights of the next MIX item may be prefetched
    int ks;            // padded row of the shared-memory copy of W1
    size_t off_static; // persistent shared memory: U list, W1, b1, w2, [pidx, plog]
    int gate_tabs;     // support channels and logits are in shared memory
    size_t off_us;     // gate scratch: per-warp gate input vectors (after z)
    size_t off_red;    // pool group's reduction buffer
    float inv_perq, inv_E, inv_kp;  // 1/d for the divisions by 4*CCp, R+1 and kp
};

struct Item {
    int kind, n, t;
};

__device__ __forceinline__ void add8(float *acc, const uint4 v) {
    acc[0] += bf16lo(v.x); acc[1] += bf16hi(v.x);
    acc[2] += bf16lo(v.y); acc[3] += bf16hi(v.y);
    acc[4] += bf16lo(v.z); acc[5] += bf16hi(v.z);
    acc[6] += bf16lo(v.w); acc[7] += bf16hi(v.w);
}

// ================================================================ pool group
struct PoolMap {
    int V, span, rows, row, cvl, ppt;
    bool pref;  // this thread's part of a tile fits the prefetch registers
};

__device__ __forceinline__ PoolMap pool_map(const FusedParams &P, int pt) {
    PoolMap m;
    m.V = P.C >> 3;
    m.span = m.V < kPoolThreads ? m.V : kPoolThreads;
    m.rows = kPoolThreads / m.span;
    m.row = pt / m.span;
    m.cvl = pt - m.row * m.span;
    m.ppt = (P.PP + m.rows - 1) / m.rows;
    m.pref = (m.V <= kPoolThreads) && (m.ppt <= kPoolPref);
    return m;
}

__device__ __forceinline__ void pool_prefetch(const FusedParams &P, const PoolMap &m, uint32_t j,
                                              uint4 *pre) {
    if (j >= P.pool_items || !m.pref || m.row >= m.rows) return;
    const int n = (int)(j / (uint32_t)P.PT), t = (int)(j - (uint32_t)n * P.PT);
    const int p0 = t * P.PP, np = min(P.PP, P.HW - p0);
    const uint16_t *col = P.x + ((size_t)n * P.HW + p0) * P.C + m.cvl * 8;
#pragma unroll
    for (int s = 0; s < kPoolPref; ++s) {
        const int p = m.row + s * m.rows;
        if (s < m.ppt && p < np) pre[s] = ld_stream(col + (size_t)p * P.C);
    }
}

__device__ void pool_loop(const FusedParams &P, unsigned char *sm, uint32_t ready, uint32_t drop) {
    const int pt = threadIdx.x - kMixThreads;
    const PoolMap m = pool_map(P, pt);
    float *red = reinterpret_cast<float *>(sm + P.off_red);
    uint4 pre[kPoolPref];
#pragma unroll
    for (int s = 0; s < kPoolPref; ++s) pre[s] = make_uint4(0u, 0u, 0u, 0u);
    uint32_t j = blockIdx.x;
    pool_prefetch(P, m, j, pre);
    for (; j < P.pool_items; j += gridDim.x) {
        const int n = (int)(j / (uint32_t)P.PT), t = (int)(j - (uint32_t)n * P.PT);
        const int p0 = t * P.PP, np = min(P.PP, P.HW - p0);
        unsigned long long *out = P.partial + ((size_t)n * P.PT + t) * P.C;
        const bool publish = j + 1u != drop;
        bar_sync(kBarPool, kPoolThreads);  // red of the previous tile is consumed
        if (m.row < m.rows) {
            if (m.pref) {
                float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int s = 0; s < kPoolPref; ++s) {
                    const int p = m.row + s * m.rows;
                    if (s < m.ppt && p < np) add8(acc, pre[s]);
                }
                if (m.rows > 1) {
                    float4 *dst = reinterpret_cast<float4 *>(red + (m.row * m.span + m.cvl) * 8);
                    dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
                    dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
                } else if (publish) {
#pragma unroll
                    for (int q = 0; q < 8; ++q) st_tagged(out + m.cvl * 8 + q, acc[q], ready);
                }
            } else {
                const uint16_t *xt = P.x + ((size_t)n * P.HW + p0) * P.C;
                for (int cv = m.cvl; cv < m.V; cv += m.span) {
                    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                    for (int p = m.row; p < np; p += m.rows)
                        add8(acc, ld_stream(xt + (size_t)p * P.C + cv * 8));
                    if (m.rows > 1) {
                        float4 *dst = reinterpret_cast<float4 *>(red + (m.row * m.span + cv) * 8);
                        dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
                        dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
                    } else if (publish) {
#pragma unroll
                        for (int q = 0; q < 8; ++q) st_tagged(out + cv * 8 + q, acc[q], ready);
                    }
                }
            }
        }
        pool_prefetch(P, m, j + gridDim.x, pre);
        if (m.rows > 1) {
            bar_sync(kBarPool, kPoolThreads);
            for (int q = pt; q < m.span * 8; q += kPoolThreads) {
                float s = 0.f;
                for (int r = 0; r < m.rows; ++r) s += red[r * m.span * 8 + q];
                if (publish) st_tagged(out + q, s, ready);
            }
        }
    }
}

// ================================================================ mix group
// Items of the mix list before stage s: GATE(s') for s' < s, MIX(s' - lag).
__device__ __forceinline__ uint32_t mix_items_before(const FusedParams &P, int s) {
    const int g = min(s, P.N);
    const int m = min(max(s - P.lag, 0), P.N);
    return (uint32_t)g * P.GB + (uint32_t)m * P.MT;
}

__device__ Item mix_decode(const FusedParams &P, uint32_t i) {
    Item it{kNone, 0, 0};
    if (i >= P.mix_items) return it;
    int lo = 0, hi = P.N + P.lag;  // items_before(lo) <= i < items_before(hi)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (mix_items_before(P, mid) <= i) lo = mid;
        else hi = mid;
    }
    int r = (int)(i - mix_items_before(P, lo));
    if (lo < P.N) {
        if (r < P.GB) return Item{kGate, lo, r};
        r -= P.GB;
    }
    return Item{kMix, lo - P.lag, r};
}

// ---------------------------------------------------------------- GATE
__device__ void gate_item(const FusedParams &P, int n, int b, unsigned char *sm,
                          const float *W1s, const float *b1s, const float *w2s,
                          const int32_t *pidx_s, const float *plog_s, uint32_t ready,
                          uint32_t item, bool publish) {
    float *zs = reinterpret_cast<float *>(sm);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *uw = reinterpret_cast<float *>(sm + P.off_us) + warp * P.k;

    // z[n] = (sum of the tile sums, in tile order) / HW; each sum waits for its tag
    bool ok = true;
    const unsigned long long *pn = P.partial + (size_t)n * P.PT * P.C;
    for (int c = threadIdx.x; c < P.C && ok; c += kMixThreads) {
        const unsigned long long *pc = pn + c;
        float s = 0.f;
        for (int t0 = 0; t0 < P.PT && ok; t0 += 8) {
            unsigned long long v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (t0 + u < P.PT) v[u] = ld_tagged(pc + (size_t)(t0 + u) * P.C);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (t0 + u < P.PT && ok) {
                    if (!tag_ok(v[u], ready))
                        ok = wait_tagged(pc + (size_t)(t0 + u) * P.C, ready, v[u], P.ctrl, item);
                    s += tag_val(v[u]);
                }
            }
        }
        const float zc = s / (float)P.HW;
        zs[c] = zc;
        if (b == 0) P.z[(size_t)n * P.C + c] = zc;
    }
    if (!bar_and(kBarMix, kMixThreads, ok)) return;

    // one warp per expert: u = z at the support in deployment order,
    // h = ReLU(W1 u + b1) with a lane per hidden unit, g = w2 . h + b2,
    // tau (Eq. (tau)) and the weights a = softmax(L / tau) (Eq. (weights))
    const int k = P.k, ks = P.ks;
    const float b2 = __ldg(P.b2);
    const int e_end = min(P.R, (b + 1) * kGateExperts);
    for (int e = b * kGateExperts + warp; e < e_end; e += kMixWarps) {
        const int32_t *ie = (P.gate_tabs ? pidx_s : P.pidx) + (size_t)e * k;
        const float *L = (P.gate_tabs ? plog_s : P.plog) + (size_t)e * k;
        for (int i = lane; i < k; i += 32) uw[i] = zs[ie[i]];
        __syncwarp();
        float gp = 0.f;
        for (int j = lane; j < k; j += 32) {
            const float *wr = W1s + j * ks;
            float h = b1s[j];
            for (int i = 0; i < k; ++i) h = fmaf(wr[i], uw[i], h);
            gp = fmaf(w2s[j], fmaxf(h, 0.f), gp);
        }
        const float g = warp_sum(gp) + b2;
        const float tau = P.tmin + (P.tmax - P.tmin) / (1.f + expf(-g));
        const float L0 = L[0];  // position 0 holds the largest logit
        const float ex0 = lane < k ? expf((L[lane] - L0) / tau) : 0.f;
        const float ex1 = lane + 32 < k ? expf((L[lane + 32] - L0) / tau) : 0.f;
        const float zsum = warp_sum(ex0 + ex1);
        unsigned long long *ae = P.a + ((size_t)n * P.R + e) * k;
        if (publish) {
            if (lane < k) st_tagged(ae + lane, ex0 / zsum, ready);
            if (lane + 32 < k) st_tagged(ae + lane + 32, ex1 / zsum, ready);
        }
        if (lane == 0) P.tau[(size_t)n * P.R + e] = tau;
        __syncwarp();
    }
}

// ---------------------------------------------------------------- MIX
template <int GS>
__device__ __forceinline__ void mix_prefetch(const FusedParams &P, const Item &it, uint4 *pre) {
    constexpr int TP = 8 * GS;
    const int p0 = it.t * TP, np = min(TP, P.HW - p0);
    const int CC = P.C >> 3, CCp = (CC + 7) & ~7, per_q = 4 * CCp, units = GS * per_q;
    const uint16_t *xt = P.x + ((size_t)it.n * P.HW + p0) * P.C;
#pragma unroll
    for (int r = 0; r < kPref / 2; ++r) {
        const int u = threadIdx.x + r * kMixThreads;
        int q, j, cc;
        stage_unit_coords(u, per_q, P.inv_perq, q, j, cc);
        const int pa = q + 2 * GS * j, pb = pa + GS;
        uint4 va = make_uint4(0u, 0u, 0u, 0u), vb = va;
        if (u < units && cc < CC) {
            if (pa < np) va = __ldcs(reinterpret_cast<const uint4 *>(xt + (size_t)pa * P.C + cc * 8));
            if (pb < np) vb = __ldcs(reinterpret_cast<const uint4 *>(xt + (size_t)pb * P.C + cc * 8));
        }
        pre[2 * r] = va;
        pre[2 * r + 1] = vb;
    }
}

// Tagged table weights of a MIX item for this thread's entries (checked at use).
__device__ __forceinline__ void weights_prefetch(const FusedParams &P, const Item &it,
                                                 unsigned long long *wp) {
    const int kp = P.geom.kp;
    const unsigned long long *an = P.a + (size_t)it.n * P.R * P.k;
#pragma unroll
    for (int r = 0; r < kWPref; ++r) {
        const int q = threadIdx.x + r * kMixThreads;
        const int el = fdiv(q, kp, P.inv_kp), i = q - el * kp;
        if (el < P.R && i < P.k) wp[r] = ld_tagged(an + (size_t)el * P.k + i);
    }
}

// The prefetched tile goes to shared memory, transposed (layout of stage_x_tile).
template <int GS>
__device__ __forceinline__ void mix_stage(const FusedParams &P, const Item &it, const uint4 *pre,
                                          unsigned char *xs) {
    constexpr int TP = 8 * GS, RB = 16 * GS;
    const int p0 = it.t * TP, np = min(TP, P.HW - p0);
    const int CC = P.C >> 3, CCp = (CC + 7) & ~7, per_q = 4 * CCp, units = GS * per_q;
#pragma unroll
    for (int r = 0; r < kPref / 2; ++r) {
        const int u = threadIdx.x + r * kMixThreads;
        int q, j, cc;
        stage_unit_coords(u, per_q, P.inv_perq, q, j, cc);
        if (u < units && cc < CC) store_unit<GS>(xs, q, j, cc, pre[2 * r], pre[2 * r + 1]);
    }
    const uint16_t *xt = P.x + ((size_t)it.n * P.HW + p0) * P.C;
    for (int u = threadIdx.x + (kPref / 2) * kMixThreads; u < units; u += kMixThreads) {
        int q, j, cc;
        stage_unit_coords(u, per_q, P.inv_perq, q, j, cc);
        if (cc >= CC) continue;
        const int pa = q + 2 * GS * j, pb = pa + GS;
        uint4 va = make_uint4(0u, 0u, 0u, 0u), vb = va;
        if (pa < np) va = __ldcs(reinterpret_cast<const uint4 *>(xt + (size_t)pa * P.C + cc * 8));
        if (pb < np) vb = __ldcs(reinterpret_cast<const uint4 *>(xt + (size_t)pb * P.C + cc * 8));
        store_unit<GS>(xs, q, j, cc, va, vb);
    }
    for (int q = threadIdx.x; q < RB / 4; q += kMixThreads)
        reinterpret_cast<uint32_t *>(xs + (size_t)P.C * RB)[q] = 0u;
}

template <int GS>
__device__ void mix_item(const FusedParams &P, const Item &it, unsigned char *sm,
                         const int32_t *s_resid, uint32_t ready, uint32_t item,
                         unsigned long long *wp) {
    constexpr int TP = 8 * GS, RB = 16 * GS, G = kMixThreads / GS;
    constexpr int FM = (GS < 8 ? GS : 8) - 1;
    const MixGeom &g = P.geom;
    const unsigned char *xs = sm;
    uint16_t *ys = reinterpret_cast<uint16_t *>(sm + g.off_ys);
    float *rp = reinterpret_cast<float *>(sm + g.off_rp);
    float *pp = reinterpret_cast<float *>(sm + g.off_pp);
    uint4 *tab = reinterpret_cast<uint4 *>(sm + g.off_tab);
    const int n = it.n;
    const int R = P.R, k = P.k, E = R + 1, Es = P.Es, kp = g.kp;
    const int p0 = it.t * TP, np = min(TP, P.HW - p0);
    const int gid = threadIdx.x / GS, lig = threadIdx.x - gid * GS;
    const int warp = threadIdx.x >> 5, h = (threadIdx.x & 31) / GS;
    const uint32_t lx = (uint32_t)lig << 4;

    // residual expert: each group sums a slice of U for its positions
    {
        float2 r0 = make_float2(0.f, 0.f), r1 = r0, r2 = r0, r3 = r0;
        const int per = (P.nU + G - 1) / G;
        const int u0 = gid * per, u1 = min(P.nU, u0 + per);
        for (int u = u0; u < u1; ++u) {
            const uint32_t c = (uint32_t)s_resid[u];
            const uint4 v = lds128(xs + (((c * RB) | (((c >> 3) & FM) << 4)) ^ lx));
            r0.x += bf16lo(v.x); r0.y += bf16hi(v.x);
            r1.x += bf16lo(v.y); r1.y += bf16hi(v.y);
            r2.x += bf16lo(v.z); r2.y += bf16hi(v.z);
            r3.x += bf16lo(v.w); r3.y += bf16hi(v.w);
        }
        float *rg = rp + gid * TP + lig;
        rg[0 * GS] = r0.x; rg[1 * GS] = r0.y; rg[2 * GS] = r1.x; rg[3 * GS] = r1.y;
        rg[4 * GS] = r2.x; rg[5 * GS] = r2.y; rg[6 * GS] = r3.x; rg[7 * GS] = r3.y;
    }

    const unsigned long long *an = P.a + (size_t)n * R * k;
    for (int e0 = 0; e0 < R; e0 += g.EB) {
        const int eb = min(g.EB, R - e0);
        bool ok = true;
        if (e0 > 0) bar_sync(kBarMix, kMixThreads);  // the previous chunk's table is consumed
        if (P.wpref) {
            // one chunk of at most kWPref * kMixThreads entries, offsets fixed,
            // weights prefetched with the x tile
#pragma unroll
            for (int r = 0; r < kWPref; ++r) {
                const int q = threadIdx.x + r * kMixThreads;
                if (q < eb * kp) {
                    const int el = fdiv(q, kp, P.inv_kp), i = q - el * kp;
                    float w = 0.f;
                    if (i < k && ok) {
                        if (!tag_ok(wp[r], ready))
                            ok = wait_tagged(an + (size_t)el * k + i, ready, wp[r], P.ctrl, item);
                        w = tag_val(wp[r]);
                    }
                    reinterpret_cast<uint32_t *>(tab + tslot(el, kp, i >> 1))[2 + (i & 1)] =
                        __float_as_uint(w);
                }
            }
        } else {
            for (int q = threadIdx.x; q < eb * kp; q += kMixThreads) {
                const int el = fdiv(q, kp, P.inv_kp), i = q - el * kp, e = e0 + el;
                uint32_t *tw = reinterpret_cast<uint32_t *>(tab + tslot(el, kp, i >> 1));
                float w = 0.f;
                if (i < k && ok) {
                    unsigned long long v = ld_tagged(an + (size_t)e * k + i);
                    if (!tag_ok(v, ready)) ok = wait_tagged(an + (size_t)e * k + i, ready, v, P.ctrl, item);
                    w = tag_val(v);
                }
                if (!P.static_off) {
                    uint32_t off = (uint32_t)P.C * RB;
                    if (i < k) {
                        const uint32_t c = (uint32_t)__ldg(P.pidx + (size_t)e * k + i);
                        off = (c * RB) | (((c >> 3) & FM) << 4);
                    }
                    tw[i & 1] = off;
                }
                tw[2 + (i & 1)] = __float_as_uint(w);
            }
        }
        if (!bar_and(kBarMix, kMixThreads, ok)) return;
        if (g.S == 1) {
            // expert pairs (2P, 2P+1) per lane group; the groups of a warp take
            // pairs GS apart so that their bf16x2 stores hit disjoint banks
            const int NP = (eb + 1) >> 1;
            const int nbase = ((NP + 31) >> 5) * GS;
            for (int bi = warp; bi < nbase; bi += kMixWarps) {
                const int pr = ((bi / GS) << 5) + (bi % GS) + GS * h;
                if (pr >= NP) continue;
                const int ea = 2 * pr, ebb = ea + 1;
                float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
                float2 b0 = a0, b1 = a0, b2 = a0, b3 = a0;
                if (ebb < eb)
                    mix_entries2(xs, tab + tslot(ea, kp, 0), tab + tslot(ebb, kp, 0), kp >> 1, lx,
                                 a0, a1, a2, a3, b0, b1, b2, b3);
                else
                    mix_entries(xs, tab + tslot(ea, kp, 0), kp >> 1, lx, a0, a1, a2, a3);
                uint32_t *yw = reinterpret_cast<uint32_t *>(ys + lig * Es + e0 + ea);
                const int st = (GS * Es) >> 1;  // words between the lane's positions
                yw[0 * st] = pack_bf16x2(a0.x, b0.x);
                yw[1 * st] = pack_bf16x2(a0.y, b0.y);
                yw[2 * st] = pack_bf16x2(a1.x, b1.x);
                yw[3 * st] = pack_bf16x2(a1.y, b1.y);
                yw[4 * st] = pack_bf16x2(a2.x, b2.x);
                yw[5 * st] = pack_bf16x2(a2.y, b2.y);
                yw[6 * st] = pack_bf16x2(a3.x, b3.x);
                yw[7 * st] = pack_bf16x2(a3.y, b3.y);
            }
        } else {
            const int S = g.S, kq = g.kq;
            const int jobs = eb * S;
            for (int jb = gid; jb < jobs; jb += G) {
                const int el = jb / S, part = jb - el * S;
                const int i0 = part * kq, i1 = min(kp, i0 + kq);
                float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2 = a0, a3 = a0;
                mix_entries(xs, tab + tslot(el, kp, i0 >> 1), (i1 - i0) >> 1, lx, a0, a1, a2, a3);
                float *pj = pp + (size_t)jb * TP + lig;
                pj[0 * GS] = a0.x; pj[1 * GS] = a0.y; pj[2 * GS] = a1.x; pj[3 * GS] = a1.y;
                pj[4 * GS] = a2.x; pj[5 * GS] = a2.y; pj[6 * GS] = a3.x; pj[7 * GS] = a3.y;
            }
            bar_sync(kBarMix, kMixThreads);
            for (int q = threadIdx.x; q < eb * TP; q += kMixThreads) {
                const int el = q / TP, px = q - el * TP;
                float s = 0.f;
                for (int part = 0; part < S; ++part) s += pp[(size_t)(el * S + part) * TP + px];
                ys[px * Es + e0 + el] = f32_to_bf16(s);
            }
        }
    }
    bar_sync(kBarMix, kMixThreads);
    for (int px = threadIdx.x; px < TP; px += kMixThreads) {
        float s = 0.f;
        for (int gg = 0; gg < G; ++gg) s += rp[gg * TP + px];
        ys[px * Es + R] = f32_to_bf16(P.nU > 0 ? s / (float)P.nU : 0.f);
    }
    bar_sync(kBarMix, kMixThreads);

    // the [np][E] output block is contiguous in y: 16-byte streaming stores
    const int cnt = np * E;
    uint16_t *dst = P.y + ((size_t)n * P.HW + p0) * E;
    const int head =
        min(cnt, (int)(((16u - ((uint32_t)reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u) >> 1));
    for (int o = threadIdx.x; o < head; o += kMixThreads) {
        const int p = fdiv(o, E, P.inv_E);
        __stcs(dst + o, ys[p * Es + (o - p * E)]);
    }
    const int nv = (cnt - head) >> 3;
    for (int v = threadIdx.x; v < nv; v += kMixThreads) {
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
    for (int o = head + nv * 8 + threadIdx.x; o < cnt; o += kMixThreads) {
        const int p = fdiv(o, E, P.inv_E);
        __stcs(dst + o, ys[p * Es + (o - p * E)]);
    }
}

template <int GS>
__device__ void mix_loop(const FusedParams &P, unsigned char *sm, const int32_t *s_resid,
                         const float *W1s, const float *b1s, const float *w2s,
                         const int32_t *pidx_s, const float *plog_s, uint32_t ready,
                         uint32_t drop) {
    uint4 pre[kPref];
    unsigned long long wp[kWPref];
#pragma unroll
    for (int s = 0; s < kPref; ++s) pre[s] = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int r = 0; r < kWPref; ++r) wp[r] = 0ull;
    uint32_t cur = blockIdx.x;
    Item it = mix_decode(P, cur);
    if (it.kind == kMix) {
        mix_prefetch<GS>(P, it, pre);
        if (P.wpref) weights_prefetch(P, it, wp);
    }
    while (cur < P.mix_items) {
        bar_sync(kBarMix, kMixThreads);  // shared memory of the previous item is free
        if (it.kind == kMix) mix_stage<GS>(P, it, pre, sm);
        bar_sync(kBarMix, kMixThreads);
        const uint32_t nxt = cur + gridDim.x;
        const Item in = mix_decode(P, nxt);
        if (in.kind == kMix) mix_prefetch<GS>(P, in, pre);
        if (it.kind == kGate)
            gate_item(P, it.n, it.t, sm, W1s, b1s, w2s, pidx_s, plog_s, ready, cur, cur + 1u != drop);
        else if (it.kind == kMix) mix_item<GS>(P, it, sm, s_resid, ready, cur, wp);
        // the next item's weights arrive while it stages its tile
        if (in.kind == kMix && P.wpref) weights_prefetch(P, in, wp);
        cur = nxt;
        it = in;
    }
}

// ---------------------------------------------------------------- the kernel
template <int GS>
__global__ void __launch_bounds__(kFusedThreads, 1) moce_fused_kernel(const FusedParams P) {
    constexpr int RB = 16 * GS;
    constexpr int FM = (GS < 8 ? GS : 8) - 1;
    extern __shared__ __align__(16) unsigned char sm[];
    const uint32_t epoch = ld_relaxed(P.ctrl + kCtrlEpoch);
    const uint32_t ready = epoch + 1u;
    const uint32_t drop = ld_relaxed(P.ctrl + kCtrlDropItem);
    const MixGeom &g = P.geom;

    // persistent shared data: U list, W1 (rows padded to ks), b1, w2, table offsets
    int32_t *s_resid = reinterpret_cast<int32_t *>(sm + P.off_static);
    float *W1s = reinterpret_cast<float *>(s_resid + ((P.C + 3) & ~3));
    float *b1s = W1s + (size_t)P.k * P.ks;
    float *w2s = b1s + P.k;
    int32_t *pidx_s = reinterpret_cast<int32_t *>(w2s + P.k);
    float *plog_s = reinterpret_cast<float *>(pidx_s + P.R * P.k);
    for (int i = threadIdx.x; i < P.nU; i += kFusedThreads) s_resid[i] = __ldg(P.resid + i);
    if (P.gate_tabs) {
        for (int q = threadIdx.x; q < P.R * P.k; q += kFusedThreads) {
            pidx_s[q] = __ldg(P.pidx + q);
            plog_s[q] = __ldg(P.plog + q);
        }
    }
    for (int q = threadIdx.x; q < P.k * P.k; q += kFusedThreads) {
        const int j = q / P.k, i = q - j * P.k;
        W1s[j * P.ks + i] = __ldg(P.W1 + q);
    }
    for (int j = threadIdx.x; j < P.k; j += kFusedThreads) {
        b1s[j] = __ldg(P.b1 + j);
        w2s[j] = __ldg(P.w2 + j);
    }
    if (P.static_off) {
        uint4 *tab = reinterpret_cast<uint4 *>(sm + g.off_tab);
        for (int q = threadIdx.x; q < P.R * g.kp; q += kFusedThreads) {
            const int el = q / g.kp, i = q - el * g.kp;
            uint32_t off = (uint32_t)P.C * RB;
            if (i < P.k) {
                const uint32_t c = (uint32_t)__ldg(P.pidx + (size_t)el * P.k + i);
                off = (c * RB) | (((c >> 3) & FM) << 4);
            }
            reinterpret_cast<uint32_t *>(tab + tslot(el, g.kp, i >> 1))[i & 1] = off;
        }
    }
    __syncthreads();

    if (threadIdx.x < kMixThreads)
        mix_loop<GS>(P, sm, s_resid, W1s, b1s, w2s, pidx_s, plog_s, ready, drop);
    else pool_loop(P, sm, ready, drop);

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
struct FusedPlan {
    MixGeom g;
    int Es = 0, ks = 0;
    bool static_off = false, wpref = false, gate_tabs = false;
    size_t off_us = 0, off_red = 0, off_static = 0, smem = 0;
};

// Shared memory: [xs | ys | rp | pp | tab] of the mixing geometry, the pool
// group's reduction buffer, then the persistent region (U list, W1, b1, w2).
// The gate scratch (z and per-warp gate inputs) aliases the start; it may not
// reach the persistent data (the table when its offsets are written once).
bool fused_plan(int C, int R, int k, FusedPlan *plan) {
    if (C % 8 != 0 || k > kGateMaxK) return false;
    const int ks = (k % 2 == 0) ? k + 1 : k;
    // the gate's support channels and logits stay in shared memory when small
    const bool gate_tabs = (size_t)R * k * 8 <= 16 * 1024;
    const size_t stat = align_up((size_t)((C + 3) & ~3) * 4, 16) +
                        align_up((size_t)(k * ks + 2 * k) * 4, 16) +
                        (gate_tabs ? align_up((size_t)R * k * 8, 16) : 0);
    const size_t red = (size_t)kPoolThreads * 8 * 4;
    const size_t off_us = align_up((size_t)C * 4, 16);
    const size_t gate_scratch = off_us + (size_t)kMixWarps * k * 4;
    const size_t budget = 224 * 1024;
    if (budget <= stat + red) return false;
    MixGeom g;
    // R + 1 routed columns so that the staged output rows get an even stride
    if (!mix_geometry(C, R + 1, k, budget - stat - red, &g)) return false;
    if (g.EB > R) g.EB = R;
    if (g.EB % 2 && g.EB < R) g.EB -= 1;  // chunk starts stay even (bf16x2 stores)
    if (g.EB < 1) return false;
    FusedPlan p;
    p.g = g;
    p.Es = (R + 1) + ((R + 1) & 1);
    p.ks = ks;
    p.off_us = off_us;
    p.gate_tabs = gate_tabs;
    p.static_off = g.EB >= R && gate_scratch <= g.off_tab;
    p.wpref = p.static_off && R * g.kp <= kWPref * kMixThreads;
    const size_t tab_end = g.smem + 64 * (size_t)((g.EB + 63) / 64);  // tslot block shifts
    const size_t base = tab_end > gate_scratch ? tab_end : gate_scratch;
    p.off_red = align_up(base, 16);
    p.off_static = align_up(p.off_red + red, 16);
    p.smem = p.off_static + stat;
    if (p.smem > 227 * 1024) return false;
    *plan = p;
    return true;
}

template <int GS>
cudaError_t launch_fused_gs(FusedParams &P, const FusedPlan &plan, cudaStream_t s) {
    auto kern = moce_fused_kernel<GS>;
    cudaError_t err =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan.smem);
    if (err != cudaSuccess) return err;
    int dev = 0, sms = 0, per_sm = 0;
    if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
    if ((err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return err;
    if ((err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kFusedThreads,
                                                             plan.smem)) != cudaSuccess)
        return err;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const int grid = sms * per_sm;
    // GATE(n) comes about one and a half rounds of the grid before MIX(n)
    const int per_stage = P.GB + P.MT;
    const int lag = (3 * grid / 2 + per_stage - 1) / per_stage + 1;
    P.lag = lag < P.N ? lag : P.N;
    P.pool_items = (uint32_t)((unsigned long long)P.N * P.PT);
    const unsigned long long mix_total = (unsigned long long)P.N * per_stage;
    if (mix_total >= 0xffff0000ull || (unsigned long long)P.N * P.PT >= 0xffff0000ull)
        return cudaErrorInvalidValue;
    P.mix_items = (uint32_t)mix_total;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)kern, dim3(grid), dim3(kFusedThreads), args,
                                       plan.smem, s);
}

}  // namespace

bool fused_supported(int N, int HW, int C, int R, int k) {
    (void)N;
    (void)HW;
    FusedPlan plan;
    return fused_plan(C, R, k, &plan);
}

cudaError_t launch_fused(const uint16_t *x, int N, int HW, int C, int R, int k,
                         const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                         const float *W1, const float *b1, const float *w2, const float *b2,
                         float tmin, float tmax, uint16_t *y, const WsLayout &L, unsigned char *ws,
                         cudaStream_t s) {
    FusedPlan plan;
    if (!fused_plan(C, R, k, &plan)) return cudaErrorNotSupported;
    FusedParams P;
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
    P.partial = reinterpret_cast<unsigned long long *>(ws + L.partial);
    P.z = reinterpret_cast<float *>(ws + L.z);
    P.tau = reinterpret_cast<float *>(ws + L.tau);
    P.a = reinterpret_cast<unsigned long long *>(ws + L.a);
    P.PP = L.pool_px;
    P.PT = L.pool_tiles;
    P.MT = (HW + plan.g.TP - 1) / plan.g.TP;
    P.GB = L.gate_blocks;
    P.geom = plan.g;
    P.Es = plan.Es;
    P.static_off = plan.static_off ? 1 : 0;
    P.wpref = plan.wpref ? 1 : 0;
    P.ks = plan.ks;
    P.off_static = plan.off_static;
    P.off_us = plan.off_us;
    P.off_red = plan.off_red;
    P.gate_tabs = plan.gate_tabs ? 1 : 0;
    P.inv_perq = 1.0f / (float)(4 * (((C >> 3) + 7) & ~7));
    P.inv_E = 1.0f / (float)(R + 1);
    P.inv_kp = 1.0f / (float)plan.g.kp;
    switch (plan.g.GS) {
    case 16: return launch_fused_gs<16>(P, plan, s);
    case 8: return launch_fused_gs<8>(P, plan, s);
    case 4: return launch_fused_gs<4>(P, plan, s);
    default: return launch_fused_gs<2>(P, plan, s);
    }
}

}  // namespace moce
