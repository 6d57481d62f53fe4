// Routed mix and residual expert (Eq. (expert), Eq. (res)) for NHWC bf16
// layers whose example does not fit in shared memory (C_in up to thousands of
// channels, hundreds of experts, k up to hundreds), from the mixing weights
// a[n][e][i] the gate kernel wrote.
//
// One CTA of 512 threads mixes a tile of TP = 8 GS positions of one example:
//   - the tile is staged channel-major: row c holds the TP positions of
//     channel c as bf16, 16-byte chunk q holding positions q + GS m
//     (m = 0..7; word j = m 2j and 2j + 1), stored at chunk q ^ f(c),
//     f(c) = (c >> 3) mod GS, which spreads the staging stores over the
//     banks; row C is zeros;
//   - the experts' support indices and weights stream through a ring of NB
//     shared-memory buffers, EB experts per chunk, each chunk two bulk copies
//     (its rows of the index table and of the example's weights);
//   - a warp mixes EPW experts of a chunk at a time; the S = 32 / GS lane
//     groups of the warp are EPW experts x PPE parts of each expert's support
//     list (part p = entries p kq .. p kq + kq - 1, kq = k / PPE a multiple
//     of 8, read 16 bytes at a time), a group of GS lanes covering the TP
//     positions (8 per lane). A lane reads the 16-byte chunk of each of its
//     supports' rows and adds it with fma.rn.f32x2; the PPE parts are then
//     added by shuffles in a fixed order;
//   - the residual expert is U with the weight 1 / |U|, U staged once;
//   - the y tile [TP][R + 1] is staged in shared memory and leaves by 16-byte
//     stores.
// Every wait is bounded; a wait that gives up sets the workspace error word.
#include "moce_internal.cuh"

namespace moce {
namespace {

constexpr int kWideThreads = 512;
constexpr int kWideWarps = kWideThreads / 32;

__device__ __forceinline__ uint4 lds128w(const unsigned char *p) {
    return *reinterpret_cast<const uint4 *>(p);
}
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
__device__ __forceinline__ uint32_t smem_u32w(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

struct WideGeom {
    int GS = 0, TP = 0, PPE = 1, EPW = 1, YS = 0, tiles = 0;
    int kq = 0;          // entries per part (a multiple of 8)
    int EB = 0, NB = 0;  // experts per table chunk, chunk buffers
    size_t off_ys = 0, off_us = 0, off_bar = 0, off_tab = 0, smem = 0;
};

// Stage positions [0, np) of the tile (xe = its first position) channel-major
// into xs. Unit (q, cc, j): positions q + 2 GS j and q + GS (2 j + 1) of
// channel octet cc become word j of chunk q in the octet's 8 rows. The 32
// units of a warp are 8 octets x 4 words, so its loads are 128-byte runs of a
// position row and its stores spread over 16 banks.
template <int GS>
__device__ __forceinline__ void stage_wide(unsigned char *xs, const uint16_t *__restrict__ xe,
                                           int np, int C) {
    constexpr int RB = 16 * GS;
    constexpr int FM = GS - 1;
    const int CC = C >> 3;
    const int CH = (CC + 7) >> 3;  // octet groups of 8
    const int units = GS * CH * 32;
    // four units per thread per round, all loads before any store, so that
    // eight 16-byte loads per thread are in flight
    constexpr int U4 = 4;
    for (int u0 = threadIdx.x; u0 < units; u0 += U4 * kWideThreads) {
        uint4 va[U4], vb[U4];
        int dst[U4];
#pragma unroll
        for (int r = 0; r < U4; ++r) {
            const int u = u0 + r * kWideThreads;
            const int lo = u & 7, j = (u >> 3) & 3, hi = u >> 5;
            const int q = hi / CH, cc = (hi - q * CH) * 8 + lo;
            const int pa = q + 2 * GS * j, pb = pa + GS;
            const bool live = u < units && cc < CC;
            va[r] = make_uint4(0u, 0u, 0u, 0u);
            vb[r] = va[r];
            if (live && pa < np)
                va[r] = __ldcs(reinterpret_cast<const uint4 *>(xe + (size_t)pa * C + cc * 8));
            if (live && pb < np)
                vb[r] = __ldcs(reinterpret_cast<const uint4 *>(xe + (size_t)pb * C + cc * 8));
            dst[r] = live ? (cc * 8) * RB + (((q ^ (cc & FM)) << 4) | (j << 2)) : -1;
        }
#pragma unroll
        for (int r = 0; r < U4; ++r) {
            if (dst[r] < 0) continue;
            unsigned char *d = xs + dst[r];
            *reinterpret_cast<uint32_t *>(d + 0 * RB) = __byte_perm(va[r].x, vb[r].x, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 1 * RB) = __byte_perm(va[r].x, vb[r].x, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 2 * RB) = __byte_perm(va[r].y, vb[r].y, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 3 * RB) = __byte_perm(va[r].y, vb[r].y, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 4 * RB) = __byte_perm(va[r].z, vb[r].z, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 5 * RB) = __byte_perm(va[r].z, vb[r].z, 0x7632);
            *reinterpret_cast<uint32_t *>(d + 6 * RB) = __byte_perm(va[r].w, vb[r].w, 0x5410);
            *reinterpret_cast<uint32_t *>(d + 7 * RB) = __byte_perm(va[r].w, vb[r].w, 0x7632);
        }
    }
    for (int q = threadIdx.x; q < RB / 4; q += kWideThreads)
        reinterpret_cast<uint32_t *>(xs + (size_t)C * RB)[q] = 0u;
}

__device__ __forceinline__ void wmbar_init(uint32_t a, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}
__device__ __forceinline__ void wmbar_expect_tx(uint32_t a, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void wmbar_arrive(uint32_t a) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(a)
                 : "memory");
}
// Bounded wait for the phase with the given parity of the mbarrier at a;
// false when it gave up (the error word, when there is one, then says so).
__device__ __noinline__ bool wmbar_wait(uint32_t a, uint32_t parity, uint32_t *ctrl) {
    for (uint32_t it = 0; it < (1u << 20); ++it) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(a), "r"(parity), "r"(1000u)
            : "memory");
        if (ok) return true;
        if (ctrl && (it & 15u) == 15u && *(volatile uint32_t *)(ctrl + kCtrlError) != 0u)
            return false;
    }
    if (ctrl) atomicOr(ctrl + kCtrlError, kErrTimeout);
    return false;
}
__device__ __forceinline__ void wbulk_load(uint32_t dst, const void *src, uint32_t bytes,
                                           uint32_t mbar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(dst), "l"(src), "r"(bytes), "r"(mbar)
        : "memory");
}

template <int GS>
__global__ void __launch_bounds__(kWideThreads, 1) mix_wide_kernel(
    const uint16_t *__restrict__ x, int HW, int C, int R, int k,
    const int32_t *__restrict__ pidx, const float *__restrict__ a,
    const int32_t *__restrict__ resid, int nU, uint16_t *__restrict__ y, uint32_t *ctrl,
    WideGeom g, PerExample pe) {
    constexpr int TP = 8 * GS, RB = 16 * GS, FM = GS - 1;
    extern __shared__ __align__(128) unsigned char wsm[];
    unsigned char *xs = wsm;
    uint16_t *ys = reinterpret_cast<uint16_t *>(wsm + g.off_ys);
    uint16_t *us = reinterpret_cast<uint16_t *>(wsm + g.off_us);
    const uint32_t bar = smem_u32w(wsm + g.off_bar);
    const uint32_t tab0 = smem_u32w(wsm + g.off_tab);
    const int n = blockIdx.x / g.tiles, t = blockIdx.x - n * g.tiles;
    const int p0 = t * TP, np = min(TP, HW - p0);
    const int E = R + 1;
    const float *an = a + (size_t)n * R * k;
    pidx += (size_t)n * pe.sup_stride;  // per-example supports (0: shared)
    resid += (size_t)n * pe.resid_stride;
    nU = pe.count(n, nU, C);
    const int nch = (R + g.EB - 1) / g.EB;
    // table chunk j: the support indices, then the weights, of experts
    // j EB .. j EB + EB - 1 (each a contiguous run of rows in global memory)
    const uint32_t half = (uint32_t)g.EB * (uint32_t)k * 4u;
    int issued = 0;  // chunks issued (thread 0)
    auto issue = [&](int j) {
        ++issued;
        const int e0 = j * g.EB, eb = min(g.EB, R - e0);
        const uint32_t bytes = (uint32_t)eb * (uint32_t)k * 4u;
        const uint32_t b = bar + 8u * (uint32_t)(j % g.NB);
        const uint32_t d = tab0 + (uint32_t)(j % g.NB) * 2u * half;
        wmbar_expect_tx(b, 2u * bytes);
        wbulk_load(d, pidx + (size_t)e0 * k, bytes, b);
        wbulk_load(d + half, an + (size_t)e0 * k, bytes, b);
    };
    if (threadIdx.x == 0) {
        for (int q = 0; q < g.NB; ++q) {
            wmbar_init(bar + 8u * q, 1);                    // full: the two copies
            wmbar_init(bar + 8u * (g.NB + q), kWideWarps);  // empty: every warp read it
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        for (int j = 0; j < min(g.NB, nch); ++j) issue(j);
    }
    for (int i = threadIdx.x; i < nU; i += kWideThreads) us[i] = (uint16_t)__ldg(resid + i);
    stage_wide<GS>(xs, x + ((size_t)n * HW + p0) * C, np, C);
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gi = lane / GS, lig = lane - gi * GS;
    const int es = gi / g.PPE, part = gi - es * g.PPE;
    const uint32_t lx = (uint32_t)lig << 4;
    // 8 entries (channel indices c[], weights w[]) added to the lane's 8 positions
    auto mix8 = [&](const int4 c0, const int4 c1, const float4 w0, const float4 w1,
                    float2(&acc)[4]) {
        const uint32_t cu[8] = {(uint32_t)c0.x, (uint32_t)c0.y, (uint32_t)c0.z, (uint32_t)c0.w,
                                (uint32_t)c1.x, (uint32_t)c1.y, (uint32_t)c1.z, (uint32_t)c1.w};
        const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
        uint32_t off[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            off[u] = ((cu[u] * RB) | (((cu[u] >> 3) & FM) << 4)) ^ lx;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const uint4 v = lds128w(xs + off[u]);
            const float2 wu = make_float2(wv[u], wv[u]);
            acc[0] = __ffma2_rn(wu, unpack_bf16x2(v.x), acc[0]);
            acc[1] = __ffma2_rn(wu, unpack_bf16x2(v.y), acc[1]);
            acc[2] = __ffma2_rn(wu, unpack_bf16x2(v.z), acc[2]);
            acc[3] = __ffma2_rn(wu, unpack_bf16x2(v.w), acc[3]);
        }
    };
    // the PPE parts of an expert (lanes GS apart) added in a fixed order, then
    // the part-0 lanes stage the expert's TP outputs
    auto finish = [&](float2(&acc)[4], int e, bool live) {
        for (int o = GS; o < GS * g.PPE; o <<= 1) {
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                acc[m].x += __shfl_xor_sync(0xffffffffu, acc[m].x, o);
                acc[m].y += __shfl_xor_sync(0xffffffffu, acc[m].y, o);
            }
        }
        if (part == 0 && live) {
            // word m of the lane's chunk = positions lig + GS 2m, lig + GS (2m + 1)
            uint16_t *yc = ys + (size_t)lig * g.YS + e;
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                yc[(2 * m) * GS * g.YS] = f32_to_bf16(acc[m].x);
                yc[(2 * m + 1) * GS * g.YS] = f32_to_bf16(acc[m].y);
            }
        }
    };
    bool ok = true;
    for (int j = 0; j < nch; ++j) {
        const int q = j % g.NB;
        ok = __all_sync(0xffffffffu,
                        ok && wmbar_wait(bar + 8u * q, (uint32_t)(j / g.NB) & 1u, ctrl));
        if (!ok) break;  // warp-uniform
        const unsigned char *tb = wsm + g.off_tab + (size_t)q * 2 * half;
        const int32_t *ti = reinterpret_cast<const int32_t *>(tb);
        const float *tw = reinterpret_cast<const float *>(tb + half);
        const int e0 = j * g.EB, eb = min(g.EB, R - e0);
        for (int el0 = warp * g.EPW; el0 < eb; el0 += kWideWarps * g.EPW) {
            const int el = el0 + es;
            const bool live = el < eb;
            float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                             make_float2(0.f, 0.f)};
            if (live) {
                const size_t b0 = (size_t)el * k + (size_t)part * g.kq;
                const int4 *ci = reinterpret_cast<const int4 *>(ti + b0);
                const float4 *wi = reinterpret_cast<const float4 *>(tw + b0);
                for (int m = 0; m < g.kq / 4; m += 2) mix8(ci[m], ci[m + 1], wi[m], wi[m + 1], acc);
            }
            finish(acc, e0 + el, live);
        }
        __syncwarp();
        if (lane == 0) wmbar_arrive(bar + 8u * (g.NB + q));
        if (threadIdx.x == 0 && j + g.NB < nch) {
            // every warp has read buffer q: refill it
            if (wmbar_wait(bar + 8u * (g.NB + q), (uint32_t)(j / g.NB) & 1u, ctrl)) issue(j + g.NB);
        }
    }
    // the residual expert: U with the weight 1 / |U|, by warp 0 (entries
    // part, part + PPE, ...; padded with the zero row)
    if (warp == 0) {
        float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                         make_float2(0.f, 0.f)};
        const bool live = es == 0;
        const float wr = nU > 0 ? 1.f / (float)nU : 0.f;
        for (int i0 = part; live && i0 < nU; i0 += 8 * g.PPE) {
            int cc[8];
            float ww[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = i0 + g.PPE * u;
                cc[u] = i < nU ? (int)us[i] : C;
                ww[u] = i < nU ? wr : 0.f;
            }
            mix8(make_int4(cc[0], cc[1], cc[2], cc[3]), make_int4(cc[4], cc[5], cc[6], cc[7]),
                 make_float4(ww[0], ww[1], ww[2], ww[3]), make_float4(ww[4], ww[5], ww[6], ww[7]),
                 acc);
        }
        finish(acc, R, live);
    }
    // no copy may still be writing shared memory when the CTA exits
    if (threadIdx.x == 0)
        for (int j = max(0, issued - g.NB); j < issued; ++j)
            wmbar_wait(bar + 8u * (j % g.NB), (uint32_t)(j / g.NB) & 1u, ctrl);
    __syncthreads();
    // the y tile: rows of E bf16 at row stride YS
    uint16_t *yt = y + ((size_t)n * HW + p0) * E;
    if ((E & 7) == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0) {
        const int vr = E >> 3;
        for (int q = threadIdx.x; q < np * vr; q += kWideThreads) {
            const int p = q / vr, v = q - p * vr;
            __stcs(reinterpret_cast<uint4 *>(yt + (size_t)p * E) + v,
                   *reinterpret_cast<const uint4 *>(ys + (size_t)p * g.YS + 8 * v));
        }
    } else {
        for (int q = threadIdx.x; q < np * E; q += kWideThreads) {
            const int p = q / E, e = q - p * E;
            yt[q] = ys[(size_t)p * g.YS + e];
        }
    }
}

bool wide_geometry(int HW, int C, int R, int k, int nU, WideGeom *out) {
    if (k % 8 != 0) return false;  // whole 8-entry blocks; 16-byte aligned table rows
    const int E = R + 1;
    const int YS = ((E + 7) & ~7) + 8;  // padded rows: consecutive positions 16 bytes apart mod 128
    const size_t budget = 227 * 1024;
    for (int GS = 8; GS >= 2; GS >>= 1) {
        // a tile much larger than the example wastes work: prefer the next size down
        if (GS > 2 && HW <= 4 * GS) continue;
        WideGeom g;
        g.GS = GS;
        g.TP = 8 * GS;
        g.YS = YS;
        // parts per expert: the most (at most S) whose entry blocks are whole
        // multiples of 8
        const int S = 32 / GS;
        int ppe = 0;
        for (int p = 1; p <= S; p *= 2)
            if (k % (8 * p) == 0) ppe = p;
        if (ppe == 0) return false;
        g.PPE = ppe;
        g.EPW = S / ppe;
        g.kq = k / ppe;
        g.off_ys = align_up((size_t)(C + 1) * 16 * GS, 16);
        g.off_us = align_up(g.off_ys + (size_t)g.TP * YS * 2, 16);
        g.off_bar = align_up(g.off_us + (size_t)(nU > 0 ? nU : 1) * 2, 16);
        g.off_tab = align_up(g.off_bar + 64, 128);
        // chunks of 16 EPW experts (every warp busy), halved until they fit,
        // down to 4 EPW (a quarter of the warps busy)
        bool fit = false;
        for (int eb = 16 * g.EPW; eb >= 4 * g.EPW && !fit; eb /= 2) {
            const int ebc = eb < R ? eb : R;
            for (int nb = 3; nb >= 2 && !fit; --nb) {
                const size_t sm = g.off_tab + (size_t)nb * 2 * ebc * k * 4;
                if (sm <= budget) {
                    g.EB = ebc;
                    g.NB = nb;
                    g.smem = sm;
                    fit = true;
                }
            }
        }
        if (!fit) continue;
        g.tiles = (HW + g.TP - 1) / g.TP;
        *out = g;
        return true;
    }
    return false;
}

template <int GS>
cudaError_t launch_wide_gs(const uint16_t *x, int N, int HW, int C, int R, int k,
                           const int32_t *pidx, const float *a, const int32_t *resid, int nU,
                           uint16_t *y, uint32_t *ctrl, const WideGeom &g, const PerExample &pe,
                           cudaStream_t s) {
    cudaError_t err = cudaFuncSetAttribute(mix_wide_kernel<GS>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem);
    if (err != cudaSuccess) return err;
    mix_wide_kernel<GS><<<(unsigned)((size_t)N * g.tiles), kWideThreads, g.smem, s>>>(
        x, HW, C, R, k, pidx, a, resid, nU, y, ctrl, g, pe);
    return cudaGetLastError();
}

}  // namespace

bool mix_wide_supported(int HW, int C, int R, int k, int nU) {
    WideGeom g;
    return C % 8 == 0 && wide_geometry(HW, C, R, k, nU, &g);
}

cudaError_t launch_mix_wide(const uint16_t *x, int N, int HW, int C, int R, int k,
                            const int32_t *pidx, const float *a, const int32_t *resid, int nU,
                            uint16_t *y, uint32_t *ctrl, cudaStream_t s, const PerExample &pe) {
    WideGeom g;
    // per-example U: room for the largest |U(X)| = C
    if (C % 8 != 0 || !wide_geometry(HW, C, R, k, pe.nUa ? C : nU, &g)) return cudaErrorNotSupported;
    // the bulk copies read 16-byte aligned rows of the tables
    if ((reinterpret_cast<uintptr_t>(pidx) & 15u) || (reinterpret_cast<uintptr_t>(a) & 15u))
        return cudaErrorNotSupported;
    if ((size_t)N * g.tiles > 0x7fffffffu) return cudaErrorNotSupported;
    switch (g.GS) {
    case 8: return launch_wide_gs<8>(x, N, HW, C, R, k, pidx, a, resid, nU, y, ctrl, g, pe, s);
    case 4: return launch_wide_gs<4>(x, N, HW, C, R, k, pidx, a, resid, nU, y, ctrl, g, pe, s);
    default: return launch_wide_gs<2>(x, N, HW, C, R, k, pidx, a, resid, nU, y, ctrl, g, pe, s);
    }
}

}  // namespace moce
