// One tile of the NHWC bf16 routed mix + residual (Eq. (expert), Eq. (res)).
// Used by the standalone tiled mixing kernel (the shapes moce_mix_wide.cu
// does not take). See moce_mix.cu for the design notes.
#pragma once

#include "moce_internal.cuh"

namespace moce {

constexpr size_t kMixSmemBudget = 220 * 1024;

__device__ __forceinline__ uint4 lds128(const unsigned char *p) {
    return *reinterpret_cast<const uint4 *>(p);
}

__device__ __forceinline__ float2 unpack2(uint32_t w) { return make_float2(bf16lo(w), bf16hi(w)); }

// Stage positions [0, np) of the tile (xe points at its first position) into
// xs: C + 1 rows of RB = 2*TP bytes, row c = channel c, row C = zeros.
// Row c's 16-byte chunk q holds positions q + GS*(2j) (low half) and
// q + GS*(2j+1) (high half) in word j, stored at chunk position q ^ f(c)
// with f(c) = (c >> 3) & FM.
template <int GS>
__device__ __forceinline__ void stage_x_tile(unsigned char *xs, const uint16_t *__restrict__ xe,
                                             int np, int C) {
    constexpr int RB = 16 * GS;
    constexpr int FM = (GS < 8 ? GS : 8) - 1;
    const int CC = C >> 3;
    const int CCp = (CC + 7) & ~7;
    const int per_q = 4 * CCp;
    const int units = GS * per_q;
    for (int u = threadIdx.x; u < units; u += kThreads) {
        const int q = u / per_q;
        const int rem = u - q * per_q;
        const int cc = ((rem >> 5) << 3) | (rem & 7);
        const int j = (rem >> 3) & 3;
        if (cc >= CC) continue;
        const int pa = q + 2 * GS * j, pb = pa + GS;
        uint4 va = make_uint4(0u, 0u, 0u, 0u), vb = va;
        if (pa < np) va = __ldcs(reinterpret_cast<const uint4 *>(xe + (size_t)pa * C + cc * 8));
        if (pb < np) vb = __ldcs(reinterpret_cast<const uint4 *>(xe + (size_t)pb * C + cc * 8));
        unsigned char *d = xs + (size_t)(cc * 8) * RB + (((q ^ (cc & FM)) << 4) | (j << 2));
        *reinterpret_cast<uint32_t *>(d + 0 * RB) = __byte_perm(va.x, vb.x, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 1 * RB) = __byte_perm(va.x, vb.x, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 2 * RB) = __byte_perm(va.y, vb.y, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 3 * RB) = __byte_perm(va.y, vb.y, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 4 * RB) = __byte_perm(va.z, vb.z, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 5 * RB) = __byte_perm(va.z, vb.z, 0x7632);
        *reinterpret_cast<uint32_t *>(d + 6 * RB) = __byte_perm(va.w, vb.w, 0x5410);
        *reinterpret_cast<uint32_t *>(d + 7 * RB) = __byte_perm(va.w, vb.w, 0x7632);
    }
    for (int q = threadIdx.x; q < RB / 4; q += kThreads)
        reinterpret_cast<uint32_t *>(xs + (size_t)C * RB)[q] = 0u;
}

// Copy count bf16 values from shared src (16-byte aligned) to global dst with
// streaming stores, 16 bytes at a time when dst allows it.
__device__ __forceinline__ void copy_out_bf16(const uint16_t *src, uint16_t *__restrict__ dst,
                                              int count) {
    const uintptr_t da = reinterpret_cast<uintptr_t>(dst);
    int done = 0;
    if ((da & 15u) == 0) {
        const int nv = count >> 3;
        for (int v = threadIdx.x; v < nv; v += kThreads)
            __stcs(reinterpret_cast<uint4 *>(dst) + v, reinterpret_cast<const uint4 *>(src)[v]);
        done = nv << 3;
    } else if ((da & 3u) == 0) {
        const int nv = count >> 1;
        for (int v = threadIdx.x; v < nv; v += kThreads)
            __stcs(reinterpret_cast<unsigned int *>(dst) + v,
                   reinterpret_cast<const unsigned int *>(src)[v]);
        done = nv << 1;
    }
    for (int q = done + threadIdx.x; q < count; q += kThreads) __stcs(dst + q, src[q]);
}

// Mix tile t of example n. a_n = weights of example n, [R][k].
template <int GS>
__device__ __forceinline__ void mix_nhwc_bf16_tile(unsigned char *smem, const MixGeom &geom,
                                                   const uint16_t *__restrict__ x, int HW, int C,
                                                   int R, int k, const int32_t *__restrict__ pidx,
                                                   const float *__restrict__ a_n,
                                                   const int32_t *__restrict__ resid, int nU,
                                                   uint16_t *__restrict__ y, int n, int t) {
    constexpr int TP = 8 * GS;
    constexpr int RB = 16 * GS;
    constexpr int G = kThreads / GS;
    constexpr int FM = (GS < 8 ? GS : 8) - 1;
    unsigned char *xs = smem;
    uint16_t *ys = reinterpret_cast<uint16_t *>(smem + geom.off_ys);
    float *rp = reinterpret_cast<float *>(smem + geom.off_rp);
    float *pp = reinterpret_cast<float *>(smem + geom.off_pp);
    uint4 *tab = reinterpret_cast<uint4 *>(smem + geom.off_tab);
    const int E = R + 1;
    const int p0 = t * TP;
    const int np = min(TP, HW - p0);
    const int gid = threadIdx.x / GS, lig = threadIdx.x - gid * GS;
    const uint32_t lx = (uint32_t)lig << 4;

    __syncthreads();  // shared memory of a previous tile is no longer in use
    stage_x_tile<GS>(xs, x + ((size_t)n * HW + p0) * C, np, C);
    __syncthreads();

    // residual expert: every group sums a slice of U for its 8 positions per lane
    {
        float2 r0 = make_float2(0.f, 0.f), r1 = r0, r2 = r0, r3 = r0;
        const int per = (nU + G - 1) / G;
        const int u0 = gid * per, u1 = min(nU, u0 + per);
        for (int u = u0; u < u1; ++u) {
            const uint32_t c = (uint32_t)__ldg(resid + u);
            const uint32_t off = (c * RB) | (((c >> 3) & FM) << 4);
            const uint4 v = lds128(xs + (off ^ lx));
            r0.x += bf16lo(v.x); r0.y += bf16hi(v.x);
            r1.x += bf16lo(v.y); r1.y += bf16hi(v.y);
            r2.x += bf16lo(v.z); r2.y += bf16hi(v.z);
            r3.x += bf16lo(v.w); r3.y += bf16hi(v.w);
        }
        float *rg = rp + gid * TP + lig;
        rg[0 * GS] = r0.x; rg[1 * GS] = r0.y; rg[2 * GS] = r1.x; rg[3 * GS] = r1.y;
        rg[4 * GS] = r2.x; rg[5 * GS] = r2.y; rg[6 * GS] = r3.x; rg[7 * GS] = r3.y;
    }

    const int kp = geom.kp, kq = geom.kq, S = geom.S;
    for (int e0 = 0; e0 < R; e0 += geom.EB) {
        const int eb = min(geom.EB, R - e0);
        __syncthreads();  // previous chunk's table and part buffer consumed
        for (int q = threadIdx.x; q < eb * kp; q += kThreads) {
            const int el = q / kp, i = q - el * kp;
            uint32_t off = (uint32_t)C * RB;  // the zero row for the padding entry
            float w = 0.f;
            if (i < k) {
                const uint32_t c = (uint32_t)__ldg(pidx + (size_t)(e0 + el) * k + i);
                off = (c * RB) | (((c >> 3) & FM) << 4);
                w = a_n[(size_t)(e0 + el) * k + i];
            }
            uint32_t *tw = reinterpret_cast<uint32_t *>(tab + (q >> 1));
            tw[q & 1] = off;
            tw[2 + (q & 1)] = __float_as_uint(w);
        }
        __syncthreads();
        const int jobs = eb * S;
        for (int jb = gid; jb < jobs; jb += G) {
            const int el = jb / S, part = jb - el * S;
            const int i0 = part * kq, i1 = min(kp, i0 + kq);
            float2 acc0 = make_float2(0.f, 0.f), acc1 = acc0, acc2 = acc0, acc3 = acc0;
            const uint4 *te = tab + ((el * kp + i0) >> 1);
            const int npairs = (i1 - i0) >> 1;
#pragma unroll 4
            for (int i2 = 0; i2 < npairs; ++i2) {
                const uint4 en = te[i2];
                const uint4 v0 = lds128(xs + (en.x ^ lx));
                const uint4 v1 = lds128(xs + (en.y ^ lx));
                const float wa = __uint_as_float(en.z), wb = __uint_as_float(en.w);
                const float2 w0 = make_float2(wa, wa), w1 = make_float2(wb, wb);
                acc0 = __ffma2_rn(w0, unpack2(v0.x), acc0);
                acc1 = __ffma2_rn(w0, unpack2(v0.y), acc1);
                acc2 = __ffma2_rn(w0, unpack2(v0.z), acc2);
                acc3 = __ffma2_rn(w0, unpack2(v0.w), acc3);
                acc0 = __ffma2_rn(w1, unpack2(v1.x), acc0);
                acc1 = __ffma2_rn(w1, unpack2(v1.y), acc1);
                acc2 = __ffma2_rn(w1, unpack2(v1.z), acc2);
                acc3 = __ffma2_rn(w1, unpack2(v1.w), acc3);
            }
            if (S == 1) {
                uint16_t *yc = ys + lig * E + e0 + el;
                yc[(0 * GS) * E] = f32_to_bf16(acc0.x);
                yc[(1 * GS) * E] = f32_to_bf16(acc0.y);
                yc[(2 * GS) * E] = f32_to_bf16(acc1.x);
                yc[(3 * GS) * E] = f32_to_bf16(acc1.y);
                yc[(4 * GS) * E] = f32_to_bf16(acc2.x);
                yc[(5 * GS) * E] = f32_to_bf16(acc2.y);
                yc[(6 * GS) * E] = f32_to_bf16(acc3.x);
                yc[(7 * GS) * E] = f32_to_bf16(acc3.y);
            } else {
                float *pj = pp + (size_t)jb * TP + lig;
                pj[0 * GS] = acc0.x; pj[1 * GS] = acc0.y; pj[2 * GS] = acc1.x; pj[3 * GS] = acc1.y;
                pj[4 * GS] = acc2.x; pj[5 * GS] = acc2.y; pj[6 * GS] = acc3.x; pj[7 * GS] = acc3.y;
            }
        }
        if (S > 1) {
            __syncthreads();
            for (int q = threadIdx.x; q < eb * TP; q += kThreads) {
                const int el = q / TP, px = q - el * TP;
                float s = 0.f;
                for (int part = 0; part < S; ++part) s += pp[(size_t)(el * S + part) * TP + px];
                ys[px * E + e0 + el] = f32_to_bf16(s);
            }
        }
    }
    __syncthreads();
    for (int px = threadIdx.x; px < TP; px += kThreads) {
        float s = 0.f;
        for (int g = 0; g < G; ++g) s += rp[g * TP + px];
        ys[px * E + R] = f32_to_bf16(nU > 0 ? s / (float)nU : 0.f);
    }
    __syncthreads();
    copy_out_bf16(ys, y + ((size_t)n * HW + p0) * E, np * E);
}

}  // namespace moce
