// Routed mixing, Eq. (expert), and residual expert, Eq. (res):
//   y[n,p,e] = sum_i a[n,e,i] x[n,p,S_e[i]]      (e < R)
//   y[n,p,R] = mean_{c in U} x[n,p,c], 0 if U is empty.
// The weights a[n,e,i] come from the gate stage. fp32 accumulation, output
// rounded to the input dtype (bf16: round to nearest even).
//
// NHWC bf16 with C >= 512, C % 8 == 0, k % 8 == 0 and aligned tables goes to
// mix_wide_kernel (moce_mix_wide.cu); here:
//  * mix_nchw_kernel: one thread per position, channel planes are contiguous
//    so a warp's gathered loads are coalesced; any dtype.
//  * mix_nhwc_generic_kernel: one thread per output element, for NHWC inputs
//    the tiled kernels do not take (fp32, C % 8 != 0, unaligned x).
//  * mix_nhwc_bf16_tile (device function of the tiled kernel, for the other
//    NHWC bf16 shapes): a tile of TP = 8*GS positions of one example is
//    staged in shared memory transposed to channel-major rows (pixel pairs
//    packed in 32-bit words, rows XOR-swizzled in 16-byte chunks so both the
//    staging stores and the gathers are bank-conflict free); each group of GS
//    lanes owns the tile's positions (8 per lane) and mixes whole experts (or
//    1/S of one) from a per-chunk table of (row offset, weight) pairs, so a
//    gathered channel is one 16-byte shared load feeding 8 fp32 FMAs (four
//    packed f32x2 FMAs). Outputs are staged as a [TP][R+1] bf16 tile and
//    written with coalesced streaming stores.
#include "moce_mix_tile.cuh"

namespace moce {
namespace {

template <typename T>
__global__ void __launch_bounds__(kThreads) mix_nchw_kernel(const T *__restrict__ x, int HW, int C,
                                                            int R, int k,
                                                            const int32_t *__restrict__ pidx,
                                                            const float *__restrict__ a,
                                                            const int32_t *__restrict__ resid,
                                                            int nU, int EPB, T *__restrict__ y,
                                                            PerExample pe) {
    const int p = blockIdx.x * kThreads + threadIdx.x;
    const int n = blockIdx.z;
    pidx += (size_t)n * pe.sup_stride;
    resid += (size_t)n * pe.resid_stride;
    nU = pe.count(n, nU, C);
    const int e0 = blockIdx.y * EPB, e1 = min(R + 1, e0 + EPB);
    if (p >= HW) return;
    const T *xn = x + (size_t)n * C * HW + p;
    T *yn = y + (size_t)n * (R + 1) * HW + p;
    for (int e = e0; e < e1; ++e) {
        float acc = 0.f;
        if (e < R) {
            const int32_t *ie = pidx + (size_t)e * k;
            const float *ae = a + ((size_t)n * R + e) * k;
            for (int i = 0; i < k; ++i)
                acc = fmaf(__ldg(ae + i), load_elem<T>(xn + (size_t)__ldg(ie + i) * HW), acc);
        } else if (nU > 0) {
            for (int j = 0; j < nU; ++j) acc += load_elem<T>(xn + (size_t)__ldg(resid + j) * HW);
            acc = acc / (float)nU;
        }
        yn[(size_t)e * HW] = store_cvt<T>(acc);
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) mix_nhwc_generic_kernel(
    const T *__restrict__ x, int N, int HW, int C, int R, int k, const int32_t *__restrict__ pidx,
    const float *__restrict__ a, const int32_t *__restrict__ resid, int nU, T *__restrict__ y,
    PerExample pe) {
    const size_t total = (size_t)N * HW * (R + 1);
    for (size_t q = (size_t)blockIdx.x * kThreads + threadIdx.x; q < total;
         q += (size_t)gridDim.x * kThreads) {
        const size_t np = q / (R + 1);
        const int e = (int)(q - np * (R + 1));
        const size_t n = np / HW;
        const T *xp = x + np * C;
        float acc = 0.f;
        if (e < R) {
            const int32_t *ie = pidx + n * pe.sup_stride + (size_t)e * k;
            const float *ae = a + (n * R + e) * k;
            for (int i = 0; i < k; ++i) acc = fmaf(__ldg(ae + i), load_elem<T>(xp + __ldg(ie + i)), acc);
        } else {
            const int nUn = pe.count((int)n, nU, C);
            const int32_t *rn = resid + n * pe.resid_stride;
            if (nUn > 0) {
                for (int j = 0; j < nUn; ++j) acc += load_elem<T>(xp + __ldg(rn + j));
                acc = acc / (float)nUn;
            }
        }
        y[q] = store_cvt<T>(acc);
    }
}

template <int GS>
__global__ void __launch_bounds__(kThreads) mix_nhwc_bf16_tiled_kernel(
    const uint16_t *__restrict__ x, int HW, int C, int R, int k, const int32_t *__restrict__ pidx,
    const float *__restrict__ a, const int32_t *__restrict__ resid, int nU,
    uint16_t *__restrict__ y, int tiles, MixGeom geom, PerExample pe) {
    extern __shared__ __align__(16) unsigned char msm[];
    const int n = blockIdx.x / tiles, t = blockIdx.x - n * tiles;
    mix_nhwc_bf16_tile<GS>(msm, geom, x, HW, C, R, k, pidx + (size_t)n * pe.sup_stride,
                           a + (size_t)n * R * k, resid + (size_t)n * pe.resid_stride,
                           pe.count(n, nU, C), y, n, t);
}

template <int GS>
cudaError_t launch_tiled(const uint16_t *x, int N, int HW, int C, int R, int k,
                         const int32_t *pidx, const float *a, const int32_t *resid, int nU,
                         uint16_t *y, const MixGeom &g, const PerExample &pe, cudaStream_t s) {
    cudaError_t err = cudaFuncSetAttribute(mix_nhwc_bf16_tiled_kernel<GS>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem);
    if (err != cudaSuccess) return err;
    const int tiles = (HW + g.TP - 1) / g.TP;
    mix_nhwc_bf16_tiled_kernel<GS><<<(unsigned)((size_t)N * tiles), kThreads, g.smem, s>>>(
        x, HW, C, R, k, pidx, a, resid, nU, y, tiles, g, pe);
    return cudaGetLastError();
}

}  // namespace

bool mix_geometry(int C, int R, int k, size_t budget, MixGeom *out) {
    const int kp = k + (k & 1);
    for (int GS = 16; GS >= 2; GS >>= 1) {
        MixGeom g;
        g.GS = GS;
        g.TP = 8 * GS;
        g.G = kThreads / GS;
        g.kp = kp;
        const size_t xs = (size_t)(C + 1) * g.TP * 2;
        const size_t ys = align_up((size_t)g.TP * (R + 1) * 2, 16);
        const size_t rp = (size_t)g.G * g.TP * 4;
        const size_t fixed = xs + ys + rp;
        if (fixed >= budget) continue;
        const size_t per_expert = (size_t)kp * 8;  // (offset, weight) per entry
        int eb = (int)((budget - fixed) / per_expert);
        // keep room for the part buffer if experts must be split
        if (eb < 1) continue;
        if (eb > R) eb = R;
        int S = 1;
        if (eb < g.G) {
            S = (g.G + eb - 1) / eb;
            if (S > kp / 2) S = kp / 2;
            if (S < 1) S = 1;
        } else if (eb < R) {
            eb = eb / g.G * g.G;  // whole rounds of the G groups per chunk
        }
        int kq = (kp + S - 1) / S;
        kq += kq & 1;
        S = (kp + kq - 1) / kq;
        size_t pp = S > 1 ? (size_t)eb * S * g.TP * 4 : 0;
        while (eb > 1 && fixed + (size_t)eb * per_expert + pp > budget) {
            --eb;
            pp = S > 1 ? (size_t)eb * S * g.TP * 4 : 0;
        }
        if (fixed + (size_t)eb * per_expert + pp > budget) continue;
        g.EB = eb;
        g.S = S;
        g.kq = kq;
        g.off_ys = align_up(xs, 16);
        g.off_rp = align_up(g.off_ys + ys, 16);
        g.off_pp = align_up(g.off_rp + rp, 16);
        g.off_tab = align_up(g.off_pp + pp, 16);
        g.smem = align_up(g.off_tab + (size_t)eb * per_expert, 16);
        if (g.smem > budget) continue;
        *out = g;
        return true;
    }
    return false;
}

cudaError_t launch_mix(const void *x, int N, int HW, int C, int R, int k, moce_dtype_t dt,
                       moce_layout_t lay, const int32_t *pidx, const float *a,
                       const int32_t *resid, int nU, void *y, uint32_t *ctrl, cudaStream_t s,
                       const PerExample &pe) {
    if (N == 0 || HW == 0) return cudaSuccess;
    const bool shared = pe.sup_stride == 0 && pe.resid_stride == 0 && pe.nUa == nullptr;
    if (lay == MOCE_NCHW) {
        const int EPB = 8;
        const dim3 grid((HW + kThreads - 1) / kThreads, (R + 1 + EPB - 1) / EPB, N);
        if (dt == MOCE_BF16)
            mix_nchw_kernel<uint16_t><<<grid, kThreads, 0, s>>>((const uint16_t *)x, HW, C, R, k,
                                                                 pidx, a, resid, nU, EPB,
                                                                 (uint16_t *)y, pe);
        else
            mix_nchw_kernel<float><<<grid, kThreads, 0, s>>>((const float *)x, HW, C, R, k, pidx, a,
                                                              resid, nU, EPB, (float *)y, pe);
        return cudaGetLastError();
    }
    // the wide kernel pays off from 512 channels (at 256 the tiled kernel is faster)
    if (C >= 512 && dt == MOCE_BF16 && C % 8 == 0 &&
        (reinterpret_cast<uintptr_t>(x) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(pidx) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(a) & 15u) == 0 &&
        mix_wide_supported(HW, C, R, k, shared ? nU : C))
        return launch_mix_wide((const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU,
                               (uint16_t *)y, ctrl, s, pe);
    MixGeom g;
    const bool tiled = dt == MOCE_BF16 && C % 8 == 0 &&
                       (reinterpret_cast<uintptr_t>(x) & 15u) == 0 &&
                       mix_geometry(C, R, k, kMixSmemBudget, &g);
    if (tiled) {
        switch (g.GS) {
        case 16: return launch_tiled<16>((const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU, (uint16_t *)y, g, pe, s);
        case 8: return launch_tiled<8>((const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU, (uint16_t *)y, g, pe, s);
        case 4: return launch_tiled<4>((const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU, (uint16_t *)y, g, pe, s);
        default: return launch_tiled<2>((const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU, (uint16_t *)y, g, pe, s);
        }
    }
    const size_t total = (size_t)N * HW * (R + 1);
    size_t blocks = (total + kThreads - 1) / kThreads;
    if (blocks > 65535u * 16u) blocks = 65535u * 16u;
    if (dt == MOCE_BF16)
        mix_nhwc_generic_kernel<uint16_t><<<(unsigned)blocks, kThreads, 0, s>>>(
            (const uint16_t *)x, N, HW, C, R, k, pidx, a, resid, nU, (uint16_t *)y, pe);
    else
        mix_nhwc_generic_kernel<float><<<(unsigned)blocks, kThreads, 0, s>>>(
            (const float *)x, N, HW, C, R, k, pidx, a, resid, nU, (float *)y, pe);
    return cudaGetLastError();
}

}  // namespace moce
