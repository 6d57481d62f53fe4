// Backward of the layer with static supports (Sec. 3.2: the task loss
// differentiates through the selected logit values, never the indices).
// Given dy = dJ/dy for a scalar J, the gradients with respect to x, the
// selected logits and the gate parameters, per example n (chain rule
// through Eq. (expert), Eq. (res), Eq. (weights), Eq. (tau) and the pool):
//   da_{e,i}  = sum_p dy_{p,e} x_{p,S_e[i]}
//   ds_{e,i}  = a_{e,i} (da_{e,i} - sum_j a_{e,j} da_{e,j})
//   dL_{e,i} += ds_{e,i} / tau_e,  dtau_e = -sum_i ds_{e,i} L_{e,i} / tau_e^2
//   dg_e      = dtau_e (tau_max - tau_min) sigma_e (1 - sigma_e)
//   dw2_j += dg_e r_{e,j}, db2 += dg_e, dh_{e,j} = dg_e w2_j [h_{e,j} > 0]
//   dW1_{j,i} += dh_{e,j} u_{e,i}, db1_j += dh_{e,j}, du_{e,i} = sum_j W1_{j,i} dh_{e,j}
//   dz_c   = sum over (e, i) with S_e[i] = c of du_{e,i}
//   dx_{p,c} = sum over (e, i) with S_e[i] = c of a_{e,i} dy_{p,e}
//              + [c in U] dy_{p,R} / |U| + dz_c / HW
// Kernels (every sum in a fixed order, so two calls give the same bits):
//   the inverse support index first: a stable counting sort of the R k
//     entries by channel (channel -> its (e, i) in increasing order), the
//     channels in decreasing entry count, and per-entry tables (the entry's
//     swizzled dy row offset in a tile, its index);
//   dy transposed once to expert-major rows (bwd_dy_transpose_kernel);
//   da and the pool, NHWC bf16 with C % 8 == 0 (bwd_da_nhwc_kernel): the x
//     tile staged as swizzled channel-major bf16 rows by 16-byte loads and a
//     register transpose; CPR lanes per channel hold the channel's positions
//     in fp32 (their sum is the pool partial) and take the channel's entries
//     one after another, each an 8-position dot product with the entry's dy
//     row added over the lanes by a fixed shuffle tree; other layouts and
//     dtypes: bwd_da_kernel (fp32 rows, a thread per (e, i) pair); column
//     sums over the tiles give da and z;
//   the gate: u gathered from z, hpre = W1 u + b1 and du = W1^T dh as tiled
//     FP32 products over all N C_out rows; a warp per row between them for
//     g, tau, the weights and the backward through the softmax, tau and the
//     sigmoid;
//   parameter gradients as fixed-order column sums over the rows (dW1 as a
//     tiled product split over rows, then a column sum over the splits);
//   dz from the inverse index; dx (bwd_dx_nhwc_kernel): lanes (channel, chunk
//     of 8 positions) add the channel's entries from the staged dy rows, the
//     residual row and dz / HW; other layouts and dtypes: bwd_dx_kernel.
#include <math.h>

#include "moce_internal.cuh"

namespace moce {
namespace {

constexpr int kBwdThreads = 256;

template <typename T> __device__ __forceinline__ float ld_val(const T *p);
template <> __device__ __forceinline__ float ld_val<float>(const float *p) { return *p; }
template <> __device__ __forceinline__ float ld_val<uint16_t>(const uint16_t *p) {
    return __uint_as_float((uint32_t)*p << 16);
}

__device__ __forceinline__ size_t at(int layout, int n, int p, int c, int HW, int C) {
    return layout == 0 ? ((size_t)n * HW + p) * (size_t)C + c : ((size_t)n * C + c) * (size_t)HW + p;
}

// Partial da of tile t of example n over all R k pairs, part[n][t][e k + i],
// and the tile's channel sums psum[n][t][c] (the pool).
template <typename T>
__global__ void __launch_bounds__(kBwdThreads) bwd_da_kernel(
    const T *__restrict__ x, const T *__restrict__ dy, int layout, int HW, int C, int R, int k,
    int TP, int tiles, const int32_t *__restrict__ pidx, float *__restrict__ part,
    float *__restrict__ psum) {
    extern __shared__ float bsm[];
    const int n = blockIdx.x / tiles, t = blockIdx.x - n * tiles;
    const int p0 = t * TP, np = min(TP, HW - p0);
    const int RS = TP + 1;  // padded rows: threads on different rows hit different banks
    float *xt = bsm;                        // [C][RS]
    float *dt = bsm + (size_t)C * RS;       // [R][RS] (the routed experts of dy)
    const int E = R + 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = kBwdThreads / 32;
    if (layout == 0) {  // rows of C (E) channels per position: lanes along channels
        for (int p = warp; p < TP; p += nw)
            for (int c = lane; c < C; c += 32)
                xt[c * RS + p] = p < np ? ld_val<T>(x + at(0, n, p0 + p, c, HW, C)) : 0.f;
        for (int p = warp; p < TP; p += nw)
            for (int e = lane; e < R; e += 32)
                dt[e * RS + p] = p < np ? ld_val<T>(dy + at(0, n, p0 + p, e, HW, E)) : 0.f;
    } else {  // rows of HW positions per channel: lanes along positions
        for (int c = warp; c < C; c += nw)
            for (int p = lane; p < TP; p += 32)
                xt[c * RS + p] = p < np ? ld_val<T>(x + at(1, n, p0 + p, c, HW, C)) : 0.f;
        for (int e = warp; e < R; e += nw)
            for (int p = lane; p < TP; p += 32)
                dt[e * RS + p] = p < np ? ld_val<T>(dy + at(1, n, p0 + p, e, HW, E)) : 0.f;
    }
    __syncthreads();
    // the pool, fused: this tile's channel sums (positions past HW are zero)
    float *ps = psum + ((size_t)n * tiles + t) * (size_t)C;
    for (int c = threadIdx.x; c < C; c += kBwdThreads) {
        const float *xr = xt + (size_t)c * RS;
        float s = 0.f;
        for (int p = 0; p < TP; ++p) s += xr[p];
        ps[c] = s;
    }
    float *out = part + ((size_t)n * tiles + t) * (size_t)R * k;
    for (int j = threadIdx.x; j < R * k; j += kBwdThreads) {
        const int e = j / k, c = __ldg(pidx + j);
        const float *xr = xt + (size_t)c * RS, *dr = dt + (size_t)e * RS;
        float s = 0.f;
        for (int p = 0; p < TP; ++p) s = fmaf(dr[p], xr[p], s);
        out[j] = s;
    }
}

// ---------------------------------------------------------------- NHWC bf16 tiles
// The fast kernels for NHWC bf16 layers with C % 8 == 0 keep TP positions of
// one example on chip as channel-major bf16 rows (TP * 2 bytes: CPR = TP / 8
// chunks of 16 bytes, 8 positions each). Chunk q of row r sits at chunk
// q ^ swz(r), so that the 8 lanes that read the CPR chunks of one row hit
// distinct bank groups, and 32 lanes that write one word of 32 consecutive
// rows spread over all 8 (a 4-way conflict, the least for 32 lanes on one
// bank of a group).
__device__ __forceinline__ int swz_x(int c, int CPR) {  // x rows: channel c
    return ((c >> 3) >> (CPR == 8 ? 0 : CPR == 4 ? 1 : 2)) & (CPR - 1);
}
__device__ __forceinline__ int swz_d(int e, int CPR) {  // dy rows: expert e
    return (e >> (CPR == 8 ? 0 : CPR == 4 ? 1 : 2)) & (CPR - 1);
}

// e = j / k for quotients below 2^20 (the float estimate is off by at most one).
__device__ __forceinline__ int div_k(int j, int k, float inv_k) {
    int e = __float2int_rz((float)j * inv_k);
    if (e * k > j) --e;
    else if ((e + 1) * k <= j) ++e;
    return e;
}

__device__ __forceinline__ void fma8(float *acc, float w, uint4 v) {
    acc[0] = fmaf(w, bf16lo(v.x), acc[0]); acc[1] = fmaf(w, bf16hi(v.x), acc[1]);
    acc[2] = fmaf(w, bf16lo(v.y), acc[2]); acc[3] = fmaf(w, bf16hi(v.y), acc[3]);
    acc[4] = fmaf(w, bf16lo(v.z), acc[4]); acc[5] = fmaf(w, bf16hi(v.z), acc[5]);
    acc[6] = fmaf(w, bf16lo(v.w), acc[6]); acc[7] = fmaf(w, bf16hi(v.w), acc[7]);
}

// dy of example n transposed to expert-major rows of HWp positions (HWp =
// HW rounded up to 64, zero past HW): dyT[n][e][p] = dy[n][p][e]. 64
// positions x 32 experts per CTA through shared memory; stores of two
// positions per lane, 128 bytes per warp.
__global__ void __launch_bounds__(256) bwd_dy_transpose_kernel(const uint16_t *__restrict__ dy,
                                                               int HW, int HWp, int E,
                                                               uint16_t *__restrict__ dyT) {
    __shared__ uint16_t tt[32][66];
    const int p0 = blockIdx.x * 64, e0 = blockIdx.y * 32, n = blockIdx.z;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int e = e0 + tx;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        const int p = ty + 8 * r;
        tt[tx][p] = (p0 + p < HW && e < E) ? __ldg(dy + ((size_t)n * HW + p0 + p) * E + e)
                                          : (uint16_t)0;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int el = ty + 8 * r, ee = e0 + el;
        if (ee < E) {
            const uint32_t w = (uint32_t)tt[el][2 * tx] | ((uint32_t)tt[el][2 * tx + 1] << 16);
            *reinterpret_cast<uint32_t *>(dyT + ((size_t)n * E + ee) * HWp + p0 + 2 * tx) = w;
        }
    }
}

// Rows 0..E-1 of a TP-position tile from dyT (row stride HWp) into the
// swizzled channel-major layout: 16-byte copies, four in flight per thread.
template <int TP, int NT = 256>
__device__ __forceinline__ void stage_dyT_rows(const uint16_t *__restrict__ src, int HWp, int E,
                                               unsigned char *ds) {
    constexpr int CPR = TP / 8;
    const int total = E * CPR;
    for (int v0 = threadIdx.x; v0 < total; v0 += 4 * NT) {
        uint4 w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int v = v0 + u * NT, e = v / CPR, q = v % CPR;
            w[u] = v < total ? __ldg(reinterpret_cast<const uint4 *>(src + (size_t)e * HWp) + q)
                             : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int v = v0 + u * NT, e = v / CPR, q = v % CPR;
            if (v < total)
                *reinterpret_cast<uint4 *>(ds + (size_t)e * TP * 2 + ((q ^ swz_d(e, CPR)) << 4)) =
                    w[u];
        }
    }
}

// da partials of one tile and the pool partials, NHWC bf16, C % 8 == 0.
// Staging: a thread loads 8 positions x 8 channels (eight 16-byte loads),
// transposes them in registers and stores one chunk in each of 8 rows (8
// consecutive channel groups hit 8 bank groups at TP = 64; 2 or 4 share one
// at TP = 32 or 16).
// Compute, channel-major: CPR lanes per channel, one chunk of 8 positions
// each, unpacked to fp32 once; the channel's tile sum is the pool partial,
// then for each entry j of the channel (dtab[m] = {swizzled dy row offset,
// j}) an 8-position dot product with the entry's dy row, added over the CPR
// lanes by a fixed shuffle tree. Channels come in decreasing entry count
// (corder), so the lanes of a warp loop about equally long; which lane takes
// a channel does not change its sums.
template <int TP, int NT>
__global__ void __launch_bounds__(NT) bwd_da_nhwc_kernel(
    const uint16_t *__restrict__ x, const uint16_t *__restrict__ dyT, int HW, int HWp, int C,
    int R, int tiles, const int32_t *__restrict__ corder, const int32_t *__restrict__ ptr,
    const int2 *__restrict__ dtab, int J, float *__restrict__ part, float *__restrict__ psum) {
    constexpr int CPR = TP / 8;
    // entries of a channel in flight per step: wide layers' channels have many
    constexpr int kEU = TP == 64 ? 4 : 8;
    extern __shared__ __align__(16) unsigned char fsm[];
    unsigned char *xs = fsm;                       // [C][TP] bf16
    unsigned char *ds = fsm + (size_t)C * TP * 2;  // [R][TP] bf16
    const int n = blockIdx.x / tiles, t = blockIdx.x - n * tiles;
    const int p0 = t * TP, np = min(TP, HW - p0);
    const int C8 = C >> 3;
    const uint16_t *xn = x + ((size_t)n * HW + p0) * C;
    for (int v = threadIdx.x; v < CPR * C8; v += NT) {
        const int pg = v / C8, c8 = v - pg * C8;
        uint4 w[8];
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const int p = pg * 8 + r;
            w[r] = p < np ? __ldg(reinterpret_cast<const uint4 *>(xn + (size_t)p * C) + c8)
                          : make_uint4(0u, 0u, 0u, 0u);
        }
        const uint32_t *wv = reinterpret_cast<const uint32_t *>(w);  // wv[r * 4 + channel pair]
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int pair = u >> 1;
            const uint32_t sel = (u & 1) ? 0x7632u : 0x5410u;
            uint4 o;
            o.x = __byte_perm(wv[0 * 4 + pair], wv[1 * 4 + pair], sel);
            o.y = __byte_perm(wv[2 * 4 + pair], wv[3 * 4 + pair], sel);
            o.z = __byte_perm(wv[4 * 4 + pair], wv[5 * 4 + pair], sel);
            o.w = __byte_perm(wv[6 * 4 + pair], wv[7 * 4 + pair], sel);
            const int c = c8 * 8 + u;
            *reinterpret_cast<uint4 *>(xs + (size_t)c * TP * 2 + ((pg ^ swz_x(c, CPR)) << 4)) = o;
        }
    }
    stage_dyT_rows<TP, NT>(dyT + (size_t)n * (R + 1) * HWp + p0, HWp, R, ds);
    __syncthreads();
    const int lane = threadIdx.x & 31, q = lane % CPR;
    constexpr int SPW = 32 / CPR;  // channels per warp step
    float *out = part + ((size_t)n * tiles + t) * (size_t)J;
    float *ps = psum + ((size_t)n * tiles + t) * C;
    for (int sb = (threadIdx.x >> 5) * SPW; sb < C; sb += (NT / 32) * SPW) {
        const int sl = sb + lane / CPR;
        const bool valid = sl < C;
        const int c = valid ? __ldg(corder + sl) : 0;
        const uint4 xv = *reinterpret_cast<const uint4 *>(xs + (size_t)c * TP * 2 +
                                                          ((q ^ swz_x(c, CPR)) << 4));
        float xf[8] = {bf16lo(xv.x), bf16hi(xv.x), bf16lo(xv.y), bf16hi(xv.y),
                       bf16lo(xv.z), bf16hi(xv.z), bf16lo(xv.w), bf16hi(xv.w)};
        float pl = xf[0];
#pragma unroll
        for (int r = 1; r < 8; ++r) pl += xf[r];
#pragma unroll
        for (int o = CPR / 2; o > 0; o >>= 1) pl += __shfl_xor_sync(0xffffffffu, pl, o);
        if (valid && q == 0) ps[c] = pl;
        const int m0 = valid ? __ldg(ptr + c) : 0;
        const int cnt = valid ? __ldg(ptr + c + 1) - m0 : 0;
        const int cmax = (int)__reduce_max_sync(0xffffffffu, (unsigned)cnt);
        const uint32_t qx = (uint32_t)q << 4;
        for (int i = 0; i < cmax; i += kEU) {
            int2 tb[kEU];
            float d[kEU];
#pragma unroll
            for (int u = 0; u < kEU; ++u)
                tb[u] = i + u < cnt ? __ldg(dtab + m0 + i + u) : make_int2(0, -1);
#pragma unroll
            for (int u = 0; u < kEU; ++u) {
                const uint4 dv = *reinterpret_cast<const uint4 *>(ds + ((uint32_t)tb[u].x ^ qx));
                float sm = bf16lo(dv.x) * xf[0];
                sm = fmaf(bf16hi(dv.x), xf[1], sm);
                sm = fmaf(bf16lo(dv.y), xf[2], sm);
                sm = fmaf(bf16hi(dv.y), xf[3], sm);
                sm = fmaf(bf16lo(dv.z), xf[4], sm);
                sm = fmaf(bf16hi(dv.z), xf[5], sm);
                sm = fmaf(bf16lo(dv.w), xf[6], sm);
                sm = fmaf(bf16hi(dv.w), xf[7], sm);
                d[u] = sm;
            }
#pragma unroll
            for (int o = CPR / 2; o > 0; o >>= 1)
#pragma unroll
                for (int u = 0; u < kEU; ++u) d[u] += __shfl_xor_sync(0xffffffffu, d[u], o);
            if (q == 0) {
#pragma unroll
                for (int u = 0; u < kEU; ++u)
                    if (tb[u].y >= 0) out[tb[u].y] = d[u];
            }
        }
    }
}

// Byte offset of the staged tables in a dx tile's shared memory (after the
// R + 1 dy rows), and whether an example's tables (J weights, J row offsets,
// C + 1 row pointers) are staged.
__host__ __device__ inline size_t dx_tab_off(int R, int TP) {
    return align_up((size_t)(R + 1) * TP * 2, 16);
}
inline size_t dx_tab_bytes(int J, int C) { return (size_t)J * 8 + (size_t)(C + 1) * 4; }
constexpr size_t kDxTabMax = 96 * 1024;

// dx of one tile, NHWC bf16 dy: lane = (channel c, chunk q of 8 positions);
// the entries of c in increasing order (doff[m]: the entry's swizzled dy row
// offset; am[n][m]: its weight a), then the residual expert and dz / HW.
template <int TP>
__global__ void __launch_bounds__(256) bwd_dx_nhwc_kernel(
    const uint16_t *__restrict__ dyT, int HW, int HWp, int C, int R, int J, int tiles,
    const float *am, const int32_t *ptr, const int32_t *doff, const uint8_t *__restrict__ inU,
    float inv_nU, const float *__restrict__ dz, float *__restrict__ dx, int tab) {
    constexpr int CPR = TP / 8;
    extern __shared__ __align__(16) unsigned char fsm[];
    unsigned char *ds = fsm;  // [R + 1][TP] bf16
    const int n = blockIdx.x / tiles, t = blockIdx.x - n * tiles;
    const int p0 = t * TP, np = min(TP, HW - p0);
    stage_dyT_rows<TP>(dyT + (size_t)n * (R + 1) * HWp + p0, HWp, R + 1, ds);
    const float *an = am + (size_t)n * J;
    if (tab) {  // the example's tables fit: entry weights, row offsets and row pointers staged
        float *tw = reinterpret_cast<float *>(fsm + dx_tab_off(R, TP));
        int32_t *to = reinterpret_cast<int32_t *>(tw + J);
        int32_t *tp = to + J;
        for (int m = threadIdx.x; m < J; m += 256) {
            tw[m] = __ldg(an + m);
            to[m] = __ldg(doff + m);
        }
        for (int c = threadIdx.x; c <= C; c += 256) tp[c] = __ldg(ptr + c);
        an = tw;
        doff = to;
        ptr = tp;
    }
    __syncthreads();
    const float inv_HW = 1.f / (float)HW;
    float *dxn = dx + ((size_t)n * HW + p0) * C;
    const uint32_t roff = (uint32_t)R * TP * 2 + ((uint32_t)swz_d(R, CPR) << 4);
    for (int T = threadIdx.x; T < C * CPR; T += 256) {
        const int c = T / CPR, q = T % CPR;
        const uint32_t qx = (uint32_t)q << 4;
        float acc[8];
        const float base = dz[(size_t)n * C + c] * inv_HW;
#pragma unroll
        for (int r = 0; r < 8; ++r) acc[r] = base;
        const int m1 = ptr[c + 1];
        int m = ptr[c];
        for (; m + 4 <= m1; m += 4) {  // four entries' loads in flight
            uint32_t of[4];
            float ww[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                of[u] = (uint32_t)doff[m + u];
                ww[u] = an[m + u];
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                fma8(acc, ww[u], *reinterpret_cast<const uint4 *>(ds + (of[u] ^ qx)));
        }
        for (; m < m1; ++m)
            fma8(acc, an[m], *reinterpret_cast<const uint4 *>(ds + ((uint32_t)doff[m] ^ qx)));
        if (inU[c]) fma8(acc, inv_nU, *reinterpret_cast<const uint4 *>(ds + (roff ^ qx)));
#pragma unroll
        for (int r = 0; r < 8; ++r)
            if (q * 8 + r < np) dxn[(size_t)(q * 8 + r) * C + c] = acc[r];
    }
}

// Tables of the fast kernels, from the inverse index: for entry slot m (entry
// j = ent[m] of expert e = j / k), dtab[m] = {e's dy row offset in a da tile
// of TPa positions, swizzle folded in; j}, doff[m] = the same in a dx tile
// of TPx positions, and am[n][m] = a[n][j].
__global__ void bwd_tables_kernel(const int32_t *__restrict__ ent, int J, int k, float inv_k,
                                  int TPa, int TPx, int2 *__restrict__ dtab,
                                  int32_t *__restrict__ doff) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= J) return;
    const int j = ent[m], e = div_k(j, k, inv_k);
    if (TPa) dtab[m] = make_int2(e * TPa * 2 + (swz_d(e, TPa / 8) << 4), j);
    doff[m] = e * TPx * 2 + (swz_d(e, TPx / 8) << 4);
}
__global__ void bwd_gather_a_kernel(const float *__restrict__ a, const int32_t *__restrict__ ent,
                                    int N, int J, float *__restrict__ am) {
    const size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= (size_t)N * J) return;
    const size_t n = q / J;
    am[q] = a[n * J + ent[q - n * J]];
}

// Channels in decreasing entry count (any order within a count): bins of
// the counts, their starts from the largest count down, then a slot each.
__global__ void bwd_count_bins_kernel(const int32_t *__restrict__ cnt, int C, int R,
                                      int32_t *__restrict__ bins) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c < C) atomicAdd(bins + min(cnt[c], R), 1);
}
__global__ void __launch_bounds__(1024) bwd_bins_scan_kernel(int32_t *__restrict__ bins, int R) {
    __shared__ int32_t part[1024];
    const int t = threadIdx.x, B = R + 1, per = (B + 1023) / 1024;
    const int r0 = min(B, t * per), r1 = min(B, r0 + per);  // runs of bins R, R-1, ...
    int sm = 0;
    for (int r = r0; r < r1; ++r) sm += bins[R - r];
    part[t] = sm;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {
        const int v = t >= o ? part[t - o] : 0;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    int w = part[t] - sm;
    for (int r = r0; r < r1; ++r) {
        const int b = bins[R - r];
        bins[R - r] = w;
        w += b;
    }
}
__global__ void bwd_order_kernel(const int32_t *__restrict__ cnt, int C, int R,
                                 int32_t *__restrict__ bins, int32_t *__restrict__ corder) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c < C) corder[atomicAdd(bins + min(cnt[c], R), 1)] = c;
}

// Deterministic column sums: out[b][chunk][col] = (sum over the chunk's rows
// r of A[b][r][col]) / div. A CTA of 32 columns x 8 row lanes: lane y sums
// rows y, y + 8, ... of the chunk in order, then a fixed tree adds the 8
// lanes, so the result never depends on scheduling.
constexpr int kSumLanes = 8;
__global__ void __launch_bounds__(32 * kSumLanes) colsum_kernel(const float *__restrict__ A,
                                                                size_t rows, int K, size_t RB,
                                                                float div, float *__restrict__ out) {
    __shared__ float red[kSumLanes][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int col = blockIdx.x * 32 + tx;
    const size_t chunk = blockIdx.y, b = blockIdx.z;
    const size_t r0 = chunk * RB, r1 = min(rows, r0 + RB);
    const float *Ab = A + b * rows * (size_t)K;
    float s = 0.f;
    if (col < K)
        for (size_t r = r0 + ty; r < r1; r += kSumLanes) s += Ab[r * K + col];
    red[ty][tx] = s;
    __syncthreads();
#pragma unroll
    for (int o = kSumLanes / 2; o > 0; o >>= 1) {
        if (ty < o) red[ty][tx] += red[ty + o][tx];
        __syncthreads();
    }
    if (ty == 0 && col < K) out[(b * gridDim.y + chunk) * K + col] = red[0][tx] / div;
}

// Rows per chunk of the first pass: at most 256 chunks, then one more pass.
size_t colsum_rb(size_t rows) {
    size_t rb = (rows + 255) / 256;
    rb = (rb + 7) / 8 * 8;
    return rb < 64 ? 64 : rb;
}
size_t colsum_tmp_elems(int batch, size_t rows, int K) {
    const size_t ch = (rows + colsum_rb(rows) - 1) / colsum_rb(rows);
    return ch > 1 ? (size_t)batch * ch * K : 0;
}
// out[b][K] = (sum over rows of A[b][rows][K]) / div; tmp holds
// colsum_tmp_elems floats.
void colsum(const float *A, int batch, size_t rows, int K, float div, float *out, float *tmp,
            cudaStream_t s) {
    const size_t rb = colsum_rb(rows), ch = (rows + rb - 1) / rb;
    const dim3 blk(32 * kSumLanes);
    const unsigned gx = (unsigned)((K + 31) / 32);
    if (ch <= 1) {
        colsum_kernel<<<dim3(gx, 1, batch), blk, 0, s>>>(A, rows, K, rb, div, out);
        return;
    }
    colsum_kernel<<<dim3(gx, (unsigned)ch, batch), blk, 0, s>>>(A, rows, K, rb, 1.f, tmp);
    colsum_kernel<<<dim3(gx, 1, batch), blk, 0, s>>>(tmp, ch, K, ch, div, out);
}

// FP32 tiled product C[z][m][n] = bias[n] + sum over kk in split z of
// A(m, kk) B(kk, n), with A(m, kk) = A[m a_m + kk a_k], B(kk, n) =
// B[kk b_k + n b_n] (one of each pair of strides is 1). 64 x 64 tiles,
// 16-deep slices in shared memory, 4 x 4 outputs per thread.
struct GemmArgs {
    const float *A;
    size_t a_m, a_k;
    const float *B;
    size_t b_k, b_n;
    const float *bias;
    float *C;
    int M, Nn;
    size_t K, kchunk;
};
__global__ void __launch_bounds__(256) sgemm_kernel(GemmArgs g) {
    __shared__ __align__(16) float As[16][68], Bs[16][68];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int m0 = blockIdx.x * 64, n0 = blockIdx.y * 64;
    const size_t k0 = (size_t)blockIdx.z * g.kchunk, k1 = min(g.K, k0 + g.kchunk);
    float acc[4][4] = {};
    for (size_t kb = k0; kb < k1; kb += 16) {
#pragma unroll
        for (int l = 0; l < 4; ++l) {
            const int q = tid + 256 * l;
            int m, kk;
            if (g.a_k == 1) { kk = q & 15; m = q >> 4; } else { m = q & 63; kk = q >> 6; }
            const size_t gk = kb + kk;
            const int gm = m0 + m;
            As[kk][m] = gm < g.M && gk < k1 ? g.A[gm * g.a_m + gk * g.a_k] : 0.f;
            int n;
            if (g.b_n == 1) { n = q & 63; kk = q >> 6; } else { kk = q & 15; n = q >> 4; }
            const size_t gk2 = kb + kk;
            const int gn = n0 + n;
            Bs[kk][n] = gn < g.Nn && gk2 < k1 ? g.B[gk2 * g.b_k + gn * g.b_n] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            const float4 av = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
            const float4 bv = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
            const float ar[4] = {av.x, av.y, av.z, av.w}, br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(ar[i], br[j], acc[i][j]);
        }
        __syncthreads();
    }
    float *Cz = g.C + (size_t)blockIdx.z * g.M * g.Nn;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
        if (m >= g.M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (n < g.Nn) Cz[(size_t)m * g.Nn + n] = acc[i][j] + (g.bias ? __ldg(g.bias + n) : 0.f);
        }
    }
}
void sgemm(const GemmArgs &g, int splits, cudaStream_t s) {
    const dim3 grid((unsigned)((g.M + 63) / 64), (unsigned)((g.Nn + 63) / 64), (unsigned)splits);
    sgemm_kernel<<<grid, 256, 0, s>>>(g);
}

// u[r][i] = z[n][S_e[i]] for rows r = n R + e (Sec. 3.3: the gate reads the
// pooled descriptors of the expert's support, in packed order).
__global__ void bwd_gather_kernel(const float *__restrict__ z, int C, int R, int k,
                                  const int32_t *__restrict__ pidx, size_t total,
                                  float *__restrict__ u) {
    const size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= total) return;
    const size_t r = q / k;
    const int i = (int)(q - r * k);
    const size_t n = r / R;
    const int e = (int)(r - n * R);
    u[q] = z[n * C + __ldg(pidx + (size_t)e * k + i)];
}

// A warp per row r = n R + e, from the hidden pre-activations hpre = W1 u + b1:
// g, sigma, tau (Eq. (tau)), the weights a (Eq. (weights)) and the backward
// through them: dlp = ds / tau, dg, dgr_j = dg ReLU(h_j) (for dw2) and
// dh_j = dg w2_j [h_j > 0] (for W1, b1 and u).
__global__ void __launch_bounds__(256) bwd_gate_rows_kernel(
    const float *__restrict__ hpre, const float *__restrict__ da, size_t rows, int R, int k,
    const float *__restrict__ plog, const float *__restrict__ w2, const float *__restrict__ b2,
    float tmin, float tmax, float *__restrict__ a_out, float *__restrict__ dlp_out,
    float *__restrict__ dg_out, float *__restrict__ dgr_out, float *__restrict__ dh_out) {
    const int lane = threadIdx.x & 31;
    const size_t r = (size_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (r >= rows) return;
    const int e = (int)(r % R);
    const size_t base = r * k;
    const float *h = hpre + base;
    float g = 0.f;
    for (int j = lane; j < k; j += 32) g = fmaf(__ldg(w2 + j), fmaxf(h[j], 0.f), g);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
    g += __ldg(b2);
    const float sig = 1.f / (1.f + expf(-g));
    const float tau = tmin + (tmax - tmin) * sig;
    const float *L = plog + (size_t)e * k;
    float Lm = -INFINITY;
    for (int i = lane; i < k; i += 32) Lm = fmaxf(Lm, __ldg(L + i));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) Lm = fmaxf(Lm, __shfl_xor_sync(0xffffffffu, Lm, o));
    float sum = 0.f;
    for (int i = lane; i < k; i += 32) sum += expf((__ldg(L + i) - Lm) / tau);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    float ada = 0.f;
    for (int i = lane; i < k; i += 32) {
        const float ai = expf((__ldg(L + i) - Lm) / tau) / sum;
        a_out[base + i] = ai;
        ada = fmaf(ai, da[base + i], ada);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ada += __shfl_xor_sync(0xffffffffu, ada, o);
    float dtau = 0.f;
    for (int i = lane; i < k; i += 32) {
        const float ds = a_out[base + i] * (da[base + i] - ada);
        dlp_out[base + i] = ds / tau;
        dtau -= ds * __ldg(L + i) / (tau * tau);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dtau += __shfl_xor_sync(0xffffffffu, dtau, o);
    const float dg = dtau * (tmax - tmin) * sig * (1.f - sig);
    if (lane == 0) dg_out[r] = dg;
    for (int j = lane; j < k; j += 32) {
        const float hj = h[j];
        dgr_out[base + j] = dg * fmaxf(hj, 0.f);
        dh_out[base + j] = hj > 0.f ? dg * __ldg(w2 + j) : 0.f;
    }
}

// Inverse support index: a stable counting sort of the entries j = e k + i
// by channel pidx[j], so each channel lists its entries in increasing j and
// every later sum over them runs in that order. Blocks of `chunk` entries
// (a multiple of 32, about J / 256):
// per-block channel counts, a scan over (channel, block), then each block
// places its entries in order (one warp, 32 entries a step, equal channels
// ranked by lane).
int inv_chunk(int J) {
    int ch = (J + 255) / 256;
    ch = (ch + 31) / 32 * 32;
    return ch < 64 ? 64 : ch;
}
__global__ void __launch_bounds__(32) bwd_inv_hist_kernel(const int32_t *__restrict__ pidx, int J,
                                                          int C, int chunk,
                                                          int32_t *__restrict__ hist) {
    extern __shared__ int32_t cnt_s[];
    const int b = blockIdx.x, lane = threadIdx.x;
    for (int c = lane; c < C; c += 32) cnt_s[c] = 0;
    __syncwarp();
    const int j1 = min(J, (b + 1) * chunk);
    for (int j0 = b * chunk; j0 < j1; j0 += 32) {
        const int j = j0 + lane;
        int c = j < j1 ? __ldg(pidx + j) : -1;
        if ((unsigned)c >= (unsigned)C) c = -1 - lane;  // past the end: a key of its own
        const uint32_t peers = __match_any_sync(0xffffffffu, c);
        if (c >= 0 && (peers & ((1u << lane) - 1u)) == 0) cnt_s[c] += __popc(peers);
        __syncwarp();
    }
    for (int c = lane; c < C; c += 32) hist[(size_t)b * C + c] = cnt_s[c];
}

// Per channel: hist[b][c] becomes the entries of channel c in blocks before
// b; cnt[c] the channel's total. Then ptr = the exclusive scan of cnt (one
// CTA of 1024 threads, each over a run of consecutive channels).
__global__ void bwd_inv_colscan_kernel(int32_t *__restrict__ hist, int nb, int C,
                                       int32_t *__restrict__ cnt) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    int s = 0;
    for (int b0 = 0; b0 < nb; b0 += 8) {  // eight loads in flight, then the stores
        int v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = b0 + u < nb ? hist[(size_t)(b0 + u) * C + c] : 0;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (b0 + u < nb) hist[(size_t)(b0 + u) * C + c] = s;
            s += v[u];
        }
    }
    cnt[c] = s;
}
__global__ void __launch_bounds__(1024) bwd_inv_scan_kernel(const int32_t *__restrict__ cnt, int C,
                                                            int32_t *__restrict__ ptr) {
    __shared__ int32_t part[1024];
    const int t = threadIdx.x, per = (C + 1023) / 1024;
    const int c0 = min(C, t * per), c1 = min(C, c0 + per);
    int s = 0;
    for (int c = c0; c < c1; ++c) s += cnt[c];
    part[t] = s;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {  // inclusive Hillis-Steele scan
        const int v = t >= o ? part[t - o] : 0;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    int w = part[t] - s;
    for (int c = c0; c < c1; ++c) {
        ptr[c] = w;
        w += cnt[c];
    }
    if (t == 1023) ptr[C] = part[1023];
}
__global__ void __launch_bounds__(32) bwd_inv_place_kernel(const int32_t *__restrict__ pidx, int J,
                                                           int C, int chunk,
                                                           const int32_t *__restrict__ hist,
                                                           const int32_t *__restrict__ ptr,
                                                           int32_t *__restrict__ ent) {
    extern __shared__ int32_t pos_s[];
    const int b = blockIdx.x, lane = threadIdx.x;
    for (int c = lane; c < C; c += 32) pos_s[c] = ptr[c] + hist[(size_t)b * C + c];
    __syncwarp();
    const int j1 = min(J, (b + 1) * chunk);
    for (int j0 = b * chunk; j0 < j1; j0 += 32) {
        const int j = j0 + lane;
        int c = j < j1 ? __ldg(pidx + j) : -1;
        if ((unsigned)c >= (unsigned)C) c = -1 - lane;
        const uint32_t peers = __match_any_sync(0xffffffffu, c);
        if (c >= 0) {
            ent[pos_s[c] + __popc(peers & ((1u << lane) - 1u))] = j;
        }
        __syncwarp();
        if (c >= 0 && (peers & ((1u << lane) - 1u)) == 0) pos_s[c] += __popc(peers);
        __syncwarp();
    }
}

// dz[n][c] = sum over the channel's entries j (increasing) of du[n][j].
__global__ void bwd_dz_kernel(const float *__restrict__ du, int N, int C, int J,
                              const int32_t *__restrict__ ptr, const int32_t *__restrict__ ent,
                              float *__restrict__ dz) {
    const size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= (size_t)N * C) return;
    const size_t n = q / C;
    const int c = (int)(q - n * C);
    float s = 0.f;
    for (int m = ptr[c]; m < ptr[c + 1]; ++m) s += du[n * J + ent[m]];
    dz[q] = s;
}

// dx of tile t of example n: thread per channel, TPX positions in registers.
constexpr int TPX = 16;
template <typename T>
__global__ void __launch_bounds__(kBwdThreads) bwd_dx_kernel(
    const T *__restrict__ dy, int layout, int HW, int C, int R, int k, int tiles,
    const float *__restrict__ a, const int32_t *__restrict__ ptr, const int32_t *__restrict__ ent,
    const uint8_t *__restrict__ inU, float inv_nU, const float *__restrict__ dz,
    float *__restrict__ dx) {
    extern __shared__ float dsm[];
    const int n = blockIdx.x / tiles, t = blockIdx.x - n * tiles;
    const int p0 = t * TPX, np = min(TPX, HW - p0);
    const int E = R + 1, RS = TPX + 1;
    float *dt = dsm;  // [E][RS]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = kBwdThreads / 32;
    if (layout == 0) {
        for (int p = warp; p < TPX; p += nw)
            for (int e = lane; e < E; e += 32)
                dt[e * RS + p] = p < np ? ld_val<T>(dy + at(0, n, p0 + p, e, HW, E)) : 0.f;
    } else {
        for (int e = warp; e < E; e += nw)
            for (int p = lane; p < TPX; p += 32)
                dt[e * RS + p] = p < np ? ld_val<T>(dy + at(1, n, p0 + p, e, HW, E)) : 0.f;
    }
    __syncthreads();
    const float *an = a + (size_t)n * R * k;
    const float inv_HW = 1.f / (float)HW;
    for (int c = threadIdx.x; c < C; c += kBwdThreads) {
        float acc[TPX];
        const float base = dz[(size_t)n * C + c] * inv_HW;
#pragma unroll
        for (int p = 0; p < TPX; ++p) acc[p] = base;
        for (int m = ptr[c]; m < ptr[c + 1]; ++m) {
            const int j = ent[m];
            const float w = an[j];
            const float *dr = dt + (size_t)(j / k) * RS;
#pragma unroll
            for (int p = 0; p < TPX; ++p) acc[p] = fmaf(w, dr[p], acc[p]);
        }
        if (inU[c]) {
            const float *dr = dt + (size_t)R * RS;
#pragma unroll
            for (int p = 0; p < TPX; ++p) acc[p] = fmaf(inv_nU, dr[p], acc[p]);
        }
#pragma unroll
        for (int p = 0; p < TPX; ++p)
            if (p < np) dx[at(layout, n, p0 + p, c, HW, C)] = acc[p];
    }
}

__global__ void bwd_set_resid_kernel(const int32_t *__restrict__ resid, int nU,
                                     uint8_t *__restrict__ inU) {
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q < nU) inU[__ldg(resid + q)] = 1;
}

// Positions per tile of the fast da kernel (0: none fits): the largest of 64,
// 32, 16 whose tiles leave room for two CTAs per SM, else for one.
size_t da_fast_smem(int C, int R, int TP) { return (size_t)(C + R) * TP * 2; }
int da_fast_tile(int C, int R) {
    if (C % 8) return 0;
    for (int TP = 64; TP >= 16; TP >>= 1)
        if (da_fast_smem(C, R, TP) <= 113 * 1024) return TP;
    for (int TP = 64; TP >= 16; TP >>= 1)
        if (da_fast_smem(C, R, TP) <= 227 * 1024) return TP;
    return 0;
}
constexpr int kDxFastTile = 64;

// Positions per da tile: the largest of 64, 32, 16, 8 whose staged rows fit.
int da_tile(int C, int R) {
    for (int TP = 64; TP >= 8; TP >>= 1)
        if ((size_t)(C + R) * (TP + 1) * 4 <= 200 * 1024) return TP;
    return 0;
}

}  // namespace

// Workspace of the backward (moce_backward_workspace_bytes).
struct BwdLayout {
    size_t psum = 0, z = 0, part = 0, da = 0, u = 0, h = 0, a = 0, dlp = 0, dg = 0, dgr = 0,
           dh = 0, du = 0, wpart = 0, tmp = 0, hist = 0, cnt = 0, ptr = 0, ent = 0, inU = 0,
           dz = 0, bins = 0, corder = 0, dtab = 0, doff = 0, am = 0, dyT = 0, total = 0;
    int TP = 0, tiles = 0, splits = 0;
    size_t kchunk = 0;
};

static BwdLayout bwd_layout(int N, int HW, int C, int R, int k) {
    BwdLayout B;
    B.TP = da_tile(C, R);
    if (B.TP == 0 || (size_t)(R + 1) * (TPX + 1) * 4 > 227 * 1024 || (size_t)C * 4 > 227 * 1024) {
        B.TP = 0;
        return B;
    }
    const int tf = da_fast_tile(C, R);
    const int tmin = tf && tf < B.TP ? tf : B.TP;
    B.tiles = (HW + tmin - 1) / tmin;  // partial rows for either da kernel
    const size_t rows = (size_t)N * R, J = (size_t)R * k, kk = (size_t)k * k;
    // dW1 = sum over rows of dh (x) u: split over rows so that about 600 CTAs run
    const size_t wt = (size_t)((k + 63) / 64) * ((k + 63) / 64);
    size_t splits = (600 + wt - 1) / wt, max_splits = (rows + 63) / 64;
    if (splits > max_splits) splits = max_splits;
    if (splits < 1) splits = 1;
    B.kchunk = align_up((rows + splits - 1) / splits, 16);
    B.splits = (int)((rows + B.kchunk - 1) / B.kchunk);
    if (B.splits < 1) B.splits = 1;
    auto mx = [](size_t a, size_t b) { return a > b ? a : b; };
    size_t tmp = colsum_tmp_elems(N, B.tiles, (int)J);
    tmp = mx(tmp, colsum_tmp_elems(N, B.tiles, C));
    tmp = mx(tmp, colsum_tmp_elems(1, N, (int)J));
    tmp = mx(tmp, colsum_tmp_elems(1, rows, k));
    tmp = mx(tmp, colsum_tmp_elems(1, B.splits, (int)kk));
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
    B.psum = take((size_t)N * B.tiles * C * 4);
    B.z = take((size_t)N * C * 4);
    B.part = take((size_t)N * B.tiles * J * 4);
    B.da = take(rows * k * 4);
    B.u = take(rows * k * 4);
    B.h = take(rows * k * 4);
    B.a = take(rows * k * 4);
    B.dlp = take(rows * k * 4);
    B.dg = take(rows * 4);
    B.dgr = take(rows * k * 4);
    B.dh = take(rows * k * 4);
    B.du = take(rows * k * 4);
    B.wpart = take((size_t)B.splits * kk * 4);
    B.tmp = take(tmp * 4);
    B.hist = take((size_t)((J + inv_chunk((int)J) - 1) / inv_chunk((int)J)) * C * 4);
    B.cnt = take((size_t)C * 4);
    B.ptr = take((size_t)(C + 1) * 4);
    B.ent = take(J * 4);
    B.inU = take((size_t)C);
    B.dz = take((size_t)N * C * 4);
    B.bins = take((size_t)(R + 1) * 4);
    B.corder = take((size_t)C * 4);
    B.dtab = take(J * 8);
    B.doff = take(J * 4);
    B.am = take(rows * k * 4);
    B.dyT = take((size_t)N * (R + 1) * align_up((size_t)HW, 64) * 2);
    B.total = off;
    return B;
}

size_t backward_ws_bytes(int N, int HW, int C, int R, int k) {
    const BwdLayout B = bwd_layout(N, HW, C, R, k);
    return B.TP ? B.total : 0;
}

cudaError_t launch_backward(const void *x, const void *dy, int N, int HW, int C, int R, int k,
                            moce_dtype_t dt, moce_layout_t lay, const int32_t *pidx,
                            const float *plog, const int32_t *resid, int nU, const float *W1,
                            const float *b1, const float *w2, const float *b2, float tmin,
                            float tmax, float *dx, float *dlogit, float *dW1, float *db1,
                            float *dw2, float *db2, unsigned char *ws, cudaStream_t s) {
    const BwdLayout B = bwd_layout(N, HW, C, R, k);
    if (B.TP == 0) return cudaErrorNotSupported;
    const int layout = lay == MOCE_NHWC ? 0 : 1;
    cudaError_t err = cudaSuccess;
    auto F = [&](size_t off) { return reinterpret_cast<float *>(ws + off); };
    auto I = [&](size_t off) { return reinterpret_cast<int32_t *>(ws + off); };
    const int J = R * k;
    const size_t rows = (size_t)N * R;
    float *tmp = F(B.tmp);
    const float inv_k = 1.f / (float)k;
    // the inverse support index (channel -> its entries in increasing order)
    const int ich = inv_chunk(J), nb = (J + ich - 1) / ich;
    const size_t smem_inv = (size_t)C * 4;
    err = cudaFuncSetAttribute(bwd_inv_hist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)smem_inv);
    if (err != cudaSuccess) return err;
    err = cudaFuncSetAttribute(bwd_inv_place_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)smem_inv);
    if (err != cudaSuccess) return err;
    bwd_inv_hist_kernel<<<nb, 32, smem_inv, s>>>(pidx, J, C, ich, I(B.hist));
    bwd_inv_colscan_kernel<<<(C + 255) / 256, 256, 0, s>>>(I(B.hist), nb, C, I(B.cnt));
    bwd_inv_scan_kernel<<<1, 1024, 0, s>>>(I(B.cnt), C, I(B.ptr));
    bwd_inv_place_kernel<<<nb, 32, smem_inv, s>>>(pidx, J, C, ich, I(B.hist), I(B.ptr),
                                                  I(B.ent));
    // da and the pool (x read once)
    const bool fast = dt == MOCE_BF16 && lay == MOCE_NHWC && C % 8 == 0 &&
                      (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
    const int TPf = fast ? da_fast_tile(C, R) : 0;
    const int TP = TPf ? TPf : B.TP, tiles = (HW + TP - 1) / TP;
    const bool fast_dx = dt == MOCE_BF16 && lay == MOCE_NHWC &&
                         (size_t)(R + 1) * kDxFastTile * 2 <= 227 * 1024;
    const int HWp = (int)align_up((size_t)HW, 64);
    uint16_t *dyT = reinterpret_cast<uint16_t *>(ws + B.dyT);
    if (TPf || fast_dx)
        bwd_dy_transpose_kernel<<<dim3(HWp / 64, (R + 1 + 31) / 32, N), 256, 0, s>>>(
            (const uint16_t *)dy, HW, HWp, R + 1, dyT);
    if (TPf || fast_dx)
        bwd_tables_kernel<<<(J + 255) / 256, 256, 0, s>>>(I(B.ent), J, k, inv_k, TPf, kDxFastTile,
                                                          reinterpret_cast<int2 *>(ws + B.dtab),
                                                          I(B.doff));
    if (TPf) {
        err = cudaMemsetAsync(I(B.bins), 0, (size_t)(R + 1) * 4, s);
        if (err != cudaSuccess) return err;
        bwd_count_bins_kernel<<<(C + 255) / 256, 256, 0, s>>>(I(B.cnt), C, R, I(B.bins));
        bwd_bins_scan_kernel<<<1, 1024, 0, s>>>(I(B.bins), R);
        bwd_order_kernel<<<(C + 255) / 256, 256, 0, s>>>(I(B.cnt), C, R, I(B.bins), I(B.corder));
        const size_t smem = da_fast_smem(C, R, TPf);
        const unsigned grid = (unsigned)((size_t)N * tiles);
        auto run = [&](auto kern) {
            cudaError_t e2 = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  (int)smem);
            if (e2 != cudaSuccess) return e2;
            kern<<<grid, TPf == 64 ? 256 : 512, smem, s>>>((const uint16_t *)x, dyT, HW, HWp, C, R, tiles,
                                         I(B.corder), I(B.ptr),
                                         reinterpret_cast<const int2 *>(ws + B.dtab), J, F(B.part),
                                         F(B.psum));
            return cudaSuccess;
        };
        // small tiles (wide layers) run one CTA per SM: 16 warps hide the table loads better
        err = TPf == 64 ? run(bwd_da_nhwc_kernel<64, 256>)
              : TPf == 32 ? run(bwd_da_nhwc_kernel<32, 512>) : run(bwd_da_nhwc_kernel<16, 512>);
        if (err != cudaSuccess) return err;
    } else {
        const size_t smem_da = (size_t)(C + R) * (B.TP + 1) * 4;
        if (dt == MOCE_BF16) {
            err = cudaFuncSetAttribute(bwd_da_kernel<uint16_t>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_da);
            if (err != cudaSuccess) return err;
            bwd_da_kernel<uint16_t><<<(unsigned)((size_t)N * tiles), kBwdThreads, smem_da, s>>>(
                (const uint16_t *)x, (const uint16_t *)dy, layout, HW, C, R, k, TP, tiles, pidx,
                F(B.part), F(B.psum));
        } else {
            err = cudaFuncSetAttribute(bwd_da_kernel<float>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_da);
            if (err != cudaSuccess) return err;
            bwd_da_kernel<float><<<(unsigned)((size_t)N * tiles), kBwdThreads, smem_da, s>>>(
                (const float *)x, (const float *)dy, layout, HW, C, R, k, TP, tiles, pidx,
                F(B.part), F(B.psum));
        }
    }
    colsum(F(B.part), N, tiles, J, 1.f, F(B.da), tmp, s);
    float *z = F(B.z);
    colsum(F(B.psum), N, tiles, C, (float)HW, z, tmp, s);
    // the gate: u, hpre = W1 u + b1, the per-row backward, du = W1^T dh
    bwd_gather_kernel<<<(unsigned)((rows * k + 255) / 256), 256, 0, s>>>(z, C, R, k, pidx,
                                                                         rows * k, F(B.u));
    GemmArgs g{};
    g.A = F(B.u), g.a_m = k, g.a_k = 1;
    g.B = W1, g.b_k = 1, g.b_n = k;  // B(i, j) = W1[j][i]
    g.bias = b1, g.C = F(B.h), g.M = (int)rows, g.Nn = k, g.K = k, g.kchunk = k;
    sgemm(g, 1, s);
    bwd_gate_rows_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, s>>>(
        F(B.h), F(B.da), rows, R, k, plog, w2, b2, tmin, tmax, F(B.a), F(B.dlp), F(B.dg),
        F(B.dgr), F(B.dh));
    g = GemmArgs{};
    g.A = F(B.dh), g.a_m = k, g.a_k = 1;
    g.B = W1, g.b_k = k, g.b_n = 1;  // B(j, i) = W1[j][i]
    g.C = F(B.du), g.M = (int)rows, g.Nn = k, g.K = k, g.kchunk = k;
    sgemm(g, 1, s);
    // parameter gradients, summed over the rows (examples and experts) in a fixed order
    g = GemmArgs{};
    g.A = F(B.dh), g.a_m = 1, g.a_k = k;  // A(j, r) = dh[r][j]
    g.B = F(B.u), g.b_k = k, g.b_n = 1;   // B(r, i) = u[r][i]
    g.C = F(B.wpart), g.M = k, g.Nn = k, g.K = rows, g.kchunk = B.kchunk;
    sgemm(g, B.splits, s);
    colsum(F(B.wpart), 1, B.splits, k * k, 1.f, dW1, tmp, s);
    colsum(F(B.dh), 1, rows, k, 1.f, db1, tmp, s);
    colsum(F(B.dgr), 1, rows, k, 1.f, dw2, tmp, s);
    colsum(F(B.dg), 1, rows, 1, 1.f, db2, tmp, s);
    // dlogit[e][i] = sum over examples of ds / tau (rows n R + e)
    colsum(F(B.dlp), 1, N, J, 1.f, dlogit, tmp, s);
    // dz and dx
    uint8_t *inU = ws + B.inU;
    err = cudaMemsetAsync(inU, 0, (size_t)C, s);
    if (err != cudaSuccess) return err;
    if (nU > 0) bwd_set_resid_kernel<<<(nU + 255) / 256, 256, 0, s>>>(resid, nU, inU);
    bwd_dz_kernel<<<(unsigned)(((size_t)N * C + 255) / 256), 256, 0, s>>>(
        F(B.du), N, C, J, I(B.ptr), I(B.ent), F(B.dz));
    const float inv_nU = nU > 0 ? 1.f / (float)nU : 0.f;
    const int tab = dx_tab_bytes(J, C) <= kDxTabMax &&
                    dx_tab_off(R, kDxFastTile) + dx_tab_bytes(J, C) <= 227 * 1024 ? 1 : 0;
    const size_t smem_fx =
        tab ? dx_tab_off(R, kDxFastTile) + dx_tab_bytes(J, C) : (size_t)(R + 1) * kDxFastTile * 2;
    if (fast_dx) {
        bwd_gather_a_kernel<<<(unsigned)((rows * k + 255) / 256), 256, 0, s>>>(F(B.a), I(B.ent), N,
                                                                              J, F(B.am));
        const int tiles_x = (HW + kDxFastTile - 1) / kDxFastTile;
        err = cudaFuncSetAttribute(bwd_dx_nhwc_kernel<kDxFastTile>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_fx);
        if (err != cudaSuccess) return err;
        bwd_dx_nhwc_kernel<kDxFastTile><<<(unsigned)((size_t)N * tiles_x), 256, smem_fx, s>>>(
            dyT, HW, HWp, C, R, J, tiles_x, F(B.am), I(B.ptr), I(B.doff), inU, inv_nU, F(B.dz), dx,
            tab);
        return cudaGetLastError();
    }
    const int tiles_x = (HW + TPX - 1) / TPX;
    const size_t smem_x = (size_t)(R + 1) * (TPX + 1) * 4;
    if (dt == MOCE_BF16) {
        err = cudaFuncSetAttribute(bwd_dx_kernel<uint16_t>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_x);
        if (err != cudaSuccess) return err;
        bwd_dx_kernel<uint16_t><<<(unsigned)((size_t)N * tiles_x), kBwdThreads, smem_x, s>>>(
            (const uint16_t *)dy, layout, HW, C, R, k, tiles_x, F(B.a), I(B.ptr), I(B.ent), inU,
            inv_nU, F(B.dz), dx);
    } else {
        err = cudaFuncSetAttribute(bwd_dx_kernel<float>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_x);
        if (err != cudaSuccess) return err;
        bwd_dx_kernel<float><<<(unsigned)((size_t)N * tiles_x), kBwdThreads, smem_x, s>>>(
            (const float *)dy, layout, HW, C, R, k, tiles_x, F(B.a), I(B.ptr), I(B.ent), inU,
            inv_nU, F(B.dz), dx);
    }
    return cudaGetLastError();
}

}  // namespace moce
