// Internal declarations of the MoCE CUDA library (sm_103a). Not part of the ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "moce.h"

namespace moce {

constexpr int kThreads = 256;  // threads of the step kernels

__host__ __device__ inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// ---------------------------------------------------------------- workspace
// Control words at the start of a forward workspace.
enum CtrlWord : int {
    kCtrlExitCounter = 0,  // CTAs that finished the stream kernel
    kCtrlEpoch = 1,        // number of completed stream forwards (data tags are epoch + 1)
    kCtrlError = 2,        // 0, or kErrTimeout
    kCtrlErrorItem = 3,    // 1 + the work item whose wait gave up
    kCtrlDropItem = 4,     // fault injection for tests: 1 + a work item that must not publish
    kCtrlWords = 64
};
constexpr uint32_t kErrTimeout = 1u;


// Pixels per pooling tile: about 32 KB of bf16 input per tile.
inline int pool_tile_px(int C) {
    int pp = 16384 / (C > 0 ? C : 1);
    int p2 = 4;
    while (p2 * 2 <= pp && p2 < 256) p2 *= 2;
    return p2;
}

// Positions per tile of the stream path (moce_stream.cu).
constexpr int kStreamTile = 64;

struct WsLayout {
    size_t ctrl = 0;      // kCtrlWords uint32
    size_t partial = 0;   // [N][pool_tiles][C] fp32 pooling tile sums (step kernels);
                          // [N][ceil(HW/64)][C] tagged 64-bit words {fp32 bits, epoch + 1}:
                          // tile sums beyond the fixed-point range (stream path)
    size_t z = 0;         // [N][C] fp32
    size_t tau = 0;       // [N][R] fp32
    size_t a = 0;         // [N][R][k] fp32 mixing weights (step kernels)
    size_t zacc = 0;      // [2][N][C] 64-bit channel accumulator words (stream path)
    size_t sync = 0;      // [2][N] uint32; [N + n]: the tag (epoch + 1) of the forward that
                          // produced example n's weights (stream path)
    size_t sblk = 0;      // [N] weight blocks of the stream path (stream_table_bytes(R) each)
    size_t total = 0;
    int pool_px = 0;
    int pool_tiles = 0;
};

// Bytes of one example's weight block on the stream path: 16 floats per
// expert plus 16 bytes per 8 experts (bank offset of the mixing groups).
inline size_t stream_table_bytes(int R) {
    return R <= 64 ? (size_t)64 * R + (size_t)16 * ((R + 7) / 8) : 0;
}

inline WsLayout ws_layout(int N, int HW, int C, int R, int k) {
    WsLayout L;
    L.pool_px = pool_tile_px(C);
    L.pool_tiles = (HW + L.pool_px - 1) / L.pool_px;
    const size_t stream_tiles = (size_t)(HW + kStreamTile - 1) / kStreamTile;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
    auto mx = [](size_t a, size_t b) { return a > b ? a : b; };
    L.ctrl = take(kCtrlWords * 4);
    L.partial = take((size_t)N * mx((size_t)L.pool_tiles * C * 4, stream_tiles * C * 8));
    L.z = take((size_t)N * C * 4);
    L.tau = take((size_t)N * R * 4);
    L.a = take((size_t)N * R * k * 4);
    L.zacc = take((size_t)2 * N * C * 8);
    L.sync = take((size_t)N * 8);
    L.sblk = take((size_t)N * stream_table_bytes(R));
    L.total = off;
    return L;
}

// ---------------------------------------------------------------- device helpers
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint16_t f32_to_bf16(float f) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

template <typename T> __device__ __forceinline__ float load_elem(const T *p);
template <> __device__ __forceinline__ float load_elem<float>(const float *p) { return __ldg(p); }
template <> __device__ __forceinline__ float load_elem<uint16_t>(const uint16_t *p) {
    return bf16_to_f32(__ldg(p));
}
template <typename T> __device__ __forceinline__ T store_cvt(float v);
template <> __device__ __forceinline__ float store_cvt<float>(float v) { return v; }
template <> __device__ __forceinline__ uint16_t store_cvt<uint16_t>(float v) { return f32_to_bf16(v); }

// ---------------------------------------------------------------- tiled mix geometry
// The NHWC bf16 mixing kernels stage a tile of TP = 8*GS pixels of one
// example in shared memory, transposed to channel-major rows of TP bf16
// (pixel pairs packed in 32-bit words); groups of GS lanes each own 8 pixels
// per lane and mix whole experts (or 1/S of an expert).
struct MixGeom {
    int GS = 0, TP = 0, G = 0;  // lanes per group, pixels per tile, groups per CTA
    int EB = 0;                 // experts per table chunk
    int S = 1;                  // parts each expert's k entries are split into
    int kp = 0;                 // k rounded up to even (entries per expert in the table)
    int kq = 0;                 // entries per part (even)
    size_t off_ys = 0, off_rp = 0, off_pp = 0, off_tab = 0, smem = 0;
};

bool mix_geometry(int C, int R, int k, size_t smem_budget, MixGeom *g);

// Per-example supports of the mixing kernels: example n reads its supports
// at pidx + n sup_stride, its U at resid + n resid_stride and |U| at nUa[n]
// (a device array; when nUa is null every example has the scalar nU).
struct PerExample {
    size_t sup_stride = 0, resid_stride = 0;
    const int32_t *nUa = nullptr;
    // |U| of example n, held to [0, C]: a row of U has C entries, so a count
    // outside that range (not one moce_dynamic_supports writes) reads no
    // further than the row
    __device__ __forceinline__ int count(int n, int nU, int C) const {
        return nUa ? min(max(nUa[n], 0), C) : nU;
    }
};

// ---------------------------------------------------------------- launchers (host)
cudaError_t launch_pack(int C, int R, int k, const int32_t *idx, const float *lg, int32_t *pidx,
                        float *plog, int32_t *resid, uint32_t *ws_words, cudaStream_t s);

// Tiling of the NHWC pool (moce_pool.cu): vec channels per load, CB vectors
// per CTA column block (chunks blocks), PT positions per span, spans spans per
// example (1: z written directly; more: tile sums plus pool_finalize_kernel).
struct PoolPlan {
    int vec = 1, CB = 1, PT = 1, spans = 1;
    unsigned chunks = 1;
};
PoolPlan pool_plan(const void *x, int N, int HW, int C, moce_dtype_t dt);
// kernel launches of launch_pool for these arguments
int pool_launches(const void *x, int N, int HW, int C, moce_dtype_t dt, moce_layout_t lay);
cudaError_t launch_pool(const void *x, int N, int HW, int C, moce_dtype_t dt, moce_layout_t lay,
                        float *z, const WsLayout &L, unsigned char *ws, cudaStream_t s);

// sup_stride: elements between two examples' supports in pidx / plog (0:
// every example shares one set of supports).
cudaError_t launch_gate(const float *z, int N, int C, int R, int k, const int32_t *pidx,
                        const float *plog, const float *W1, const float *b1, const float *w2,
                        const float *b2, float tmin, float tmax, float *tau, float *a,
                        cudaStream_t s, size_t sup_stride = 0);

// ctrl: the workspace control words (bounded waits report MOCE_ERR_TIMEOUT there).
cudaError_t launch_mix(const void *x, int N, int HW, int C, int R, int k, moce_dtype_t dt,
                       moce_layout_t lay, const int32_t *pidx, const float *a,
                       const int32_t *resid, int nU, void *y, uint32_t *ctrl, cudaStream_t s,
                       const PerExample &pe = PerExample());

// Mixing kernel for wide layers (moce_mix_wide.cu): NHWC bf16, C % 8 == 0,
// x 16-byte aligned.
bool mix_wide_supported(int HW, int C, int R, int k, int nU);
cudaError_t launch_mix_wide(const uint16_t *x, int N, int HW, int C, int R, int k,
                            const int32_t *pidx, const float *a, const int32_t *resid, int nU,
                            uint16_t *y, uint32_t *ctrl, cudaStream_t s, const PerExample &pe);

// Support maintenance (moce_train.cu): TopK over full routing rows and the
// coverage regularizer.
// Shared memory of one TopK row (the k selected pairs padded to a power of
// two, and the row's order keys).
size_t topk_smem_bytes(int C, int k);
size_t train_ws_bytes(int R, int C);
cudaError_t launch_topk(const float *L, int R, int C, int k, int32_t *idx, float *lg,
                        uint32_t *err, cudaStream_t s);
cudaError_t launch_coverage(const float *L, int R, int C, double eps, float *loss, float *u,
                            float *grad, unsigned char *ws, cudaStream_t s);

// Backward with static supports (moce_backward.cu); 0 / cudaErrorNotSupported
// when a staged tile does not fit.
size_t backward_ws_bytes(int N, int HW, int C, int R, int k);
cudaError_t launch_backward(const void *x, const void *dy, int N, int HW, int C, int R, int k,
                            moce_dtype_t dt, moce_layout_t lay, const int32_t *pidx,
                            const float *plog, const int32_t *resid, int nU, const float *W1,
                            const float *b1, const float *w2, const float *b2, float tmin,
                            float tmax, float *dx, float *dlogit, float *dW1, float *db1,
                            float *dw2, float *db2, unsigned char *ws, cudaStream_t s);

// Input-conditioned supports (moce_dynamic.cu). Workspace: the routing
// buffers first (their offsets depend on N, C, R, k, d only), then a forward
// workspace (ws_layout) at fwd_off.
struct DynLayout {
    size_t err = 0, h = 0, Ld = 0, sidx = 0, slog = 0, resid = 0, nU = 0;
    size_t routing = 0;  // bytes of the routing buffers
    size_t fwd_off = 0;
    WsLayout fwd;
    size_t total = 0;
};
DynLayout dyn_layout(int N, int HW, int C, int R, int k, int d);
bool dynamic_supported(int C, int k);
// From pooled descriptors z [N][C]: h [N][d], the logits Ld [N][R][C], the
// per-example supports sidx / slog [N][R][k] (deployment order), U(X) in
// resid [N][C] (ascending) and |U(X)| in nU [N]. err: TopK's non-finite flag.
cudaError_t launch_dynamic_supports(const float *z, int N, int C, int R, int k, int d,
                                    const float *L, const float *Wh, const float *bh,
                                    const float *V, const float *Q, float *h, float *Ld,
                                    int32_t *sidx, float *slog, int32_t *resid, int32_t *nU,
                                    uint32_t *err, cudaStream_t s);

cudaError_t launch_stream(const uint16_t *x, int N, int HW, int C, int R, int k,
                          const int32_t *pidx, const float *plog, const int32_t *resid, int nU,
                          const float *W1, const float *b1, const float *w2, const float *b2,
                          float tmin, float tmax, uint16_t *y, const WsLayout &L,
                          unsigned char *ws, cudaStream_t s);

bool stream_supported(int N, int HW, int C, int R, int k);

}  // namespace moce
