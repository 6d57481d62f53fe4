// Host entry points of the C ABI declared in include/moce.h: argument
// validation, workspace layout and kernel selection. Every check happens on
// the host before anything is enqueued.
#include <math.h>

#include "moce_internal.cuh"

using namespace moce;

namespace {

constexpr int kMaxChannels = 65535;  // 16-bit support indices (Sec. 3.5)

bool shape_ok(int N, int H, int W, int C, int R, int k) {
    if (N < 0 || N > 65535 || H < 0 || W < 0) return false;  // N is a grid dimension
    if (C < 1 || C > kMaxChannels || R < 1 || k < 1 || k > C) return false;
    if ((long long)H * W > (1ll << 30)) return false;
    if ((long long)N * H * W * (C > R + 1 ? C : R + 1) > (1ll << 46)) return false;
    if ((long long)R * k > (1ll << 31) - 1) return false;
    return true;
}

bool dtype_ok(moce_dtype_t d) { return d == MOCE_F32 || d == MOCE_BF16; }
bool layout_ok(moce_layout_t l) { return l == MOCE_NHWC || l == MOCE_NCHW; }

bool tau_ok(float tmin, float tmax) {
    return isfinite(tmin) && isfinite(tmax) && tmin > 0.f && tmin <= tmax;
}

moce_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? MOCE_OK : MOCE_ERR_CUDA; }

size_t pack_ws_bytes(int C) { return (2 + (size_t)(C + 31) / 32) * 4; }

}  // namespace

namespace moce {
size_t gate_smem_bytes(int k);
}

extern "C" {

const char *moce_status_string(moce_status_t s) {
    switch (s) {
    case MOCE_OK: return "MOCE_OK";
    case MOCE_ERR_INVALID_VALUE: return "MOCE_ERR_INVALID_VALUE";
    case MOCE_ERR_BAD_SUPPORT: return "MOCE_ERR_BAD_SUPPORT";
    case MOCE_ERR_UNSUPPORTED: return "MOCE_ERR_UNSUPPORTED";
    case MOCE_ERR_CUDA: return "MOCE_ERR_CUDA";
    case MOCE_ERR_TIMEOUT: return "MOCE_ERR_TIMEOUT";
    }
    return "MOCE_ERR_UNKNOWN";
}

size_t moce_pack_workspace_bytes(int C_in, int C_out, int k) {
    if (!shape_ok(0, 0, 0, C_in, C_out, k)) return 0;
    return pack_ws_bytes(C_in);
}

moce_status_t moce_pack_supports(int C_in, int C_out, int k, const int32_t *support_idx,
                                 const float *support_logits, int32_t *packed_idx,
                                 float *packed_logits, int32_t *resid_idx, int32_t *n_resid_host,
                                 void *ws, size_t ws_bytes, moce_stream_t stream) {
    if (!shape_ok(0, 0, 0, C_in, C_out, k)) return MOCE_ERR_INVALID_VALUE;
    if (!support_idx || !support_logits || !packed_idx || !packed_logits || !resid_idx ||
        !n_resid_host || !ws)
        return MOCE_ERR_INVALID_VALUE;
    if (ws_bytes < pack_ws_bytes(C_in) || (reinterpret_cast<uintptr_t>(ws) & 3u))
        return MOCE_ERR_INVALID_VALUE;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    uint32_t *words = static_cast<uint32_t *>(ws);
    cudaError_t err = launch_pack(C_in, C_out, k, support_idx, support_logits, packed_idx,
                                  packed_logits, resid_idx, words, s);
    if (err != cudaSuccess) return MOCE_ERR_CUDA;
    uint32_t head[2] = {0u, 0u};
    err = cudaMemcpyAsync(head, words, sizeof(head), cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess) err = cudaStreamSynchronize(s);
    if (err != cudaSuccess) return MOCE_ERR_CUDA;
    if (head[0] != 0u) return MOCE_ERR_BAD_SUPPORT;
    *n_resid_host = (int32_t)head[1];
    return MOCE_OK;
}

size_t moce_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k) {
    if (!shape_ok(N, H, W, C_in, C_out, k)) return 0;
    return ws_layout(N, H * W, C_in, C_out, k).total;
}

moce_status_t moce_workspace_init(void *ws, size_t ws_bytes, moce_stream_t stream) {
    if (!ws) return MOCE_ERR_INVALID_VALUE;
    return cuda_status(cudaMemsetAsync(ws, 0, ws_bytes, reinterpret_cast<cudaStream_t>(stream)));
}

moce_status_t moce_workspace_offsets(int N, int H, int W, int C_in, int C_out, int k,
                                     size_t *z_offset, size_t *tau_offset) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !z_offset || !tau_offset)
        return MOCE_ERR_INVALID_VALUE;
    const WsLayout L = ws_layout(N, H * W, C_in, C_out, k);
    *z_offset = L.z;
    *tau_offset = L.tau;
    return MOCE_OK;
}

moce_status_t moce_pool(const void *x, int N, int H, int W, int C_in, moce_dtype_t dtype,
                        moce_layout_t layout, float *z, void *ws, size_t ws_bytes,
                        moce_stream_t stream) {
    if (!shape_ok(N, H, W, C_in, 1, 1) || !dtype_ok(dtype) || !layout_ok(layout))
        return MOCE_ERR_INVALID_VALUE;
    if (N > 0 && (H * W < 1 || !x || !z || !ws)) return MOCE_ERR_INVALID_VALUE;
    const WsLayout L = ws_layout(N, H * W, C_in, 1, 1);
    if (layout == MOCE_NHWC && ws_bytes < L.total) return MOCE_ERR_INVALID_VALUE;
    if (reinterpret_cast<uintptr_t>(ws) & 255u) return MOCE_ERR_INVALID_VALUE;
    return cuda_status(launch_pool(x, N, H * W, C_in, dtype, layout, z, L,
                                   static_cast<unsigned char *>(ws),
                                   reinterpret_cast<cudaStream_t>(stream)));
}

moce_status_t moce_gate(const float *z, int N, int C_in, int C_out, int k,
                        const int32_t *packed_idx, const float *packed_logits, const float *W1,
                        const float *b1, const float *w2, const float *b2, float tau_min,
                        float tau_max, float *tau, float *mix_w, moce_stream_t stream) {
    if (!shape_ok(N, 1, 1, C_in, C_out, k) || !tau_ok(tau_min, tau_max))
        return MOCE_ERR_INVALID_VALUE;
    if (N > 0 && (!z || !packed_idx || !packed_logits || !W1 || !b1 || !w2 || !b2 || !tau))
        return MOCE_ERR_INVALID_VALUE;
    if (gate_smem_bytes(k) > 227 * 1024) return MOCE_ERR_UNSUPPORTED;
    return cuda_status(launch_gate(z, N, C_in, C_out, k, packed_idx, packed_logits, W1, b1, w2, b2,
                                   tau_min, tau_max, tau, mix_w,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

// Which kernel path serves these arguments when the caller asks for `want`
// (MOCE_PATH_AUTO picks the fastest that supports them); MOCE_PATH_AUTO is
// returned when the requested path cannot run them.
static moce_path_t pick_path(const void *x, int N, int HW, int C_in, int C_out, int k,
                             moce_dtype_t dtype, moce_layout_t layout, moce_path_t want) {
    const bool vec = dtype == MOCE_BF16 && layout == MOCE_NHWC && C_in % 8 == 0 &&
                     (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
    const bool stream = vec && stream_supported(N, HW, C_in, C_out, k);
    switch (want) {
        case MOCE_PATH_AUTO: return stream ? MOCE_PATH_STREAM : MOCE_PATH_STEPS;
        case MOCE_PATH_STREAM: return stream ? want : MOCE_PATH_AUTO;
        case MOCE_PATH_STEPS: return want;
        default: break;
    }
    return MOCE_PATH_AUTO;
}

static bool path_ok(moce_path_t p) {
    return p == MOCE_PATH_AUTO || p == MOCE_PATH_STEPS || p == MOCE_PATH_STREAM;
}

moce_status_t moce_forward_path(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                moce_dtype_t dtype, moce_layout_t layout,
                                const int32_t *packed_idx, const float *packed_logits,
                                const int32_t *resid_idx, int n_resid, const float *W1,
                                const float *b1, const float *w2, const float *b2, float tau_min,
                                float tau_max, void *y, void *ws, size_t ws_bytes,
                                moce_path_t path, moce_stream_t stream) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !dtype_ok(dtype) || !layout_ok(layout) ||
        !tau_ok(tau_min, tau_max) || !path_ok(path))
        return MOCE_ERR_INVALID_VALUE;
    if (n_resid < 0 || n_resid > C_in || (n_resid > 0 && !resid_idx)) return MOCE_ERR_INVALID_VALUE;
    const int HW = H * W;
    if (N == 0 || HW == 0) return MOCE_OK;
    if (!x || !packed_idx || !packed_logits || !W1 || !b1 || !w2 || !b2 || !y || !ws)
        return MOCE_ERR_INVALID_VALUE;
    const WsLayout L = ws_layout(N, HW, C_in, C_out, k);
    if (ws_bytes < L.total || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MOCE_ERR_INVALID_VALUE;
    if (gate_smem_bytes(k) > 227 * 1024) return MOCE_ERR_UNSUPPORTED;
    const moce_path_t run = pick_path(x, N, HW, C_in, C_out, k, dtype, layout, path);
    if (run == MOCE_PATH_AUTO) return MOCE_ERR_UNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    unsigned char *wsb = static_cast<unsigned char *>(ws);
    const uint16_t *xv = static_cast<const uint16_t *>(x);
    uint16_t *yv = static_cast<uint16_t *>(y);
    if (run == MOCE_PATH_STREAM)
        return cuda_status(launch_stream(xv, N, HW, C_in, C_out, k, packed_idx, packed_logits,
                                         resid_idx, n_resid, W1, b1, w2, b2, tau_min, tau_max, yv,
                                         L, wsb, s));
    float *z = reinterpret_cast<float *>(wsb + L.z);
    float *tau = reinterpret_cast<float *>(wsb + L.tau);
    float *a = reinterpret_cast<float *>(wsb + L.a);
    cudaError_t err = launch_pool(x, N, HW, C_in, dtype, layout, z, L, wsb, s);
    if (err == cudaSuccess)
        err = launch_gate(z, N, C_in, C_out, k, packed_idx, packed_logits, W1, b1, w2, b2, tau_min,
                          tau_max, tau, a, s);
    if (err == cudaSuccess)
        err = launch_mix(x, N, HW, C_in, C_out, k, dtype, layout, packed_idx, a, resid_idx,
                         n_resid, y, reinterpret_cast<uint32_t *>(wsb + L.ctrl), s);
    return cuda_status(err);
}

moce_status_t moce_forward(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                           moce_dtype_t dtype, moce_layout_t layout, const int32_t *packed_idx,
                           const float *packed_logits, const int32_t *resid_idx, int n_resid,
                           const float *W1, const float *b1, const float *w2, const float *b2,
                           float tau_min, float tau_max, void *y, void *ws, size_t ws_bytes,
                           moce_stream_t stream) {
    return moce_forward_path(x, N, H, W, C_in, C_out, k, dtype, layout, packed_idx, packed_logits,
                             resid_idx, n_resid, W1, b1, w2, b2, tau_min, tau_max, y, ws, ws_bytes,
                             MOCE_PATH_AUTO, stream);
}

int moce_forward_launches(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                          moce_dtype_t dtype, moce_layout_t layout) {
    return moce_forward_path_launches(x, N, H, W, C_in, C_out, k, dtype, layout, MOCE_PATH_AUTO);
}

int moce_forward_path_launches(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                               moce_dtype_t dtype, moce_layout_t layout, moce_path_t path) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !dtype_ok(dtype) || !layout_ok(layout) ||
        !path_ok(path))
        return 0;
    if (N == 0 || H * W == 0) return 0;
    if (gate_smem_bytes(k) > 227 * 1024) return 0;
    switch (pick_path(x, N, H * W, C_in, C_out, k, dtype, layout, path)) {
        case MOCE_PATH_STREAM: return 1;
        case MOCE_PATH_STEPS:  // pool (one launch, or two with tile sums), gate, mix
            return pool_launches(x, N, H * W, C_in, dtype, layout) + 2;
        default: return 0;
    }
}

const char *moce_forward_kernel(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                moce_dtype_t dtype, moce_layout_t layout) {
    return moce_forward_path_kernel(x, N, H, W, C_in, C_out, k, dtype, layout, MOCE_PATH_AUTO);
}

const char *moce_forward_path_kernel(const void *x, int N, int H, int W, int C_in, int C_out,
                                     int k, moce_dtype_t dtype, moce_layout_t layout,
                                     moce_path_t path) {
    if (moce_forward_path_launches(x, N, H, W, C_in, C_out, k, dtype, layout, path) == 0)
        return nullptr;
    switch (pick_path(x, N, H * W, C_in, C_out, k, dtype, layout, path)) {
        case MOCE_PATH_STEPS: return "pool+gate+mix";
        case MOCE_PATH_STREAM: return "moce_stream_kernel";
        default: return nullptr;
    }
}

size_t moce_train_workspace_bytes(int C_in, int C_out) {
    if (!shape_ok(0, 0, 0, C_in, C_out, 1)) return 0;
    return train_ws_bytes(C_out, C_in);
}

moce_status_t moce_topk_supports(const float *logits, int C_in, int C_out, int k,
                                 int32_t *packed_idx, float *packed_logits, void *ws,
                                 size_t ws_bytes, moce_stream_t stream) {
    if (!shape_ok(0, 0, 0, C_in, C_out, k)) return MOCE_ERR_INVALID_VALUE;
    if (!logits || !packed_idx || !packed_logits || !ws) return MOCE_ERR_INVALID_VALUE;
    if (ws_bytes < train_ws_bytes(C_out, C_in) || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MOCE_ERR_INVALID_VALUE;
    if (topk_smem_bytes(C_in, k) > 227 * 1024) return MOCE_ERR_UNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    uint32_t *err_word = static_cast<uint32_t *>(ws);
    cudaError_t err = cudaMemsetAsync(err_word, 0, 4, s);
    if (err == cudaSuccess)
        err = launch_topk(logits, C_out, C_in, k, packed_idx, packed_logits, err_word, s);
    uint32_t flag = 0;
    if (err == cudaSuccess) err = cudaMemcpyAsync(&flag, err_word, 4, cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess) err = cudaStreamSynchronize(s);
    if (err != cudaSuccess) return MOCE_ERR_CUDA;
    return flag ? MOCE_ERR_BAD_SUPPORT : MOCE_OK;
}

moce_status_t moce_coverage_loss(const float *logits, int C_in, int C_out, float eps,
                                 float *loss, float *usage, float *grad, void *ws,
                                 size_t ws_bytes, moce_stream_t stream) {
    if (!shape_ok(0, 0, 0, C_in, C_out, 1) || !(eps >= 0.f) || !isfinite(eps))
        return MOCE_ERR_INVALID_VALUE;
    if (!logits || !loss || !ws) return MOCE_ERR_INVALID_VALUE;
    if (ws_bytes < train_ws_bytes(C_out, C_in) || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MOCE_ERR_INVALID_VALUE;
    return cuda_status(launch_coverage(logits, C_out, C_in, (double)eps, loss, usage, grad,
                                       static_cast<unsigned char *>(ws),
                                       reinterpret_cast<cudaStream_t>(stream)));
}

moce_status_t moce_mix(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                       moce_dtype_t dtype, moce_layout_t layout, const int32_t *sup_idx,
                       const float *mix_w, const int32_t *resid_idx, int n_resid,
                       const int32_t *n_resid_per_example, void *y, void *ws, size_t ws_bytes,
                       moce_stream_t stream) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !dtype_ok(dtype) || !layout_ok(layout))
        return MOCE_ERR_INVALID_VALUE;
    const bool per = n_resid_per_example != nullptr;
    if (!per && (n_resid < 0 || n_resid > C_in || (n_resid > 0 && !resid_idx)))
        return MOCE_ERR_INVALID_VALUE;
    if (N == 0 || H * W == 0) return MOCE_OK;
    if (!x || !sup_idx || !mix_w || !y || !ws || (per && !resid_idx)) return MOCE_ERR_INVALID_VALUE;
    const WsLayout L = ws_layout(N, H * W, C_in, C_out, k);
    if (ws_bytes < L.total || (reinterpret_cast<uintptr_t>(ws) & 255u)) return MOCE_ERR_INVALID_VALUE;
    PerExample pe;
    if (per) {
        pe.sup_stride = (size_t)C_out * k;
        pe.resid_stride = (size_t)C_in;
        pe.nUa = n_resid_per_example;
    }
    unsigned char *wsb = static_cast<unsigned char *>(ws);
    return cuda_status(launch_mix(x, N, H * W, C_in, C_out, k, dtype, layout, sup_idx, mix_w,
                                  resid_idx, per ? 0 : n_resid, y,
                                  reinterpret_cast<uint32_t *>(wsb + L.ctrl),
                                  reinterpret_cast<cudaStream_t>(stream), pe));
}

static bool dyn_shape_ok(int N, int H, int W, int C_in, int C_out, int k, int d) {
    return shape_ok(N, H, W, C_in, C_out, k) && d >= 1 && d <= 4096 &&
           (long long)N * C_out <= (1ll << 31) - 1 &&
           (long long)N * C_out * C_in <= (1ll << 40);
}

size_t moce_dynamic_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k, int d) {
    if (!dyn_shape_ok(N, H, W, C_in, C_out, k, d) || !dynamic_supported(C_in, k)) return 0;
    return dyn_layout(N, H * W, C_in, C_out, k, d).total;
}

moce_status_t moce_dynamic_supports(const float *z, int N, int C_in, int C_out, int k, int d,
                                    const float *logits, const float *Wh, const float *bh,
                                    const float *V, const float *Q, int32_t *sup_idx,
                                    float *sup_logits, int32_t *resid_idx, int32_t *n_resid,
                                    void *ws, size_t ws_bytes, moce_stream_t stream) {
    if (!dyn_shape_ok(N, 1, 1, C_in, C_out, k, d)) return MOCE_ERR_INVALID_VALUE;
    if (!dynamic_supported(C_in, k)) return MOCE_ERR_UNSUPPORTED;
    if (N == 0) return MOCE_OK;
    if (!z || !logits || !Wh || !bh || !V || !Q || !sup_idx || !sup_logits || !resid_idx ||
        !n_resid || !ws)
        return MOCE_ERR_INVALID_VALUE;
    const DynLayout D = dyn_layout(N, 1, C_in, C_out, k, d);
    if (ws_bytes < D.routing || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MOCE_ERR_INVALID_VALUE;
    unsigned char *wsb = static_cast<unsigned char *>(ws);
    return cuda_status(launch_dynamic_supports(
        z, N, C_in, C_out, k, d, logits, Wh, bh, V, Q, reinterpret_cast<float *>(wsb + D.h),
        reinterpret_cast<float *>(wsb + D.Ld), sup_idx, sup_logits, resid_idx, n_resid,
        reinterpret_cast<uint32_t *>(wsb + D.err), reinterpret_cast<cudaStream_t>(stream)));
}

// Gate and mix with per-example supports; z already pooled at L.z of wsf.
static cudaError_t run_with_supports(const void *x, int N, int HW, int C, int R, int k,
                                     moce_dtype_t dt, moce_layout_t lay, const int32_t *sidx,
                                     const float *slog, const int32_t *resid, const int32_t *nU,
                                     const float *W1, const float *b1, const float *w2,
                                     const float *b2, float tmin, float tmax, void *y,
                                     const WsLayout &L, unsigned char *wsf, cudaStream_t s) {
    float *z = reinterpret_cast<float *>(wsf + L.z);
    float *tau = reinterpret_cast<float *>(wsf + L.tau);
    float *a = reinterpret_cast<float *>(wsf + L.a);
    cudaError_t err = launch_gate(z, N, C, R, k, sidx, slog, W1, b1, w2, b2, tmin, tmax, tau, a, s,
                                  (size_t)R * k);
    if (err != cudaSuccess) return err;
    PerExample pe;
    pe.sup_stride = (size_t)R * k;
    pe.resid_stride = (size_t)C;
    pe.nUa = nU;
    return launch_mix(x, N, HW, C, R, k, dt, lay, sidx, a, resid, 0, y,
                      reinterpret_cast<uint32_t *>(wsf + L.ctrl), s, pe);
}

moce_status_t moce_forward_supports(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                    moce_dtype_t dtype, moce_layout_t layout,
                                    const int32_t *sup_idx, const float *sup_logits,
                                    const int32_t *resid_idx, const int32_t *n_resid,
                                    const float *W1, const float *b1, const float *w2,
                                    const float *b2, float tau_min, float tau_max, void *y,
                                    void *ws, size_t ws_bytes, moce_stream_t stream) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !dtype_ok(dtype) || !layout_ok(layout) ||
        !tau_ok(tau_min, tau_max))
        return MOCE_ERR_INVALID_VALUE;
    const int HW = H * W;
    if (N == 0 || HW == 0) return MOCE_OK;
    if (!x || !sup_idx || !sup_logits || !resid_idx || !n_resid || !W1 || !b1 || !w2 || !b2 ||
        !y || !ws)
        return MOCE_ERR_INVALID_VALUE;
    const WsLayout L = ws_layout(N, HW, C_in, C_out, k);
    if (ws_bytes < L.total || (reinterpret_cast<uintptr_t>(ws) & 255u)) return MOCE_ERR_INVALID_VALUE;
    if (gate_smem_bytes(k) > 227 * 1024) return MOCE_ERR_UNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    unsigned char *wsb = static_cast<unsigned char *>(ws);
    cudaError_t err = launch_pool(x, N, HW, C_in, dtype, layout,
                                  reinterpret_cast<float *>(wsb + L.z), L, wsb, s);
    if (err == cudaSuccess)
        err = run_with_supports(x, N, HW, C_in, C_out, k, dtype, layout, sup_idx, sup_logits,
                                resid_idx, n_resid, W1, b1, w2, b2, tau_min, tau_max, y, L, wsb, s);
    return cuda_status(err);
}

moce_status_t moce_forward_dynamic(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                   int d, moce_dtype_t dtype, moce_layout_t layout,
                                   const float *logits, const float *Wh, const float *bh,
                                   const float *V, const float *Q, const float *W1,
                                   const float *b1, const float *w2, const float *b2,
                                   float tau_min, float tau_max, void *y, int32_t *sup_idx,
                                   float *sup_logits, int32_t *n_resid, void *ws, size_t ws_bytes,
                                   moce_stream_t stream) {
    if (!dyn_shape_ok(N, H, W, C_in, C_out, k, d) || !dtype_ok(dtype) || !layout_ok(layout) ||
        !tau_ok(tau_min, tau_max))
        return MOCE_ERR_INVALID_VALUE;
    if (!dynamic_supported(C_in, k)) return MOCE_ERR_UNSUPPORTED;
    const int HW = H * W;
    if (N == 0 || HW == 0) return MOCE_OK;
    if (!x || !logits || !Wh || !bh || !V || !Q || !W1 || !b1 || !w2 || !b2 || !y || !ws)
        return MOCE_ERR_INVALID_VALUE;
    const DynLayout D = dyn_layout(N, HW, C_in, C_out, k, d);
    if (ws_bytes < D.total || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return MOCE_ERR_INVALID_VALUE;
    if (gate_smem_bytes(k) > 227 * 1024) return MOCE_ERR_UNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    unsigned char *wsb = static_cast<unsigned char *>(ws);
    unsigned char *wsf = wsb + D.fwd_off;
    const WsLayout &L = D.fwd;
    float *z = reinterpret_cast<float *>(wsf + L.z);
    int32_t *sidx = sup_idx ? sup_idx : reinterpret_cast<int32_t *>(wsb + D.sidx);
    float *slog = sup_logits ? sup_logits : reinterpret_cast<float *>(wsb + D.slog);
    int32_t *nU = n_resid ? n_resid : reinterpret_cast<int32_t *>(wsb + D.nU);
    int32_t *resid = reinterpret_cast<int32_t *>(wsb + D.resid);
    cudaError_t err = launch_pool(x, N, HW, C_in, dtype, layout, z, L, wsf, s);
    if (err == cudaSuccess)
        err = launch_dynamic_supports(z, N, C_in, C_out, k, d, logits, Wh, bh, V, Q,
                                      reinterpret_cast<float *>(wsb + D.h),
                                      reinterpret_cast<float *>(wsb + D.Ld), sidx, slog, resid, nU,
                                      reinterpret_cast<uint32_t *>(wsb + D.err), s);
    if (err == cudaSuccess)
        err = run_with_supports(x, N, HW, C_in, C_out, k, dtype, layout, sidx, slog, resid, nU, W1,
                                b1, w2, b2, tau_min, tau_max, y, L, wsf, s);
    return cuda_status(err);
}

size_t moce_backward_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k) {
    if (!shape_ok(N, H, W, C_in, C_out, k)) return 0;
    return backward_ws_bytes(N, H * W, C_in, C_out, k);
}

moce_status_t moce_backward(const void *x, const void *dy, int N, int H, int W, int C_in,
                            int C_out, int k, moce_dtype_t dtype, moce_layout_t layout,
                            const int32_t *packed_idx, const float *packed_logits,
                            const int32_t *resid_idx, int n_resid, const float *W1,
                            const float *b1, const float *w2, const float *b2, float tau_min,
                            float tau_max, float *dx, float *dlogits, float *dW1, float *db1,
                            float *dw2, float *db2, void *ws, size_t ws_bytes,
                            moce_stream_t stream) {
    if (!shape_ok(N, H, W, C_in, C_out, k) || !dtype_ok(dtype) || !layout_ok(layout) ||
        !tau_ok(tau_min, tau_max))
        return MOCE_ERR_INVALID_VALUE;
    if (n_resid < 0 || n_resid > C_in || (n_resid > 0 && !resid_idx)) return MOCE_ERR_INVALID_VALUE;
    if (!dlogits || !dW1 || !db1 || !dw2 || !db2) return MOCE_ERR_INVALID_VALUE;
    const size_t need = backward_ws_bytes(N, H * W, C_in, C_out, k);
    if (need == 0) return MOCE_ERR_UNSUPPORTED;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int HW = H * W;
    if (N == 0 || HW == 0) {
        cudaError_t err = cudaMemsetAsync(dlogits, 0, (size_t)C_out * k * 4, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(dW1, 0, (size_t)k * k * 4, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(db1, 0, (size_t)k * 4, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(dw2, 0, (size_t)k * 4, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(db2, 0, 4, s);
        return cuda_status(err);
    }
    if (!x || !dy || !dx || !packed_idx || !packed_logits || !W1 || !b1 || !w2 || !b2 || !ws)
        return MOCE_ERR_INVALID_VALUE;
    if (ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u)) return MOCE_ERR_INVALID_VALUE;
    const cudaError_t err = launch_backward(
        x, dy, N, HW, C_in, C_out, k, dtype, layout, packed_idx, packed_logits, resid_idx, n_resid,
        W1, b1, w2, b2, tau_min, tau_max, dx, dlogits, dW1, db1, dw2, db2,
        static_cast<unsigned char *>(ws), s);
    if (err == cudaErrorNotSupported) return MOCE_ERR_UNSUPPORTED;
    return cuda_status(err);
}

moce_status_t moce_check_device_error(const void *ws, size_t ws_bytes, moce_stream_t stream) {
    if (!ws || ws_bytes < kCtrlWords * 4) return MOCE_ERR_INVALID_VALUE;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    uint32_t words[kCtrlWords];
    cudaError_t err = cudaMemcpyAsync(words, ws, sizeof(words), cudaMemcpyDeviceToHost, s);
    if (err == cudaSuccess) err = cudaStreamSynchronize(s);
    if (err != cudaSuccess) return MOCE_ERR_CUDA;
    return words[kCtrlError] ? MOCE_ERR_TIMEOUT : MOCE_OK;
}

}  // extern "C"
