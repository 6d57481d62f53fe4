/*
 * moce.h - C ABI of the MoCE layer (forward, backward, support maintenance)
 * on NVIDIA GB300 (sm_103a).
 *
 * A Mixture of Channel Experts layer ("Mixture of Channel Experts: Static
 * Sparse Supports with Input-Adaptive Mixing for Pointwise Projections",
 * Sec. 3) replaces a dense 1x1 projection C_in -> C_out + 1. Each of the
 * C_out routed experts mixes k channels of a static support with
 * softmax weights whose temperature is predicted per example from the pooled
 * descriptors of that support; one residual expert averages the channels no
 * routed expert selects.
 *
 *   z        = GAP(x)                                            Sec. 3.3
 *   tau[n,e] = tau_min + (tau_max - tau_min) * sigma(g(z[n, S_e]))  Eq. (tau)
 *              g(u) = w2 . ReLU(W1 u + b1) + b2, u in descending-logit order
 *              (Sec. 3.3 ordering rule; gate shape of Sec. 4.1)
 *   a[n,e,i] = softmax_i(L[e,i] / tau[n,e])                     Eq. (weights)
 *   y[n,p,e] = sum_i a[n,e,i] x[n,p,S_e[i]]        e < C_out    Eq. (expert)
 *   y[n,p,C_out] = mean_{c in U} x[n,p,c], 0 if U is empty      Eq. (res)
 *
 * Conventions shared by every entry point:
 *   - All tensor pointers are DEVICE pointers unless the name ends in _host.
 *     The caller owns every buffer; the library never allocates memory and
 *     keeps no global state, with one exception: moce_forward_noalloc uses a
 *     fixed scratch array in the library's device image (see there).
 *   - Calls are asynchronous on `stream` unless stated otherwise. A NULL
 *     stream is the legacy default stream.
 *   - Arguments are validated on the host before any launch; an invalid
 *     argument returns MOCE_ERR_INVALID_VALUE and enqueues nothing. A failed
 *     launch returns MOCE_ERR_CUDA. No call traps or asserts on the device.
 *   - Shapes: N examples (0..65535), H x W positions, C_in input channels (1..65535, the
 *     16-bit index range of the deployment format, Sec. 3.5), C_out routed
 *     experts (>= 1), support size k (1..C_in).
 *   - x layout MOCE_NHWC: x[((n*H + h)*W + w)*C_in + c]; MOCE_NCHW:
 *     x[((n*C_in + c)*H + h)*W + w]. y has C_out + 1 channels in the same
 *     layout and dtype as x, the residual expert at channel C_out.
 *   - dtype MOCE_BF16 stores bfloat16 bit patterns; all arithmetic is fp32 and
 *     outputs are rounded to nearest even.
 */
#ifndef MOCE_H
#define MOCE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum moce_status {
    MOCE_OK = 0,
    MOCE_ERR_INVALID_VALUE = 1, /* bad shape, null pointer, misaligned buffer, small workspace */
    MOCE_ERR_BAD_SUPPORT = 2,   /* support index out of range / repeated in a row, or non-finite logit */
    MOCE_ERR_UNSUPPORTED = 3,   /* valid arguments this build has no kernel for */
    MOCE_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed */
    MOCE_ERR_TIMEOUT = 5        /* a bounded device-side wait ran out (see moce_check_device_error) */
} moce_status_t;

typedef enum moce_dtype { MOCE_F32 = 0, MOCE_BF16 = 1 } moce_dtype_t;
typedef enum moce_layout { MOCE_NHWC = 0, MOCE_NCHW = 1 } moce_layout_t;

/*
 * Kernel path of one layer forward (moce_forward_path). Both paths compute
 * the same layer (Sec. 3.2-3.4) and give the same results within bf16 output
 * rounding; they differ in how x travels through the GPU.
 *   MOCE_PATH_AUTO      STREAM when it supports the arguments, else STEPS
 *   MOCE_PATH_STEPS     one kernel per step: pool, gate, mix (any layout and
 *                       dtype); x is read twice
 *   MOCE_PATH_STREAM    one cooperative kernel that reads x from HBM once: a
 *                       pool stream reads each tile a few items ahead of a
 *                       mix stream, which reads it again from L2 once its
 *                       example's gate (run by a few dedicated CTAs) has
 *                       published the weights (NHWC bf16, 64 <= C_in <= 256,
 *                       C_in % 64 == 0, C_out <= 64, k <= 16, x 16-byte
 *                       aligned)
 * The values 1, 2, 3 and 5 belonged to kernels this library no longer has;
 * asking for them returns MOCE_ERR_INVALID_VALUE.
 */
typedef enum moce_path {
    MOCE_PATH_AUTO = 0,
    MOCE_PATH_STEPS = 4,
    MOCE_PATH_STREAM = 6
} moce_path_t;

/* Same type as cudaStream_t, declared here so that this header needs no CUDA header. */
typedef struct CUstream_st *moce_stream_t;

/* Human-readable name of a status code (static string, never NULL). */
const char *moce_status_string(moce_status_t status);

/*
 * Bytes of device workspace moce_pack_supports needs (coverage bitmap, error
 * word, |U| counter). Returns 0 for invalid shapes.
 */
size_t moce_pack_workspace_bytes(int C_in, int C_out, int k);

/*
 * Deployment packing of static supports (Sec. 3.2: supports are fixed at
 * inference; Sec. 3.5 "Storage": deployment keeps the selected logits and
 * their indices; Sec. 3.3: the gate input is ordered by descending routing
 * logit; Sec. 3.4: U = channels no expert selects).
 *
 *   support_idx     [C_out*k] int32, row e = the k channels of expert e, any order
 *   support_logits  [C_out*k] fp32, the routing logit of each selected channel
 *   packed_idx      [C_out*k] int32 out: each row sorted by logit descending,
 *                   equal logits by ascending channel (-0.0 equals +0.0)
 *   packed_logits   [C_out*k] fp32 out: the logits in the same order
 *   resid_idx       [C_in] int32 out: U in ascending order, first *n_resid_host valid
 *   n_resid_host    HOST int32 out: |U|
 *   ws, ws_bytes    device workspace, >= moce_pack_workspace_bytes(C_in, C_out, k),
 *                   no alignment beyond 4 bytes, contents need not be initialised
 *
 * SYNCHRONOUS: returns after the result is complete (it synchronises
 * `stream`). Rejects an index outside [0, C_in), an index repeated within one
 * expert, or a NaN/Inf logit with MOCE_ERR_BAD_SUPPORT; outputs are then
 * unspecified. Inputs and outputs must not overlap. Output is bit-exact and
 * independent of the input row order.
 */
moce_status_t moce_pack_supports(int C_in, int C_out, int k, const int32_t *support_idx,
                                 const float *support_logits, int32_t *packed_idx,
                                 float *packed_logits, int32_t *resid_idx, int32_t *n_resid_host,
                                 void *ws, size_t ws_bytes, moce_stream_t stream);

/*
 * Bytes of device workspace that moce_pool and moce_forward need for a layer
 * of this shape (pooling partials, z, tau, mixing weights, scheduler
 * control words). Returns 0 for invalid shapes.
 */
size_t moce_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k);

/*
 * Zero-fill a workspace (cudaMemsetAsync on `stream`). moce_forward requires
 * a workspace that was zero-filled before its first use (this call, or any
 * zero fill); each forward leaves its scheduler words ready for the next one.
 * Call it again after a forward reported MOCE_ERR_TIMEOUT.
 */
moce_status_t moce_workspace_init(void *ws, size_t ws_bytes, moce_stream_t stream);

/*
 * Byte offsets inside the forward workspace where the last moce_forward left
 * z [N*C_in] fp32 and tau [N*C_out] fp32 (for inspection and tests).
 */
moce_status_t moce_workspace_offsets(int N, int H, int W, int C_in, int C_out, int k,
                                     size_t *z_offset, size_t *tau_offset);

/*
 * Global average pooling (Sec. 3.3): z[n*C_in + c] = mean over the H*W
 * positions of x[n, :, :, c], fp32 accumulation in a fixed order
 * (deterministic). x: device, layout/dtype as given; NHWC with bf16 needs
 * C_in % 8 == 0 and a 16-byte aligned x for the vector path, otherwise a
 * scalar path runs. z: device fp32 [N*C_in]. ws >= moce_workspace_bytes.
 * H*W must be >= 1.
 */
moce_status_t moce_pool(const void *x, int N, int H, int W, int C_in, moce_dtype_t dtype,
                        moce_layout_t layout, float *z, void *ws, size_t ws_bytes,
                        moce_stream_t stream);

/*
 * Temperature gate and mixing weights (Eq. (tau), Eq. (weights); gate shape
 * of Sec. 4.1).
 *   z               [N*C_in] fp32 pooled descriptors
 *   packed_idx      [C_out*k] int32, packed_logits [C_out*k] fp32: from
 *                   moce_pack_supports (position 0 holds the largest logit)
 *   W1 [k*k] fp32 row-major, W1[j*k + i] = weight from gate input i to hidden
 *   unit j; b1 [k]; w2 [k]; b2 [1]: all device fp32
 *   tau_min <= tau_max, tau_min > 0, both finite
 *   tau             [N*C_out] fp32 out
 *   mix_w           [N*C_out*k] fp32 out, or NULL to skip the weights
 */
moce_status_t moce_gate(const float *z, int N, int C_in, int C_out, int k,
                        const int32_t *packed_idx, const float *packed_logits, const float *W1,
                        const float *b1, const float *w2, const float *b2, float tau_min,
                        float tau_max, float *tau, float *mix_w, moce_stream_t stream);

/*
 * The whole layer forward (Sec. 3.3-3.4): pooling, gate, weights, routed
 * mixing and residual, y with C_out + 1 channels in x's layout and dtype.
 *   packed_idx/packed_logits/resid_idx/n_resid: from moce_pack_supports
 *   (0 <= n_resid <= C_in; resid_idx may be NULL when n_resid == 0)
 *   gate parameters and tau bounds as in moce_gate
 *   y: device, must not overlap x
 *   ws, ws_bytes: >= moce_workspace_bytes(N, H, W, C_in, C_out, k), 256-byte
 *   aligned, zero-filled before its first use (moce_workspace_init); one
 *   workspace serves one stream at a time.
 * NHWC bf16 with 16-byte aligned x runs the stream kernel where it fits
 * (64 <= C_in <= 256, C_in % 64 == 0, C_out <= 64, k <= 16), else one kernel
 * per step (the choice is moce_forward_path's MOCE_PATH_AUTO).
 * Asynchronous; device-side failures (a bounded wait that ran out) are
 * reported by moce_check_device_error.
 */
moce_status_t moce_forward(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                           moce_dtype_t dtype, moce_layout_t layout, const int32_t *packed_idx,
                           const float *packed_logits, const int32_t *resid_idx, int n_resid,
                           const float *W1, const float *b1, const float *w2, const float *b2,
                           float tau_min, float tau_max, void *y, void *ws, size_t ws_bytes,
                           moce_stream_t stream);

/*
 * moce_forward on a chosen kernel path (moce_path_t). Same arguments,
 * ownership and results as moce_forward; `path` outside the enum is
 * MOCE_ERR_INVALID_VALUE, and a path that cannot run these arguments
 * (dtype, layout, C_in, C_out, k, alignment of x) is MOCE_ERR_UNSUPPORTED,
 * returned before anything is enqueued. For comparing and testing the paths.
 */
moce_status_t moce_forward_path(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                moce_dtype_t dtype, moce_layout_t layout,
                                const int32_t *packed_idx, const float *packed_logits,
                                const int32_t *resid_idx, int n_resid, const float *W1,
                                const float *b1, const float *w2, const float *b2, float tau_min,
                                float tau_max, void *y, void *ws, size_t ws_bytes,
                                moce_path_t path, moce_stream_t stream);

/*
 * The layer forward for callers that cannot allocate device memory: code
 * running inside an allocator or memory-pool callback, loops that forbid
 * allocation after start-up, plugins whose host framework owns every device
 * buffer. The paper has no counterpart; it is a deployment convenience.
 *
 * Same arguments and results as moce_forward, without the workspace: the
 * scratch is a fixed 8 MiB array in this library's device image (every GPU
 * that loads the library holds it until the process exits). A layer whose
 * moce_workspace_bytes exceeds 8 MiB is rejected with MOCE_ERR_UNSUPPORTED
 * before anything is enqueued. The call itself allocates nothing.
 *   - The first call on a device looks up the array's device address (once
 *     per device, with that device current); make that first call before any
 *     stream capture.
 *   - Every call shares the one array per device: each call clears the part
 *     it uses on `stream`, then runs the forward. Calls whose work overlaps on
 *     the GPU (other streams, other host threads) race on the array.
 *   - Device-side failures (a bounded wait that ran out) are reported by
 *     moce_noalloc_check_device_error, not by the return value.
 */
moce_status_t moce_forward_noalloc(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                   moce_dtype_t dtype, moce_layout_t layout,
                                   const int32_t *packed_idx, const float *packed_logits,
                                   const int32_t *resid_idx, int n_resid, const float *W1,
                                   const float *b1, const float *w2, const float *b2,
                                   float tau_min, float tau_max, void *y, moce_stream_t stream);

/*
 * Routed mix and residual expert alone, Eq. (expert) and Eq. (res), from
 * precomputed weights mix_w [N][C_out][k] (moce_gate's output).
 *   n_resid_per_example == NULL: shared supports, sup_idx [C_out][k] and
 *     resid_idx [C_in] with n_resid entries (as moce_forward);
 *   otherwise per-example supports, sup_idx [N][C_out][k], resid_idx
 *     [N][C_in] and n_resid_per_example [N] (device), as written by
 *     moce_dynamic_supports; n_resid is ignored. A count outside [0, C_in]
 *     is held to that range (the device cannot report it), so a row of
 *     resid_idx is never read past its C_in entries.
 * ws: a forward workspace (moce_workspace_bytes). Asynchronous.
 */
moce_status_t moce_mix(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                       moce_dtype_t dtype, moce_layout_t layout, const int32_t *sup_idx,
                       const float *mix_w, const int32_t *resid_idx, int n_resid,
                       const int32_t *n_resid_per_example, void *y, void *ws, size_t ws_bytes,
                       moce_stream_t stream);

/*
 * Input-conditioned supports, Eq. (dynamic) (the variant of Sec. 5; the
 * inference path: deterministic hard per-example TopK, no noise). A router
 * reads the whole pooled descriptor z = GAP(X) and adds a rank-d offset to
 * the static routing matrix; each example then selects its own supports:
 *   h(z)      = ReLU(W_h z + b_h)                          in R^d
 *   L_e(X)_c  = L_{e,c} + sum_j q_{e,j} h_j v_{c,j}        every e, c
 *   S_e(X)    = TopK(L_e(X), k), in deployment order (descending L_e(X),
 *               equal values by ascending channel), decided in fp32
 *   U(X)      = the channels no S_e(X) selects, ascending
 * and the layer of moce_forward runs with these supports: the gate reads z
 * at S_e(X) (Sec. 3.3 ordering) and the weights use the selected L_e(X)
 * values in place of L_{e,i} (Eq. (weights)).
 *   logits  device fp32 [C_out][C_in]: the static routing matrix L
 *   Wh      device fp32 [d][C_in] (row j = router unit j), bh [d]
 *   V       device fp32 [C_in][d] (row c = channel embedding v_c)
 *   Q       device fp32 [C_out][d] (row e = expert embedding q_e)
 * (2 C_in d + d + C_out d router parameters, as the paper counts them.)
 * 4 C_in + 8 k' <= 227 KB, k' = k rounded up to a power of two (TopK keeps a
 * row in shared memory: about 57,000 channels), 1 <= d <= 4096.
 * Non-finite logits give unspecified (but in-range) supports.
 *
 * moce_dynamic_workspace_bytes: device workspace of the dynamic calls
 * (256-byte aligned, no initialisation needed); 0 for unsupported shapes.
 * Its routing buffers come first and do not depend on H and W, so
 * moce_dynamic_supports accepts the workspace of any H, W.
 *
 * moce_dynamic_supports: from pooled descriptors z [N][C_in] (moce_pool)
 * to the per-example supports sup_idx / sup_logits [N][C_out][k], U(X) in
 * resid_idx [N][C_in] (the first n_resid[n] entries of row n) and
 * n_resid [N] (all device, int32 / fp32). Asynchronous.
 *
 * moce_forward_supports: the layer with given per-example supports (as
 * moce_dynamic_supports writes them): pool, gate and mix; n_resid counts
 * are held to [0, C_in] as in moce_mix. ws: a forward workspace
 * (moce_workspace_bytes). Asynchronous.
 *
 * moce_forward_dynamic: the whole variant: pool, router, TopK, U(X), gate and
 * mix. sup_idx, sup_logits, n_resid: optional device outputs (NULL: kept in
 * the workspace). Asynchronous.
 */
size_t moce_dynamic_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k, int d);
moce_status_t moce_dynamic_supports(const float *z, int N, int C_in, int C_out, int k, int d,
                                    const float *logits, const float *Wh, const float *bh,
                                    const float *V, const float *Q, int32_t *sup_idx,
                                    float *sup_logits, int32_t *resid_idx, int32_t *n_resid,
                                    void *ws, size_t ws_bytes, moce_stream_t stream);
moce_status_t moce_forward_supports(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                    moce_dtype_t dtype, moce_layout_t layout,
                                    const int32_t *sup_idx, const float *sup_logits,
                                    const int32_t *resid_idx, const int32_t *n_resid,
                                    const float *W1, const float *b1, const float *w2,
                                    const float *b2, float tau_min, float tau_max, void *y,
                                    void *ws, size_t ws_bytes, moce_stream_t stream);
moce_status_t moce_forward_dynamic(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                   int d, moce_dtype_t dtype, moce_layout_t layout,
                                   const float *logits, const float *Wh, const float *bh,
                                   const float *V, const float *Q, const float *W1,
                                   const float *b1, const float *w2, const float *b2,
                                   float tau_min, float tau_max, void *y, int32_t *sup_idx,
                                   float *sup_logits, int32_t *n_resid, void *ws, size_t ws_bytes,
                                   moce_stream_t stream);

/*
 * SYNCHRONOUS: waits for `stream`, then reads the device error word that the
 * last moce_forward_noalloc on the current device left in the scratch array.
 * MOCE_OK, MOCE_ERR_TIMEOUT (a bounded wait of that forward gave up; its y is
 * invalid) or MOCE_ERR_CUDA. Each moce_forward_noalloc clears the word, so
 * check before the next call on the device.
 */
moce_status_t moce_noalloc_check_device_error(moce_stream_t stream);

/*
 * Number of kernel launches moce_forward makes for these arguments (the
 * path selection depends on dtype, layout, C_in and the alignment of x).
 * Returns 0 for arguments moce_forward would reject. Enqueues nothing.
 */
int moce_forward_launches(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                          moce_dtype_t dtype, moce_layout_t layout);

/*
 * Name of the kernel path moce_forward takes for these arguments:
 * "moce_stream_kernel" (one cooperative kernel) or "pool+gate+mix" (one
 * kernel per step). NULL for arguments moce_forward would reject. Enqueues
 * nothing; the string is static.
 */
const char *moce_forward_kernel(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                                moce_dtype_t dtype, moce_layout_t layout);

/*
 * moce_forward_launches and moce_forward_kernel for moce_forward_path with
 * `path`: 0 / NULL where that path cannot run the arguments.
 */
int moce_forward_path_launches(const void *x, int N, int H, int W, int C_in, int C_out, int k,
                               moce_dtype_t dtype, moce_layout_t layout, moce_path_t path);
const char *moce_forward_path_kernel(const void *x, int N, int H, int W, int C_in, int C_out,
                                     int k, moce_dtype_t dtype, moce_layout_t layout,
                                     moce_path_t path);

/*
 * Support maintenance on the full routing matrix (training side; the forward
 * uses packed, fixed supports). logits: device fp32 [C_out][C_in], row e =
 * L_e, the routing preferences of routed expert e over every input channel.
 *
 * Bytes of device workspace moce_topk_supports and moce_coverage_loss need
 * (256-byte aligned; contents need no initialisation). 0 for invalid shapes.
 */
size_t moce_train_workspace_bytes(int C_in, int C_out);

/*
 * Eq. (support), Sec. 3.2: S_e = TopK(L_e, k) for every routed expert,
 * written directly in deployment order (descending logit, equal logits by
 * ascending channel, -0.0 equal to +0.0), i.e. as moce_pack_supports would
 * order them:
 *   packed_idx    device int32 [C_out][k] out: the selected channels
 *   packed_logits device fp32 [C_out][k] out: their logits
 * SYNCHRONOUS (it validates): a non-finite logit returns
 * MOCE_ERR_BAD_SUPPORT (outputs then unspecified). Needs 4 C_in + 8 k' <=
 * 227 KB, k' = k rounded up to a power of two (MOCE_ERR_UNSUPPORTED beyond:
 * one CTA keeps a row's order keys in shared memory, selects the k-th by
 * radix passes and sorts the k selected).
 */
moce_status_t moce_topk_supports(const float *logits, int C_in, int C_out, int k,
                                 int32_t *packed_idx, float *packed_logits, void *ws,
                                 size_t ws_bytes, moce_stream_t stream);

/*
 * The coverage regularizer of Sec. 3.4 over the full routing matrix:
 *   p_{e,c} = softmax(L_e)_c over all C_in channels, u_c = (1/C_out) sum_e p_{e,c},
 *   ubar = (1/C_in) sum_c u_c, L_cov = sum_c (u_c - ubar)^2 / (ubar^2 + eps).
 *   loss  device fp32 [1] out: L_cov
 *   usage device fp32 [C_in] out: u, or NULL
 *   grad  device fp32 [C_out][C_in] out: dL_cov / dL, or NULL (the gradient
 *         reaches every logit, selected or not, Sec. 3.2)
 * eps >= 0 (the paper does not print its value). Sums run in a fixed order
 * (u, ubar and the loss in double): results do not depend on scheduling.
 * Asynchronous; logits are not validated (a non-finite logit gives a
 * non-finite loss).
 */
moce_status_t moce_coverage_loss(const float *logits, int C_in, int C_out, float eps,
                                 float *loss, float *usage, float *grad, void *ws,
                                 size_t ws_bytes, moce_stream_t stream);

/*
 * Backward of the layer with static supports (Sec. 3.2: the loss reaches the
 * selected logit values through the weights; the indices get no gradient).
 * Given dy = dJ/dy of a scalar J, by the chain rule through the pool
 * (Sec. 3.3), the gate and Eq. (tau), Eq. (weights), Eq. (expert) and Eq. (res):
 *   da[n,e,i]  = sum_p dy[n,p,e] x[n,p,S_e[i]]
 *   ds[n,e,i]  = a[n,e,i] (da[n,e,i] - sum_j a[n,e,j] da[n,e,j])
 *   dlogits[e,i] = sum_n ds[n,e,i] / tau[n,e]
 *   dtau[n,e]  = -sum_i ds[n,e,i] L[e,i] / tau[n,e]^2, and on through sigma,
 *                w2, ReLU, W1, b1 to dW1, db1, dw2, db2 (summed over n, e)
 *                and to the pooled descriptors z (du = W1^T dh)
 *   dx[n,p,c]  = sum_{(e,i): S_e[i]=c} a[n,e,i] dy[n,p,e]
 *                + [c in U] dy[n,p,C_out] / |U| + dz[n,c] / (H W)
 * Arguments as moce_forward (x, supports, U, gate parameters, tau range), plus
 *   dy      device, dtype and layout of y (C_out + 1 channels)
 *   dx      device fp32 [N][H][W][C_in] (NHWC) or [N][C_in][H][W] (NCHW) out
 *   dlogits device fp32 [C_out][k] out, in packed order
 *   dW1     device fp32 [k][k] out (row j = hidden unit j), db1 / dw2 [k] out,
 *   db2     device fp32 [1] out
 * Every output is overwritten (not accumulated). With N = 0 or H W = 0 the
 * parameter gradients are zero. Every sum runs in a fixed order: two calls
 * give the same bits. ws: moce_backward_workspace_bytes, 256-byte aligned,
 * no initialisation needed. C_in + C_out <= 5688 and C_out <= 3400
 * (MOCE_ERR_UNSUPPORTED beyond: tiles staged in shared memory; the
 * workspace size is then 0). Asynchronous.
 */
size_t moce_backward_workspace_bytes(int N, int H, int W, int C_in, int C_out, int k);
moce_status_t moce_backward(const void *x, const void *dy, int N, int H, int W, int C_in,
                            int C_out, int k, moce_dtype_t dtype, moce_layout_t layout,
                            const int32_t *packed_idx, const float *packed_logits,
                            const int32_t *resid_idx, int n_resid, const float *W1,
                            const float *b1, const float *w2, const float *b2, float tau_min,
                            float tau_max, float *dx, float *dlogits, float *dW1, float *db1,
                            float *dw2, float *db2, void *ws, size_t ws_bytes,
                            moce_stream_t stream);

/*
 * SYNCHRONOUS: waits for `stream`, then reads the device error word the
 * forward kernels leave in `ws` (a forward workspace). Returns MOCE_OK,
 * MOCE_ERR_TIMEOUT (a bounded inter-CTA wait gave up; outputs of that call
 * are invalid and the workspace must be re-initialised) or MOCE_ERR_CUDA.
 */
moce_status_t moce_check_device_error(const void *ws, size_t ws_bytes, moce_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* MOCE_H */
