/*
 * groupsparse.h - C ABI of the GB300 group-sparse linear layer.
 *
 * The layer is the pruned projection of GroupMask (Sec. 2.1, Eq. 1):
 *     M = B (x) 1_{1 x 256},   W_hat = W (.) M,   y = x W_hat^T
 * W[out][in] is a frozen bf16 weight, B[out][in/256] keeps (nonzero) or prunes
 * (zero) each 1x256 group of W, and x[T][in] holds T tokens.  Pruned groups are
 * never read: the weight is first packed into a chunk-major compressed layout
 * (gs_pack), then every gs_linear call streams only the kept groups.
 *
 * Conventions shared by every call:
 *   - Pointers named *_dev are device pointers (cudaMalloc'd or equivalent) on
 *     the current CUDA device; pointers named *_host are host pointers.
 *   - bf16 tensors are passed as raw 16-bit storage (void*), row-major, densely
 *     strided.  Device tensor pointers must be 16-byte aligned.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls are
 *     asynchronous on that stream unless stated otherwise.
 *   - Arguments are validated on the host before anything is launched; a
 *     failed validation returns GS_ERR_INVALID_ARG or GS_ERR_UNSUPPORTED and
 *     touches no device memory.
 *   - The caller owns W, mask, x, y and W_hat.  The library owns the handle's
 *     device buffers until gs_free.
 *   - One process drives one CUDA device: the kernels' shared-memory limits
 *     and the SM count that sizes their grids are configured on the first
 *     device that launches them and reused for every later call.
 *   - Kernels bound every wait they perform.  A wait that runs out records
 *     GS_ERR_DEVICE_TIMEOUT in a library-owned device flag and the kernel
 *     returns; gs_device_status reads (and clears) that flag.
 */
#ifndef GROUPSPARSE_H
#define GROUPSPARSE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum gs_status {
  GS_OK = 0,
  GS_ERR_INVALID_ARG = 1,     /* null pointer, bad size, misaligned pointer    */
  GS_ERR_UNSUPPORTED = 2,     /* valid request outside what is implemented     */
  GS_ERR_OOM = 3,             /* device allocation failed                      */
  GS_ERR_CUDA = 4,            /* a CUDA runtime/driver call or launch failed   */
  GS_ERR_DEVICE_TIMEOUT = 5   /* a kernel's bounded wait ran out               */
} gs_status;

/* Kernel family for gs_linear_ex. */
typedef enum gs_algo {
  GS_ALGO_AUTO = 0,     /* pick by token count and group shape                       */
  GS_ALGO_DECODE = 1,   /* CUDA-core/mma.sync streaming kernel (memory-bound)        */
  GS_ALGO_PREFILL = 2,  /* tcgen05/TMEM/TMA tensor-core kernel (compute-bound)        */
  GS_ALGO_PREFILL_DENSE = 3  /* tcgen05 kernel over zero-filled 256-row windows: tensor
                                work of the dense layer, no gather; 1 x 128 and 1 x 256
                                groups; GS_ALGO_AUTO picks it from T = 17 (1 x 128)
                                and from T = 129 (1 x 256)                             */
} gs_algo;

typedef struct gs_packed gs_packed;   /* opaque, library-owned */

/*
 * gs_pack - compress W with the group mask B into the chunk-major layout.
 *
 * Follows Eq. 1 (Sec. 2.1): the mask selects whole 1 x group_in groups of W;
 * only kept groups are stored.  Packed layout (bit-exact, deterministic):
 *   chunk c (input columns [256c, 256c+256)) owns packed rows
 *   [offsets[c], offsets[c+1]); within a chunk the kept rows appear in
 *   ascending row order; row_idx[j] is the output row of packed row j and
 *   tiles[j][0:256] is a bit copy of W[row_idx[j]][256c : 256c+256].
 *   win_off16[c][w] is the first packed row of chunk c whose output row is
 *   >= 16w (w = 0..ceil(out/16); entry ceil(out/16) is offsets[c+1]) and
 *   kmask16[c][w] has bit i set when row 16w+i is kept in chunk c.
 *
 * W_dev     bf16 [out][in] row-major, caller-owned, read only.
 * mask_dev  uint8 [out][in/256] row-major; nonzero = keep.  Read only.
 * out, in   out >= 1; in >= 256 and a multiple of 256; out*(in/256) < 2^31.
 * group_in  must be 256 (other group shapes: GS_ERR_UNSUPPORTED).
 * stream    work is queued on it; gs_pack synchronizes it once to learn the
 *           kept-group count before allocating the packed buffers; the
 *           remaining packing kernels complete in stream order on `stream`.
 * handle    receives the new handle (set to NULL on failure).
 * Errors: INVALID_ARG (nulls, sizes, alignment), UNSUPPORTED (group_in),
 *         OOM, CUDA.
 */
gs_status gs_pack(const void* W_dev, const uint8_t* mask_dev, int64_t out, int64_t in,
                  int32_t group_in, void* stream, gs_packed** handle);

/*
 * gs_pack_groups - gs_pack for other group shapes.  Sec. 2.1 splits W into
 * non-overlapping g_out x g_in groups and B[G_out][G_in] keeps or prunes each
 * (Eq. 1 with M = B (x) 1_{g_out x g_in}); the Sec. 3.5 granularity ablation
 * and App. E evaluate 1 x 128, 1 x 256, 16 x 16, 32 x 32, 64 x 64 and
 * 128 x 128.  Supported here: (1, 256), which is gs_pack itself, (1, 128),
 * whose layout is gs_pack's with 128-wide chunks (offsets, row_idx, tiles of
 * 128 bf16, win_off16 and kmask16 as gs_pack describes them, over chunks of
 * 128 input columns), and square g x g with g in {16, 32, 64, 128}; other
 * shapes return GS_ERR_UNSUPPORTED.
 *
 * Packed layout of square groups (bit-exact, deterministic): column block v
 * (input columns [g v, g v + g)) owns packed tiles [offsets[v], offsets[v+1]);
 * inside a column block the kept block rows u ascend; row_idx[j] is the block
 * row of tile j and tiles[j] is a bit copy of the g x g block of W at rows
 * [g u, g u + g), columns [g v, g v + g), row-major.
 *
 * W_dev     bf16 [out][in] row-major, caller-owned, read only.
 * mask_dev  uint8 [out/g_out][in/g_in] row-major; nonzero = keep.  Read only.
 * out, in   multiples of g_out and g_in (the groups tile W exactly);
 *           (out/g_out)(in/g_in) < 2^31 and in/g_in <= 65535.
 * stream, handle: as for gs_pack (one synchronization to size the buffers).
 * gs_linear, gs_linear_ex (the kernel family is chosen by the handle: square
 * groups have one tensor-core kernel for every token count),
 * gs_linear_batched, gs_unpack, gs_packed_info, gs_packed_export and gs_free
 * accept the handle.
 * Errors: INVALID_ARG (nulls, sizes, alignment), UNSUPPORTED (shape), OOM, CUDA.
 */
gs_status gs_pack_groups(const void* W_dev, const uint8_t* mask_dev, int64_t out, int64_t in, int32_t g_out,
                         int32_t g_in, void* stream, gs_packed** handle);

/* gs_packed_group_shape - the group shape a handle was packed with (either pointer may be NULL). */
gs_status gs_packed_group_shape(const gs_packed* p, int32_t* g_out, int32_t* g_in);

/*
 * gs_linear - y = x W_hat^T for the packed weight (Eq. 1 applied as a linear
 * projection, no bias), fp32 accumulation, bf16 output rounded to nearest even.
 *
 * x_dev  bf16 [T][in] row-major, caller-owned, read only.
 * p      packed handle from gs_pack; read only, so one handle may serve
 *        gs_linear / gs_linear_ex / gs_linear_batched calls on several streams
 *        at once.  The decode kernel's split-reduction scratch is kept per
 *        (handle, stream): the scratch of gs_pack's stream is made by gs_pack,
 *        and the first decode-regime call on any other stream allocates and
 *        zeroes that stream's, synchronously and outside any graph capture
 *        in progress on it.  Up to 8 streams per handle.  Calls on one stream
 *        are ordered by the stream; a CUDA graph keeps the scratch of the
 *        stream it was captured from, so its replays must be ordered with
 *        other work on that stream.
 * T      number of tokens; T == 0 is a no-op, T < 0 is INVALID_ARG.
 * y_dev  bf16 [T][out] row-major, caller-owned; fully overwritten (rows of
 *        outputs with no kept group are written as +0.0).
 * Errors: INVALID_ARG, UNSUPPORTED (a ninth stream on one handle), OOM (a new
 * stream's scratch), CUDA.  Asynchronous on `stream`.
 */
gs_status gs_linear(const void* x_dev, const gs_packed* p, int64_t T, void* y_dev, void* stream);

/* gs_linear with an explicit kernel family (same arguments and result). */
gs_status gs_linear_ex(const void* x_dev, const gs_packed* p, int64_t T, void* y_dev, void* stream,
                       gs_algo algo);

/*
 * gs_linear_batched - n independent layers, ys[i] = xs[i] W_hat_i^T for the
 * i-th handle, all with the same token count T.  In the decode regime all n
 * layers share one launch per 16 tokens (one grid streams every layer's kept
 * groups); in the prefill regime (T >= 17) up to 8 layers share one launch
 * (one list of output tiles).  Results are those of gs_linear for each layer
 * (prefill: bit for bit).  Same per-layer semantics and errors as gs_linear.
 * 1 <= n <= 32 (n == 0 is a no-op); the handles must be distinct.
 */
gs_status gs_linear_batched(int32_t n, const void* const* xs_dev, const gs_packed* const* ps,
                            int64_t T, void* const* ys_dev, void* stream);

/*
 * gs_select_groups - selector export (Sec. 2.2: at evaluation the Gumbel noise
 * is dropped and the selectors are thresholded; App. F: the exported masks use
 * the same rule).  B[i] = 1 when sigmoid(logits[i]) > 1/2, i.e. exactly when
 * logits[i] > 0: +0, -0 and NaN prune, +inf keeps.  Also counts the kept
 * groups, sum_uv B_uv of Eq. 2, from which the caller forms the preserved
 * rates (kept / (G_out G_in) per layer, since every group holds g_out g_in
 * weights).
 *
 * logits_dev  float32 [n], device, caller-owned, 16-byte aligned, read only.
 *             For one layer with 1x256 groups: [out][in/256] row-major.
 * n           number of selectors, 0 <= n < 2^36.
 * mask_dev    uint8 [n], device, caller-owned, 16-byte aligned, fully
 *             overwritten with 0 / 1: the mask layout gs_pack takes.  Must not
 *             overlap logits_dev.
 * kept_dev    int64, device, 8-byte aligned, overwritten with the number of
 *             ones written; may be NULL.
 * Results are exact (integer test on the float32 bit pattern).  n == 0
 * writes kept = 0 and launches no kernel.  Asynchronous on `stream`.
 * Errors: INVALID_ARG (n out of range, NULL or misaligned pointers, overlap),
 * CUDA.
 */
gs_status gs_select_groups(const float* logits_dev, int64_t n, uint8_t* mask_dev, int64_t* kept_dev,
                           void* stream);

/*
 * gs_unpack - the check path: W_hat_dev[r][k] = W[r][k] where the group of
 * (r, k) is kept, +0.0 (0x0000) where it is pruned (M of Eq. 1 as a select).
 * W_hat_dev  bf16 [out][in], caller-owned, fully overwritten.
 * Errors: INVALID_ARG, CUDA.  Asynchronous on `stream`.
 */
gs_status gs_unpack(const gs_packed* p, void* W_hat_dev, void* stream);

/*
 * gs_packed_info - sizes of a handle (any output pointer may be NULL).
 * kept_groups = offsets[G] = the number of kept groups (sum of B, Eq. 2);
 * device_bytes = bytes of device memory the handle owns.
 */
gs_status gs_packed_info(const gs_packed* p, int64_t* out, int64_t* in, int64_t* kept_groups,
                         size_t* device_bytes);

/*
 * gs_packed_export - synchronous copy of the packed layout to host buffers
 * (for bit-exact checks).  The layout holds exactly the kept groups of Eq. 1
 * (Sec. 2.1: B selects whole 1 x 256 groups of W) and where each one sits in
 * W; the paper prints no layout, and the one here is the chunk-major layout
 * that gs_pack describes.  Sizes: offsets int64[G+1], row_idx int32[K],
 * tiles uint16[K*256], win_off16 int32[G*(ceil(out/16)+1)],
 * kmask16 uint16[G*ceil(out/16)], with K = kept_groups.  Any pointer may be NULL.
 * For 1 x 128 handles the chunks are 128 wide: G = in/128 and tiles
 * uint16[K*128].
 * For handles of square g x g groups (gs_pack_groups): offsets int64[in/g+1],
 * row_idx int32[K] (block rows), tiles uint16[K*g*g]; win_off16 and kmask16
 * must be NULL (INVALID_ARG otherwise).
 */
gs_status gs_packed_export(const gs_packed* p, int64_t* offsets_host, int32_t* row_idx_host,
                           uint16_t* tiles_host, int32_t* win_off16_host, uint16_t* kmask16_host);

/*
 * gs_pack_index_noalloc - the index part of gs_pack (per-chunk offsets, per
 * 16-row-window offsets and kept masks, exactly as gs_packed_export reports
 * them) computed without allocating any device memory.  The paper has no
 * counterpart; this entry point exists for callers that cannot allocate device
 * memory when they pack: code running inside a CUDA graph capture, where
 * cudaMalloc is not allowed, and runtimes that hand out all device memory from
 * their own fixed arena.
 *
 * mask_dev       uint8 [out][in/256] row-major; nonzero = keep.  Read only.
 * out, in        out >= 1; in >= 256 and a multiple of 256.
 * offsets_dev    int64 [in/256 + 1], caller-owned, 8-byte aligned, overwritten.
 * win_off16_dev  int32 [in/256][ceil(out/16) + 1], caller-owned, 4-byte
 *                aligned, overwritten.
 * kmask16_dev    uint16 [in/256][ceil(out/16)], caller-owned, 2-byte aligned,
 *                overwritten.
 * The three outputs must not overlap each other or the mask.
 * Temporary counts live in one fixed array in the library's device memory
 * (2^20 entries of int32, held by every GPU that loads the library until the
 * process exits); (in/256) * ceil(out/16) above 2^20 returns
 * GS_ERR_UNSUPPORTED before anything is launched.  All calls share that array:
 * calls whose kernels overlap on the GPU (different streams without ordering)
 * race and must be serialized by the caller.  Every entry a call reads is
 * written by the same call first, so nothing needs clearing between calls.
 * The first call on a device looks up the array's device address (with that
 * device current) and caches it; make that first call before any stream
 * capture.  Asynchronous on `stream`.
 * Errors: INVALID_ARG (nulls, sizes, misaligned or overlapping buffers),
 * UNSUPPORTED (beyond the fixed array), CUDA.
 */
gs_status gs_pack_index_noalloc(const uint8_t* mask_dev, int64_t out, int64_t in, int64_t* offsets_dev,
                                int32_t* win_off16_dev, uint16_t* kmask16_dev, void* stream);

/* Releases the handle and its device buffers (NULL is a no-op). */
void gs_free(gs_packed* p);

/* Static description of a status code. */
const char* gs_status_string(gs_status s);

/*
 * gs_device_status - synchronizes `stream`, then reads and clears the device
 * error flag of the current device: GS_OK or GS_ERR_DEVICE_TIMEOUT (a bounded
 * wait in some earlier kernel ran out).  GS_ERR_CUDA if the stream itself
 * reports an error.  After a timeout, the outputs of the call that timed out
 * (and of calls issued before this status was read) are undefined.  Reading
 * the timeout also marks every decode split scratch for re-zeroing, which
 * happens on the stream of its next use, so later calls are correct again.
 */
gs_status gs_device_status(void* stream);

/*
 * gs_preserved_rates - the preserved rates of App. F from kept-group counts:
 * a projection's active weights over its total weights after the binary mask
 * is applied, and the global rate over all target projections, which is
 * 1 - s of Eq. 2 (the parameter-weighted mean).  Every group holds
 * group_weights = g_out * g_in weights (256 for 1 x 256 groups).
 *
 * n               number of layers, n >= 0.
 * kept_host       int64 [n] kept groups per layer (e.g. gs_packed_info, or the
 *                 count gs_select_groups writes).
 * d_out_host,
 * d_in_host       int64 [n] layer shapes.
 * rates_host      double [n] or NULL: kept_i * group_weights / (d_out_i d_in_i).
 * global_host     double or NULL: sum_i kept_i group_weights / sum_i d_out_i d_in_i
 *                 (0 when n == 0).
 * n_qkv, qkv_host int32 [n_qkv][3] layer indices (q, k, v); App. F reports the
 *                 three attention input projections as the plain mean of their
 *                 rates: qkv_rates_host[j] = (r_q + r_k + r_v) / 3.
 * Host only (no device work).  Errors: INVALID_ARG (negative sizes or counts,
 * more kept weights than a layer holds, an index out of range, totals at or
 * above 2^62, NULL arrays with nonzero counts).
 */
gs_status gs_preserved_rates(int32_t n, const int64_t* kept_host, const int64_t* d_out_host,
                             const int64_t* d_in_host, int64_t group_weights, double* rates_host,
                             double* global_host, int32_t n_qkv, const int32_t* qkv_host,
                             double* qkv_rates_host);

/*
 * gs_gumbel_select - one training-time sample of the selectors (Sec. 2.2: a
 * Gumbel-Sigmoid relaxation with a straight-through estimator; the
 * temperature of Table 7 is 0.4).  The paper names the relaxation without
 * printing it; the standard form is used:
 *     z = l + L,   B = [z > 0] = [sigmoid(z / tau) > 1/2],
 *     ds/dl = s (1 - s) / tau  with  s = sigmoid(z / tau)
 * where L is standard logistic noise (the difference of two standard Gumbel
 * draws), which the caller draws.  B is the binary mask of the forward pass
 * (pack W with it: gs_pack / gs_pack_groups, then gs_linear); ds/dl is the
 * derivative the straight-through estimator puts in place of dB/dl in the
 * backward pass (gs_masked_linear_backward).  It is formed as
 * t / (1 + t)^2 / tau with t = exp(-|z| / tau), which keeps its relative
 * precision where s is near 0 or 1.  z is the float32 sum rounded to nearest;
 * NaN prunes.
 *
 * logits_dev, noise_dev  float32 [n], device, 4-byte aligned, read only.
 * tau                    temperature, > 0 and finite.
 * mask_dev               uint8 [n], overwritten with 0 / 1.
 * dsdl_dev               float32 [n] or NULL, overwritten with ds/dl.
 * kept_dev               int64 or NULL, 8-byte aligned: the number of ones.
 * Outputs must not overlap the inputs or each other.  Asynchronous on stream.
 * Errors: INVALID_ARG, CUDA.
 */
gs_status gs_gumbel_select(const float* logits_dev, const float* noise_dev, int64_t n, float tau, uint8_t* mask_dev,
                           float* dsdl_dev, int64_t* kept_dev, void* stream);

/*
 * gs_masked_linear_backward - the straight-through backward pass of the masked
 * linear y = x W_hat^T, W_hat = W (.) (B (x) 1) (Eq. 1), with W frozen
 * (Sec. 2.2; the pretrained weights are not updated):
 *     dL/dW_hat = dy^T x
 *     dL/dB[u][v] = sum over the cells (r, k) of group (u, v) of W[r][k] dL/dW_hat[r][k]
 *     dL/dl[u][v] = dL/dB[u][v] ds/dl[u][v]             (the estimator)
 *     dL/dx = dy W_hat
 * Every group receives a logit gradient, pruned ones included.  The two
 * products are dense GEMMs done by cuBLAS (fp32 accumulation); the group
 * reduction and the estimator are a kernel of this library.
 *
 * x_dev       bf16 [T][in] (the forward input).      W_dev  bf16 [out][in] (dense, frozen).
 * p           handle of W packed with the sampled mask B (any supported group shape).
 * dy_dev      bf16 [T][out], the gradient of the loss with respect to y.
 * dsdl_dev    float32 [out/g_out][in/g_in]: ds/dl from gs_gumbel_select.
 * dlogits_dev float32 [out/g_out][in/g_in], overwritten.
 * dx_dev      bf16 [T][in], overwritten, or NULL (no input gradient).
 * workspace   device scratch of gs_masked_linear_backward_workspace bytes
 *             (16-byte aligned; it holds dL/dW_hat and, with dx, W_hat).
 * Not for use inside a CUDA graph capture (cuBLAS may allocate on first use).
 * Errors: INVALID_ARG (nulls, sizes, alignment, workspace too small), CUDA.
 */
gs_status gs_masked_linear_backward_workspace(const gs_packed* p, int32_t want_dx, size_t* bytes);
gs_status gs_masked_linear_backward(const void* x_dev, const void* W_dev, const gs_packed* p, const void* dy_dev,
                                    int64_t T, const float* dsdl_dev, float* dlogits_dev, void* dx_dev,
                                    void* workspace_dev, size_t workspace_bytes, void* stream);

/*
 * Test hooks for the failure paths (the paper has no counterpart; they exist
 * so that the error handling can be exercised without faulting a GPU).
 *
 * gs_debug_fail_alloc(nth) - the nth device allocation the library makes from
 * now on fails as if the device were out of memory (nth = 1: the next one;
 * 0 disarms).  gs_pack then returns GS_ERR_OOM and frees what it had
 * allocated.
 *
 * gs_debug_inject_wait(family, limit_ns) - the next launch of that kernel
 * family (GS_ALGO_DECODE, GS_ALGO_PREFILL or GS_ALGO_PREFILL_DENSE) makes its
 * first CTA (the first CTA pair for the tensor-core kernels) wait, before
 * issuing any copy or tensor-core work, on
 * a library word that nothing ever sets, for at most limit_ns (<= 1 s).  The
 * wait runs out, the kernel records GS_ERR_DEVICE_TIMEOUT and that CTA skips
 * its work; the other CTAs finish theirs.  One-shot; limit_ns = 0 disarms.
 * Errors: INVALID_ARG (negative count, unknown family, limit above 1 s).
 */
gs_status gs_debug_fail_alloc(int64_t nth);
gs_status gs_debug_inject_wait(gs_algo family, uint64_t limit_ns);

/* Number of kernel launches the library issued since the process started (all
 * families; used to report launch counts). */
int64_t gs_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* GROUPSPARSE_H */
