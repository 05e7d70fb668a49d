/*
 * ultratex.h -- C ABI of the foreground-only block-sparse attention path of
 * "UltraTex: Unleashing 2K Multi-View Diffusion for 3D Texturing".
 *
 * The path (Sec. 3.2 and Sec. 3.3 of the paper):
 *   1. ut_fg_compact  -- Background Token Dropping: gather the foreground
 *                        tokens of the multi-view canvas (Gather_{M_fg}).
 *   2. ut_block_mask  -- per head and query block, the list of key blocks to
 *                        attend to: Top-K over mean-pooled compressed scores
 *                        S_c = pool(Q) pool(K)^T, or a caller-given bitmap.
 *   3. ut_bsattn_fwd  -- block-sparse attention over the listed key blocks.
 *   4. ut_bsattn_bwd  -- its gradient (the paper trains stage 3 with it).
 *   5. ut_fg_scatter  -- put compacted rows back at their canvas positions.
 *
 * Conventions shared by every entry point
 *   - Pointers are DEVICE pointers unless the parameter name starts with h_
 *     (host memory).  The caller owns every buffer, including workspaces
 *     sized by the *_workspace_size functions.  No entry point allocates or
 *     frees memory, synchronises the device or keeps global state (the one
 *     exception to the last, ut_fg_compact_noalloc, says so below).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy stream).  All
 *     work is enqueued on it; results are valid once the stream has reached
 *     the enqueued work.
 *   - Argument errors are detected on the host BEFORE anything is enqueued
 *     and returned as UT_ERR_INVALID_ARG / UT_ERR_UNSUPPORTED /
 *     UT_ERR_CAPACITY; a failed launch returns UT_ERR_CUDA.
 *   - Errors found on the device (a bounded wait that expired, a capacity
 *     that only the device can see) are written into `dev_status`: one
 *     int32 in device memory that the caller zeroes beforehand and reads
 *     after synchronising.  The first error wins.  `dev_status` may be NULL
 *     where noted.
 *   - Token-major layout: a token row holds H heads of d elements each, head
 *     h at element offset h*d; consecutive tokens are `row_stride` elements
 *     apart.  Row starts must be 16-byte aligned.
 */
#ifndef ULTRATEX_H
#define ULTRATEX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  UT_OK = 0,
  UT_ERR_INVALID_ARG = 1,   /* null pointer, misalignment, negative size ... */
  UT_ERR_UNSUPPORTED = 2,   /* a valid but unimplemented shape or dtype */
  UT_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed */
  UT_ERR_TIMEOUT = 4,       /* (device) a bounded wait expired; kernel gave up */
  UT_ERR_CAPACITY = 5       /* an output buffer is too small */
} ut_status;

typedef enum { UT_BF16 = 0, UT_F32 = 1 } ut_dtype;

/* Background handling of ut_fg_scatter. */
enum { UT_BG_KEEP = 0, UT_BG_ZERO = 1, UT_BG_FILL = 2 };
/* Modes of ut_block_mask. */
enum { UT_MASK_TOPK = 0, UT_MASK_BITMAP = 1 };

/* Shape of the compacted attention problem.  Sec. 3.3 states it per head as
 * Q, K, V in R^{N x d} partitioned into query blocks of b_q = block rows and
 * key blocks of b_kv = block_k rows (block_k = 0: b_kv = b_q).
 * N_q = ceil(N / b_q), N_k = ceil(N / b_kv); the last block may be partial
 * (its missing key rows are excluded, its missing query rows are not
 * written).  The bf16 tensor-core kernels work on 128 x 128 tiles; a 64-row
 * block fills half of a tile: two listed 64-row blocks share one operand
 * tile, or, for 64-row blocks on both sides, an item's lists are merged into
 * 128-row tiles when that takes fewer tiles; work on the parts of a tile that
 * no listed pair covers is computed and discarded. */
typedef struct {
  int64_t n_tokens;    /* N: rows of the compacted sequence, >= 0 */
  int32_t n_heads;     /* H >= 1 */
  int32_t head_dim;    /* d: 64 or 128 */
  int32_t block;       /* b_q, rows per query block: bf16 64 or 128; fp32 32, 64, 128 */
  int32_t dtype;       /* ut_dtype of Q, K, V, O, dO, dQ, dK, dV */
  int64_t row_stride;  /* elements between consecutive tokens, >= H*d, multiple of 8 */
  int32_t block_k;     /* b_kv, rows per key block (Sec. 3.3 sizes the two separately):
                          0 = same as block; bf16 64 or 128; fp32 equal to block */
} ut_attn_shape;

const char* ut_strerror(ut_status s);

/* 1 if kernels on the current device can read and write `ptr` directly
 * (device memory, or host memory mapped into the device's address space,
 * such as pinned memory on systems with unified addressing); 0 otherwise,
 * including on any error.  No device work is enqueued. */
int32_t ut_device_accessible(const void* ptr);

/* K_rho = max(1, floor(rho * n_k)) evaluated in double precision
 * (Sec. 3.3, the Top-K retention count). */
int32_t ut_topk_count(double rho, int64_t n_k);

/* ------------------------------------------------------------------------
 * Background Token Dropping (Sec. 3.2: z~ = Gather_{M_fg}(z); retained tokens
 * are concatenated in canvas order and keep their canvas position, which is
 * their RoPE index).
 *
 *   mask      [T] uint8, nonzero = foreground.
 *   h_src     host array of n_tensors device pointers, each [T rows x row_bytes].
 *   h_dst     host array of n_tensors device pointers, each [capacity rows x row_bytes].
 *   row_bytes bytes per token row (multiple of 16; pointers 16-byte aligned).
 *   capacity  rows available in each dst and in idx_out.
 *   idx_out   [capacity] int32: canvas position of compacted row n, ascending.
 *   n_out     one int32 the kernels can address (device memory, or pinned host
 *             memory where ut_device_accessible says so: the host then reads N
 *             after an event instead of a copy that could queue behind other
 *             transfers): N = number of foreground tokens.
 *   ws        workspace of ut_fg_compact_workspace_size(T) bytes.
 *   dev_status (may be NULL) receives UT_ERR_CAPACITY when N > capacity; rows
 *             beyond capacity are then not written (n_out still holds N).
 * 1 <= n_tensors <= 8; T may be 0 (then N = 0).  Gathering reuses nothing
 * from a previous call. */
size_t ut_fg_compact_workspace_size(int64_t T);
ut_status ut_fg_compact(const uint8_t* mask, int64_t T, int32_t n_tensors,
                        const void* const* h_src, void* const* h_dst, int64_t row_bytes,
                        int64_t capacity, int32_t* idx_out, int32_t* n_out,
                        void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* ut_fg_compact without a caller workspace.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory
 * (a host that owns every allocation and passes the library only its inputs
 * and outputs, or a loop that must not enter an allocator).  Same arguments
 * and results as ut_fg_compact, minus ws / ws_bytes (T = 0 writes N = 0;
 * N > capacity reports UT_ERR_CAPACITY in dev_status as there).  Its scratch
 * is a fixed 4 KiB device array inside the library (held by every GPU that
 * loads it until exit), so T is limited to 4,194,304 canvas tokens; a larger
 * T returns UT_ERR_UNSUPPORTED before anything is enqueued.  The first call
 * in each CUDA context looks up the array's address in that context (cached
 * under the context's unique id, so a context created later, e.g. after
 * cudaDeviceReset, gets its own lookup); that first call may also make the
 * CUDA runtime load the library's device code into the context, which
 * allocates inside the driver.  Make it before any stream capture.  All calls
 * in a context share the array: calls that overlap on the GPU race and must
 * be serialised by the caller.  The entry point itself calls no allocation,
 * free or allocating library routine. */
ut_status ut_fg_compact_noalloc(const uint8_t* mask, int64_t T, int32_t n_tensors,
                                const void* const* h_src, void* const* h_dst, int64_t row_bytes,
                                int64_t capacity, int32_t* idx_out, int32_t* n_out,
                                int32_t* dev_status, void* stream);

/* ------------------------------------------------------------------------
 * Scatter compacted rows back to the canvas: dst[idx[n]] = src[n] for n < N.
 * Background rows (canvas positions not in idx) are, by bg_mode:
 *   UT_BG_KEEP  not written ("background positions are not updated", Sec. 3.2);
 *   UT_BG_ZERO  set to zero (the adjoint of the gather, for gradients);
 *   UT_BG_FILL  set to fill_row (row_bytes bytes, device), the canonical
 *               background latent of Sec. 3.4's z_mix.
 * idx must be strictly increasing and < T (as ut_fg_compact writes it).
 * n is the host-side N; T the canvas rows of each dst. */
ut_status ut_fg_scatter(const int32_t* idx, int64_t n, int32_t n_tensors,
                        const void* const* h_src, void* const* h_dst, int64_t row_bytes,
                        int32_t bg_mode, const void* fill_row, int64_t T, void* stream);

/* ------------------------------------------------------------------------
 * Canvas mask from the renders' alpha channels (Sec. 3.2, mask construction):
 * the alpha is downsampled to the token grid (a token is foreground when some
 * pixel of its factor x factor block has alpha > threshold; factor 16 at 8x
 * VAE downsampling and 2x2 patches) and the token mask is dilated by a square
 * of radius tokens (radius 1: 3 x 3).  The view masks serve both the noisy
 * targets and the conditions; the reference image has its own.
 *   alpha        [n_views + 1, height, width] uint8 (the views, then the
 *                reference), device.
 *   canvas_mask  [(2 n_views + 1) * (height/factor) * (width/factor)] uint8
 *                output, 0/1, laid out as ut_fg_compact expects it: the
 *                n_views targets, the n_views conditions (view v's mask
 *                again), the reference; raster order inside each image.
 *   factor       >= 1, dividing height and width; radius 0..16; threshold
 *                0..255.
 * Host-side argument errors return before any launch. */
ut_status ut_fg_mask_from_alpha(const uint8_t* alpha, int32_t n_views, int32_t height, int32_t width,
                                int32_t factor, int32_t radius, int32_t threshold, uint8_t* canvas_mask,
                                void* stream);

/* ------------------------------------------------------------------------
 * Rotary position embedding fused with the gather of Q / K and with the
 * scatter of dQ / dK (Sec. 3.2: every retained token keeps its original RoPE
 * index, its canvas position).  The paper does not print the formula; this
 * library's reading: canvas position t of images of rope->side tokens per side,
 * stored one after another in raster order, has the coordinates
 *   (image, y, x) = (t / side^2, (t mod side^2) / side, t mod side);
 * the head dimension is split into three axes of rope->axes[0..2] dimensions
 * (even, summing to head_dim; 16/56/56 for 128); pair k of axis a, the
 * elements (2j, 2j+1) of the head vector, is rotated by the angle
 * coordinate_a * theta^(-2k/axes[a]).  Angles are formed in fp32 from
 * frequencies computed in double precision; sin/cos in fp32; the rotated pair
 * is rounded once to dtype. */
typedef struct {
  int32_t side;     /* tokens per image side */
  int32_t axes[3];  /* head dimensions of the image, y and x axes */
  float theta;      /* frequency base (10000) */
  int32_t prefix;   /* text tokens before the images (0 or e.g. 512): canvas
                       positions t < prefix are at (0, 0, 0), i.e. unrotated,
                       and image coordinates count from t - prefix */
} ut_rope;

/* dst[n] = R(idx[n]) src[idx[n]] for n < n, every listed tensor (Q and K):
 * the gather of ut_fg_compact with the rotation applied, reusing the idx a
 * ut_fg_compact call wrote (for V, dO).
 *   src, dst   arrays of n_tensors (1..8) device pointers; src rows [T, H, d],
 *              dst rows [n, H, d], row = heads * head_dim elements of dtype.
 *   head_dim   head_dim * element size must divide 512 bytes and be a
 *              multiple of 16 (bf16: 8..256, fp32: 4..128).
 * idx values outside [0, T) are skipped.  n = 0 is a no-op. */
ut_status ut_fg_gather_rope(const int32_t* idx, int64_t n, int32_t n_tensors,
                            const void* const* h_src, void* const* h_dst, int64_t T,
                            int32_t heads, int32_t head_dim, int32_t dtype, const ut_rope* rope,
                            void* stream);

/* The gradient of ut_fg_gather_rope: dst[idx[n]] = R(idx[n])^T src[n] (the
 * inverse rotation), background rows per bg_mode: UT_BG_KEEP (not written)
 * or UT_BG_ZERO (set to zero: the adjoint of the gather).  idx strictly
 * increasing and < T (as ut_fg_compact writes it).  Same layouts as above. */
ut_status ut_fg_scatter_rope(const int32_t* idx, int64_t n, int32_t n_tensors,
                             const void* const* h_src, void* const* h_dst, int64_t T,
                             int32_t heads, int32_t head_dim, int32_t dtype, const ut_rope* rope,
                             int32_t bg_mode, void* stream);

/* ------------------------------------------------------------------------
 * Sparse Euler step of the flow-matching sampler (Sec. 3.2, Eq. euler):
 *   z[idx[n]] += dt * v[n]  for n < n,   dt = t_prev - t_curr,
 * only at the retained positions; background rows of z are not touched (they
 * stay at their initial noise, as the paper's inference does).
 *   idx       [n] int32 canvas positions (as ut_fg_compact writes them);
 *             distinct, each in [0, T).
 *   z         [T, channels] canvas latent (dtype), updated in place.
 *   v         [n, channels] predicted velocities of the retained tokens, row n
 *             for position idx[n] (dtype).
 *   channels  latent values per token; channels * element size must be a
 *             multiple of 16 bytes.
 *   dtype     UT_BF16 or UT_F32; each element is one fp32 fused multiply-add
 *             fmaf(dt, v, z) rounded once to dtype (round to nearest even).
 *   dev_status (may be NULL) receives UT_ERR_INVALID_ARG if an idx value is
 *             outside [0, T); such rows are skipped.
 * n = 0 is a no-op.  Host-side argument errors return before any launch. */
ut_status ut_fg_euler_update(const int32_t* idx, int64_t n, void* z, const void* v, int64_t T,
                             int32_t channels, int32_t dtype, float dt, int32_t* dev_status,
                             void* stream);

/* The sparse Euler step fused with the gather of the next denoising step:
 * the update of ut_fg_euler_update, and the updated row also written to
 *   zc[n] = z[idx[n]] (after the update)  for n < n,
 * the compacted latent that the next step's model call takes (Sec. 3.2: the
 * model runs on the retained tokens only, gathered by M_fg every step).  One
 * pass reads idx, v and z's retained rows once and writes them to z and zc.
 *   zc  [n, channels] device (dtype), 16-byte aligned; may not overlap z or v.
 * Other arguments, rounding and errors as ut_fg_euler_update (rows whose idx
 * is outside [0, T) are skipped in both outputs). */
ut_status ut_fg_euler_update_gather(const int32_t* idx, int64_t n, void* z, const void* v, void* zc, int64_t T,
                                    int32_t channels, int32_t dtype, float dt, int32_t* dev_status,
                                    void* stream);

/* ------------------------------------------------------------------------
 * Composite latent for decoding (Sec. 3.4, Eq. mixed_latent):
 *   z[t] = z_bg[t mod period]  where mask[t] == 0;  foreground rows unchanged.
 * The canonical background latent (one image's latent, period = its rows;
 * period = 1 repeats one row everywhere) is tile-repeated over the canvas,
 * which for images stored one after another in raster order puts tile row
 * (y, x) at position (y, x) of every image.  A plain bit copy: any dtype.
 *   mask      [T] uint8, nonzero = foreground (as given to ut_fg_compact).
 *   z         [T, row_bytes] canvas latent, updated in place.
 *   z_bg      [period, row_bytes] background tile (device).
 *   row_bytes a multiple of 16.
 * T = 0 is a no-op.  Host-side argument errors return before any launch. */
ut_status ut_fg_composite(const uint8_t* mask, int64_t T, void* z, const void* z_bg, int64_t period,
                          int64_t row_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Block mask M_c as per-(head, query block) key-block lists (Sec. 3.3).
 * Rows r = h*N_q + i (head-major).  Lists are ascending.
 *
 * UT_MASK_TOPK: S_c = pool(Q) pool(K)^T per head with mean pooling over the
 *   valid rows of each block (fp32), then per row the K_rho =
 *   ut_topk_count(rho, N_k) largest scores; equal scores go to the smaller
 *   key-block index.  `q`, `k` are the compacted [N, H, d] tensors; `bitmap`
 *   is ignored.  row_ptr[r] = r * K_rho.
 * UT_MASK_BITMAP: `bitmap` is [H, N_q, N_k] uint8 (nonzero = keep), given by
 *   the caller (structured masks); `q`, `k`, `rho` are ignored.  A row may be
 *   empty; the attention then writes O = 0 and LSE = -inf for it.
 *
 *   row_ptr   [H*N_q + 1] int32, col_idx [col_cap] int32 (CSR).
 *   col_ptr_t [H*N_k + 1] int32, row_idx_t [col_cap] int32: the transpose
 *             (per key block, ascending query blocks) for the backward; pass
 *             both NULL to skip it.
 *   ws        ut_block_mask_workspace_size(shape, mode) bytes.
 *   dev_status receives UT_ERR_CAPACITY if the bitmap holds more than
 *             col_cap entries (must be non-NULL in bitmap mode).
 * TOPK mode checks H*N_q*K_rho <= col_cap on the host. */
size_t ut_block_mask_workspace_size(const ut_attn_shape* shape, int32_t mode);
ut_status ut_block_mask(const ut_attn_shape* shape, int32_t mode,
                        const void* q, const void* k, double rho, const uint8_t* bitmap,
                        int32_t* row_ptr, int32_t* col_idx, int64_t col_cap,
                        int32_t* col_ptr_t, int32_t* row_idx_t,
                        void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* ------------------------------------------------------------------------
 * Block-sparse attention forward (Sec. 3.3):
 *   O_i = softmax(Q_i K_{S_i}^T * softmax_scale) V_{S_i}
 * for every head and query block i, S_i the list row_ptr/col_idx gives
 * (query blocks of b_q rows, listed key blocks of b_kv rows).
 * A query row whose block lists no key block gets O = 0 and LSE = -inf.
 *   q, k, v, o  [N, H, d] token-major with shape->row_stride (dtype of shape).
 *   lse         [H, N] fp32 natural-log row normalisers (m + log sum exp).
 *   softmax_scale  1/sqrt(d) in the paper; any positive value accepted.
 * bf16 runs on the tcgen05 tensor cores (fp32 accumulation, P rounded to
 * bf16 before P V, O rounded to bf16); fp32 runs a CUDA-core fp32 kernel. */
ut_status ut_bsattn_fwd(const ut_attn_shape* shape, const void* q, const void* k, const void* v,
                        const int32_t* row_ptr, const int32_t* col_idx, float softmax_scale,
                        void* o, float* lse, int32_t* dev_status, void* stream);

/* ------------------------------------------------------------------------
 * Gradient of ut_bsattn_fwd with respect to Q, K, V given dO:
 *   D_r = dO_r . O_r,  P = exp(S - LSE),  dV = P^T dO,  dS = P o (dO V^T - D),
 *   dQ = dS K * scale,  dK = dS^T Q * scale
 * over the retained block pairs only.  Needs the CSR lists and their
 * transpose (col_ptr_t / row_idx_t from ut_block_mask).
 *   o, lse      the forward's outputs.
 *   dq, dk, dv  [N, H, d] outputs (dtype of shape), fully overwritten.
 *   ws          ut_bsattn_bwd_workspace_size(shape) bytes: D and LSE*log2(e)
 *               per head and padded row, and for bf16 an fp32 dQ accumulator
 *               [H, ceil(N/128)*128, d] (about 4*H*N*d bytes) followed by
 *               the counter that hands key blocks to the kernel's CTAs.
 * bf16 runs one fused tensor-core kernel per key block (S and dP computed
 * once per retained pair); dQ is summed over key blocks with fp32 atomic
 * additions, so its last bits may differ between runs (dK, dV do not). */
size_t ut_bsattn_bwd_workspace_size(const ut_attn_shape* shape);
ut_status ut_bsattn_bwd(const ut_attn_shape* shape, const void* q, const void* k, const void* v,
                        const void* o, const float* lse, const void* dout,
                        const int32_t* row_ptr, const int32_t* col_idx,
                        const int32_t* col_ptr_t, const int32_t* row_idx_t, float softmax_scale,
                        void* dq, void* dk, void* dv, void* ws, size_t ws_bytes,
                        int32_t* dev_status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* ULTRATEX_H */
