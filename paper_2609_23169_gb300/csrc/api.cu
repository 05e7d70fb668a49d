// The C ABI declared in include/ultratex.h: argument validation on the host,
// then the launches.  Nothing here allocates, frees or synchronises.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "../../include/ultratex.h"
#include "kernels.h"

namespace ut {

static int device_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
  return sms > 0 ? sms : 1;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;  // the driver entry point, resolved once
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &p, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// Row-major [rows x inner] bf16 matrix with a row pitch; 128B-swizzled boxes of
// box_inner (64) x box_rows elements; rows past `rows` read as zero.
bool encode_tmap_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner_elems, uint64_t rows,
                         uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner_elems, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

static ut_status from_cuda(cudaError_t e) { return e == cudaSuccess ? UT_OK : UT_ERR_CUDA; }

// Limit of every bounded device wait: 2 s, or UT_WAIT_TIMEOUT_NS from the
// environment (read at each call; 0 = give up at the first wait that is not
// already satisfied, which the failure-detection tests use).
static uint64_t wait_timeout_ns() {
  const char* e = getenv("UT_WAIT_TIMEOUT_NS");
  if (e && *e) {
    char* end = nullptr;
    unsigned long long v = strtoull(e, &end, 10);
    if (end && *end == '\0') return (uint64_t)v;
  }
  return 2000000000ull;
}

// Common checks of an attention shape.  nq_out gets ceil(N / block).
static int block_k_of(const ut_attn_shape* s) { return s->block_k > 0 ? s->block_k : s->block; }

static ut_status check_shape(const ut_attn_shape* s, int* nq_out, int* nk_out = nullptr) {
  if (!s) return UT_ERR_INVALID_ARG;
  if (s->n_tokens < 0 || s->n_heads < 1 || s->block < 1 || s->head_dim < 1 || s->block_k < 0)
    return UT_ERR_INVALID_ARG;
  if (s->dtype != UT_BF16 && s->dtype != UT_F32) return UT_ERR_INVALID_ARG;
  if (s->head_dim != 64 && s->head_dim != 128) return UT_ERR_UNSUPPORTED;
  const int64_t hd = (int64_t)s->n_heads * s->head_dim;
  const int64_t esz = s->dtype == UT_BF16 ? 2 : 4;
  if (s->row_stride < hd || (s->row_stride * esz) % 16 != 0) return UT_ERR_INVALID_ARG;
  if (s->n_tokens > INT32_MAX / 2) return UT_ERR_UNSUPPORTED;
  const int64_t nq = (s->n_tokens + s->block - 1) / s->block;
  const int64_t nk = (s->n_tokens + block_k_of(s) - 1) / block_k_of(s);
  if (nq * s->n_heads > INT32_MAX / 2 || nk * s->n_heads > INT32_MAX / 2) return UT_ERR_UNSUPPORTED;
  *nq_out = (int)nq;
  if (nk_out) *nk_out = (int)nk;
  return UT_OK;
}

static bool attn_block_supported(const ut_attn_shape* s) {
  const int bk = block_k_of(s);
  if (s->dtype == UT_BF16) return (s->block == 64 || s->block == 128) && (bk == 64 || bk == 128);
  return (s->block == 32 || s->block == 64 || s->block == 128) && bk == s->block;
}

static AttnProblem attn_problem(const ut_attn_shape* s, int nq, int nk, float scale) {
  AttnProblem p{s->n_tokens, s->n_heads, s->head_dim, s->block, s->dtype, s->row_stride, nq, scale,
                block_k_of(s), nk};
  return p;
}

}  // namespace ut

using namespace ut;

extern "C" {

const char* ut_strerror(ut_status s) {
  switch (s) {
    case UT_OK: return "ok";
    case UT_ERR_INVALID_ARG: return "invalid argument";
    case UT_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case UT_ERR_CUDA: return "CUDA error";
    case UT_ERR_TIMEOUT: return "device wait timed out";
    case UT_ERR_CAPACITY: return "output capacity exceeded";
  }
  return "unknown status";
}

int32_t ut_topk_count(double rho, int64_t n_k) {
  double f = floor(rho * (double)n_k);
  int64_t k = (int64_t)f;
  if (k < 1) k = 1;
  if (k > n_k) k = n_k;
  return (int32_t)k;
}

size_t ut_fg_compact_workspace_size(int64_t T) { return fg_compact_ws(T < 0 ? 0 : T); }

ut_status ut_fg_compact(const uint8_t* mask, int64_t T, int32_t n_tensors, const void* const* h_src,
                        void* const* h_dst, int64_t row_bytes, int64_t capacity, int32_t* idx_out, int32_t* n_out,
                        void* ws, size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (T < 0 || capacity < 0 || n_tensors < 1 || n_tensors > 8 || !n_out) return UT_ERR_INVALID_ARG;
  if (T > INT32_MAX) return UT_ERR_UNSUPPORTED;
  if (row_bytes <= 0 || row_bytes % 16 != 0) return UT_ERR_INVALID_ARG;
  if (!h_src || !h_dst) return UT_ERR_INVALID_ARG;
  if (T > 0) {
    if (!mask || !ws || ws_bytes < fg_compact_ws(T)) return UT_ERR_INVALID_ARG;
    if (capacity > 0 && !idx_out) return UT_ERR_INVALID_ARG;
    for (int i = 0; i < n_tensors; ++i) {
      if (!h_src[i] || !aligned16(h_src[i])) return UT_ERR_INVALID_ARG;
      if (capacity > 0 && (!h_dst[i] || !aligned16(h_dst[i]))) return UT_ERR_INVALID_ARG;
    }
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return from_cuda(launch_fg_compact(mask, T, n_tensors, h_src, h_dst, row_bytes, capacity, idx_out, n_out, ws,
                                     dev_status, device_sms(), s));
}

ut_status ut_fg_scatter(const int32_t* idx, int64_t n, int32_t n_tensors, const void* const* h_src,
                        void* const* h_dst, int64_t row_bytes, int32_t bg_mode, const void* fill_row, int64_t T,
                        void* stream) {
  if (n < 0 || T < 0 || n > T || n_tensors < 1 || n_tensors > 8) return UT_ERR_INVALID_ARG;
  if (row_bytes <= 0 || row_bytes % 16 != 0) return UT_ERR_INVALID_ARG;
  if (bg_mode != UT_BG_KEEP && bg_mode != UT_BG_ZERO && bg_mode != UT_BG_FILL) return UT_ERR_INVALID_ARG;
  if (!h_src || !h_dst) return UT_ERR_INVALID_ARG;
  if (bg_mode == UT_BG_FILL && (!fill_row || !aligned16(fill_row))) return UT_ERR_INVALID_ARG;
  if (n > 0 && !idx) return UT_ERR_INVALID_ARG;
  for (int i = 0; i < n_tensors; ++i) {
    if (n > 0 && (!h_src[i] || !aligned16(h_src[i]))) return UT_ERR_INVALID_ARG;
    if (T > 0 && (!h_dst[i] || !aligned16(h_dst[i]))) return UT_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return from_cuda(launch_fg_scatter(idx, n, n_tensors, h_src, h_dst, row_bytes, bg_mode, fill_row, T,
                                     device_sms(), s));
}

ut_status ut_fg_mask_from_alpha(const uint8_t* alpha, int32_t n_views, int32_t height, int32_t width,
                                int32_t factor, int32_t radius, int32_t threshold, uint8_t* canvas_mask,
                                void* stream) {
  if (n_views < 0 || height < 0 || width < 0 || factor < 1 || radius < 0 || radius > 16 || threshold < 0 ||
      threshold > 255)
    return UT_ERR_INVALID_ARG;
  if (height % factor != 0 || width % factor != 0) return UT_ERR_INVALID_ARG;
  if ((int64_t)height * width * (n_views + 1) > ((int64_t)1 << 40)) return UT_ERR_UNSUPPORTED;
  if (height == 0 || width == 0) return UT_OK;
  if (!alpha || !canvas_mask) return UT_ERR_INVALID_ARG;
  return from_cuda(launch_mask_from_alpha(alpha, n_views, height, width, factor, radius, threshold, canvas_mask,
                                          static_cast<cudaStream_t>(stream)));
}

static ut_status check_rope(int64_t n, int64_t T, int32_t n_tensors, const void* const* h_src,
                            void* const* h_dst, int32_t heads, int32_t head_dim, int32_t dtype, const ut_rope* rope,
                            bool gather) {
  if (n < 0 || T < 0 || n > T || n_tensors < 1 || n_tensors > 8 || heads < 1 || head_dim < 2) return UT_ERR_INVALID_ARG;
  if (dtype != UT_BF16 && dtype != UT_F32) return UT_ERR_INVALID_ARG;
  if (!rope || !h_src || !h_dst || rope->side < 1 || rope->prefix < 0 || !(rope->theta > 0.0f) ||
      !isfinite(rope->theta))
    return UT_ERR_INVALID_ARG;
  if (rope->axes[0] < 0 || rope->axes[1] < 0 || rope->axes[2] < 0 || rope->axes[0] % 2 || rope->axes[1] % 2 ||
      rope->axes[2] % 2 || (int64_t)rope->axes[0] + rope->axes[1] + rope->axes[2] != head_dim)
    return UT_ERR_INVALID_ARG;
  const int64_t head_bytes = (int64_t)head_dim * (dtype == UT_BF16 ? 2 : 4);
  if (head_bytes % 16 != 0 || 512 % head_bytes != 0) return UT_ERR_UNSUPPORTED;
  for (int i = 0; i < n_tensors; ++i) {
    const void* rows_n = gather ? h_dst[i] : h_src[i];
    const void* rows_t = gather ? h_src[i] : h_dst[i];
    if (n > 0 && (!rows_n || !aligned16(rows_n))) return UT_ERR_INVALID_ARG;
    if (T > 0 && (!rows_t || !aligned16(rows_t))) return UT_ERR_INVALID_ARG;
  }
  return UT_OK;
}

ut_status ut_fg_gather_rope(const int32_t* idx, int64_t n, int32_t n_tensors, const void* const* h_src,
                            void* const* h_dst, int64_t T, int32_t heads, int32_t head_dim, int32_t dtype,
                            const ut_rope* rope, void* stream) {
  ut_status st = check_rope(n, T, n_tensors, h_src, h_dst, heads, head_dim, dtype, rope, true);
  if (st != UT_OK) return st;
  if (n == 0) return UT_OK;
  if (!idx) return UT_ERR_INVALID_ARG;
  return from_cuda(launch_fg_rope(idx, n, n_tensors, h_src, h_dst, heads, head_dim, dtype == UT_BF16, rope->side,
                                  rope->prefix, rope->axes, rope->theta, 0, T, device_sms(), static_cast<cudaStream_t>(stream)));
}

ut_status ut_fg_scatter_rope(const int32_t* idx, int64_t n, int32_t n_tensors, const void* const* h_src,
                             void* const* h_dst, int64_t T, int32_t heads, int32_t head_dim, int32_t dtype,
                             const ut_rope* rope, int32_t bg_mode, void* stream) {
  ut_status st = check_rope(n, T, n_tensors, h_src, h_dst, heads, head_dim, dtype, rope, false);
  if (st != UT_OK) return st;
  if (bg_mode != UT_BG_KEEP && bg_mode != UT_BG_ZERO) return UT_ERR_INVALID_ARG;
  if (n > 0 && !idx) return UT_ERR_INVALID_ARG;
  const int mode = bg_mode == UT_BG_KEEP ? 1 : 2;
  if ((mode == 1 && n == 0) || T == 0) return UT_OK;
  return from_cuda(launch_fg_rope(idx, n, n_tensors, h_src, h_dst, heads, head_dim, dtype == UT_BF16, rope->side,
                                  rope->prefix, rope->axes, rope->theta, mode, T, device_sms(), static_cast<cudaStream_t>(stream)));
}

int32_t ut_device_accessible(const void* ptr) {
  if (!ptr) return 0;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    (void)cudaGetLastError();  // not a CUDA-known pointer: clear the error
    return 0;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return 1;
  return a.type == cudaMemoryTypeHost && a.devicePointer == ptr ? 1 : 0;
}

static ut_status euler_checked(const int32_t* idx, int64_t n, void* z, const void* v, int64_t T, int32_t channels,
                               int32_t dtype, float dt, int32_t* dev_status, void* zc, bool with_zc, void* stream) {
  if (n < 0 || T < 0 || n > T || channels <= 0) return UT_ERR_INVALID_ARG;
  if (dtype != UT_BF16 && dtype != UT_F32) return UT_ERR_INVALID_ARG;
  const int64_t row_bytes = (int64_t)channels * (dtype == UT_BF16 ? 2 : 4);
  if (row_bytes % 16 != 0) return UT_ERR_INVALID_ARG;
  if (!isfinite(dt)) return UT_ERR_INVALID_ARG;
  if (n == 0) return UT_OK;
  if (!idx || !z || !v || !aligned16(z) || !aligned16(v)) return UT_ERR_INVALID_ARG;
  if (with_zc && (!zc || !aligned16(zc))) return UT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return from_cuda(launch_fg_euler(idx, n, z, v, T, row_bytes, dtype == UT_BF16, dt, dev_status, with_zc ? zc : nullptr,
                                   device_sms(), s));
}

ut_status ut_fg_euler_update(const int32_t* idx, int64_t n, void* z, const void* v, int64_t T, int32_t channels,
                             int32_t dtype, float dt, int32_t* dev_status, void* stream) {
  return euler_checked(idx, n, z, v, T, channels, dtype, dt, dev_status, nullptr, false, stream);
}

ut_status ut_fg_euler_update_gather(const int32_t* idx, int64_t n, void* z, const void* v, void* zc, int64_t T,
                                    int32_t channels, int32_t dtype, float dt, int32_t* dev_status, void* stream) {
  return euler_checked(idx, n, z, v, T, channels, dtype, dt, dev_status, zc, true, stream);
}

ut_status ut_fg_composite(const uint8_t* mask, int64_t T, void* z, const void* z_bg, int64_t period,
                          int64_t row_bytes, void* stream) {
  if (T < 0 || period < 1 || row_bytes <= 0 || row_bytes % 16 != 0) return UT_ERR_INVALID_ARG;
  if (T == 0) return UT_OK;
  if (!mask || !z || !z_bg || !aligned16(z) || !aligned16(z_bg)) return UT_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return from_cuda(launch_fg_composite(mask, T, z, z_bg, period, row_bytes, device_sms(), s));
}

size_t ut_block_mask_workspace_size(const ut_attn_shape* shape, int32_t mode) {
  int nq = 0;
  int nk = 0;
  if (check_shape(shape, &nq, &nk) != UT_OK) return 0;
  MaskProblem p{shape->n_tokens, shape->n_heads, shape->head_dim, shape->block, shape->dtype, shape->row_stride, nq,
                block_k_of(shape), nk};
  return block_mask_ws(p, mode);
}

ut_status ut_block_mask(const ut_attn_shape* shape, int32_t mode, const void* q, const void* k, double rho,
                        const uint8_t* bitmap, int32_t* row_ptr, int32_t* col_idx, int64_t col_cap,
                        int32_t* col_ptr_t, int32_t* row_idx_t, void* ws, size_t ws_bytes, int32_t* dev_status,
                        void* stream) {
  int nq = 0, nk = 0;
  ut_status st = check_shape(shape, &nq, &nk);
  if (st != UT_OK) return st;
  if (mode != UT_MASK_TOPK && mode != UT_MASK_BITMAP) return UT_ERR_INVALID_ARG;
  if ((col_ptr_t == nullptr) != (row_idx_t == nullptr)) return UT_ERR_INVALID_ARG;
  if (!row_ptr || col_cap < 0) return UT_ERR_INVALID_ARG;
  if ((int64_t)nq * nk > (int64_t)1 << 31) return UT_ERR_UNSUPPORTED;
  MaskProblem p{shape->n_tokens, shape->n_heads, shape->head_dim, shape->block, shape->dtype, shape->row_stride, nq,
                block_k_of(shape), nk};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (nq == 0) {
    cudaError_t e = cudaMemsetAsync(row_ptr, 0, sizeof(int32_t), s);
    if (e == cudaSuccess && col_ptr_t) e = cudaMemsetAsync(col_ptr_t, 0, sizeof(int32_t), s);
    return from_cuda(e);
  }
  if (!ws || ws_bytes < block_mask_ws(p, mode)) return UT_ERR_INVALID_ARG;
  if (mode == UT_MASK_TOPK) {
    if (!(rho > 0.0) || !(rho <= 1.0)) return UT_ERR_INVALID_ARG;
    if (!q || !k || !aligned16(q) || !aligned16(k)) return UT_ERR_INVALID_ARG;
    const int32_t kr = ut_topk_count(rho, nk);
    if ((int64_t)shape->n_heads * nq * kr > col_cap || !col_idx) return UT_ERR_CAPACITY;
    return from_cuda(launch_block_mask_topk(p, q, k, kr, row_ptr, col_idx, col_ptr_t, row_idx_t, col_cap, ws,
                                            dev_status, device_sms(), s));
  }
  if (!bitmap || !dev_status) return UT_ERR_INVALID_ARG;
  if (col_cap > 0 && !col_idx) return UT_ERR_INVALID_ARG;
  return from_cuda(
      launch_block_mask_bitmap(p, bitmap, row_ptr, col_idx, col_ptr_t, row_idx_t, col_cap, ws, dev_status, s));
}

ut_status ut_bsattn_fwd(const ut_attn_shape* shape, const void* q, const void* k, const void* v,
                        const int32_t* row_ptr, const int32_t* col_idx, float softmax_scale, void* o, float* lse,
                        int32_t* dev_status, void* stream) {
  int nq = 0, nk = 0;
  ut_status st = check_shape(shape, &nq, &nk);
  if (st != UT_OK) return st;
  if (!attn_block_supported(shape)) return UT_ERR_UNSUPPORTED;
  if (!(softmax_scale > 0.f) || !isfinite(softmax_scale)) return UT_ERR_INVALID_ARG;
  if (shape->n_tokens == 0) return UT_OK;
  if (!q || !k || !v || !o || !lse || !row_ptr || !col_idx) return UT_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return UT_ERR_INVALID_ARG;
  const AttnProblem p = attn_problem(shape, nq, nk, softmax_scale);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (shape->dtype == UT_F32) return from_cuda(launch_attn_fwd_simt(p, q, k, v, row_ptr, col_idx, o, lse, s));
  return from_cuda(launch_attn_fwd_tc(p, q, k, v, row_ptr, col_idx, o, lse, dev_status, wait_timeout_ns(),
                                      device_sms(), s));
}

size_t ut_bsattn_bwd_workspace_size(const ut_attn_shape* shape) {
  int nq = 0, nk = 0;
  if (check_shape(shape, &nq, &nk) != UT_OK) return 0;
  const AttnProblem p = attn_problem(shape, nq, nk, 1.f);
  const size_t a = attn_bwd_simt_ws(p), b = attn_bwd_tc_ws(p);
  return (a > b ? a : b) + 256;
}

ut_status ut_bsattn_bwd(const ut_attn_shape* shape, const void* q, const void* k, const void* v, const void* o,
                        const float* lse, const void* dout, const int32_t* row_ptr, const int32_t* col_idx,
                        const int32_t* col_ptr_t, const int32_t* row_idx_t, float softmax_scale, void* dq, void* dk,
                        void* dv, void* ws, size_t ws_bytes, int32_t* dev_status, void* stream) {
  int nq = 0, nk = 0;
  ut_status st = check_shape(shape, &nq, &nk);
  if (st != UT_OK) return st;
  if (!attn_block_supported(shape)) return UT_ERR_UNSUPPORTED;
  if (!(softmax_scale > 0.f) || !isfinite(softmax_scale)) return UT_ERR_INVALID_ARG;
  if (shape->n_tokens == 0) return UT_OK;
  if (!q || !k || !v || !o || !lse || !dout || !row_ptr || !col_idx || !col_ptr_t || !row_idx_t || !dq || !dk ||
      !dv)
    return UT_ERR_INVALID_ARG;
  const AttnProblem p = attn_problem(shape, nq, nk, softmax_scale);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (shape->dtype == UT_F32) {
    if (!ws || ws_bytes < attn_bwd_simt_ws(p)) return UT_ERR_INVALID_ARG;
    return from_cuda(launch_attn_bwd_simt(p, q, k, v, o, lse, dout, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk,
                                          dv, ws, s));
  }
  if (!ws || ws_bytes < attn_bwd_tc_ws(p) || !aligned16(ws)) return UT_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(dout) || !aligned16(dq) ||
      !aligned16(dk) || !aligned16(dv))
    return UT_ERR_INVALID_ARG;
  return from_cuda(launch_attn_bwd_tc(p, q, k, v, o, lse, dout, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk, dv,
                                      ws, dev_status, wait_timeout_ns(), device_sms(), s));
}

}  // extern "C"
