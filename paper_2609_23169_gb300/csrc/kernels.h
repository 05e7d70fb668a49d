// Host-side launchers implemented by the .cu files; api.cu validates
// arguments and calls these.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ut {

// compact.cu
size_t fg_compact_ws(int64_t T);
cudaError_t launch_fg_compact(const uint8_t* mask, int64_t T, int n_tensors, const void* const* src,
                              void* const* dst, int64_t row_bytes, int64_t capacity, int32_t* idx, int32_t* n_out,
                              void* ws, int32_t* status, int sms, cudaStream_t stream);
cudaError_t launch_fg_scatter(const int32_t* idx, int64_t N, int n_tensors, const void* const* src, void* const* dst,
                              int64_t row_bytes, int bg_mode, const void* fill, int64_t T, int sms,
                              cudaStream_t stream);

// sampler.cu
cudaError_t launch_fg_euler(const int32_t* idx, int64_t n, void* z, const void* v, int64_t T, int64_t row_bytes,
                            bool bf16, float dt, int32_t* status, void* zc, int sms, cudaStream_t stream);
cudaError_t launch_fg_composite(const uint8_t* mask, int64_t T, void* z, const void* tile, int64_t period,
                                int64_t row_bytes, int sms, cudaStream_t stream);

// rope.cu (mode: 0 gather, 1 scatter keeping the background, 2 scatter zeroing it)
cudaError_t launch_fg_rope(const int32_t* idx, int64_t n, int n_tensors, const void* const* src, void* const* dst,
                           int heads, int head_dim, bool bf16, int side, int prefix, const int32_t axes[3],
                           float theta, int mode, int64_t T, int sms, cudaStream_t stream);

// mask_alpha.cu
cudaError_t launch_mask_from_alpha(const uint8_t* alpha, int n_views, int height, int width, int factor,
                                   int radius, int threshold, uint8_t* canvas, cudaStream_t stream);

// blockmask.cu
struct MaskProblem {
  int64_t N;
  int H, d, block, dtype;
  int64_t row_stride;
  int nq;       // query blocks of `block` rows
  int block_k;  // rows per key block
  int nk;       // key blocks
};
size_t block_mask_ws(const MaskProblem& p, int mode);
cudaError_t launch_block_mask_topk(const MaskProblem& p, const void* q, const void* k, int k_rho, int32_t* row_ptr,
                                   int32_t* col_idx, int32_t* col_ptr_t, int32_t* row_idx_t, int64_t col_cap,
                                   void* ws, int32_t* status, int sms, cudaStream_t stream);
cudaError_t launch_block_mask_bitmap(const MaskProblem& p, const uint8_t* bitmap, int32_t* row_ptr, int32_t* col_idx,
                                     int32_t* col_ptr_t, int32_t* row_idx_t, int64_t col_cap, void* ws,
                                     int32_t* status, cudaStream_t stream);

// attention problems
struct AttnProblem {
  int64_t N;
  int H, d, block, dtype;
  int64_t row_stride;
  int nq;        // query blocks of `block` rows (rows of the CSR lists per head)
  float scale;
  int block_k;   // rows per key block
  int nk;        // key blocks (rows of the transposed lists per head)
};

// attn_simt.cu (fp32 path and the generic CUDA-core backward)
cudaError_t launch_attn_fwd_simt(const AttnProblem& p, const void* q, const void* k, const void* v,
                                 const int32_t* row_ptr, const int32_t* col_idx, void* o, float* lse,
                                 cudaStream_t stream);
size_t attn_bwd_simt_ws(const AttnProblem& p);
cudaError_t launch_attn_bwd_simt(const AttnProblem& p, const void* q, const void* k, const void* v, const void* o,
                                 const float* lse, const void* dout, const int32_t* row_ptr, const int32_t* col_idx,
                                 const int32_t* col_ptr_t, const int32_t* row_idx_t, void* dq, void* dk, void* dv,
                                 void* ws, cudaStream_t stream);

// attn_fwd_tc.cu (bf16 tcgen05 forward)
cudaError_t launch_attn_fwd_tc(const AttnProblem& p, const void* q, const void* k, const void* v,
                               const int32_t* row_ptr, const int32_t* col_idx, void* o, float* lse, int32_t* status,
                               uint64_t timeout_ns, int sms, cudaStream_t stream);

// attn_bwd_tc.cu (bf16 tcgen05 backward: preprocess, fused dK/dV/dQ, dQ finalize)
size_t attn_bwd_tc_ws(const AttnProblem& p);
cudaError_t launch_attn_bwd_tc(const AttnProblem& p, const void* q, const void* k, const void* v, const void* o,
                               const float* lse, const void* dout, const int32_t* row_ptr, const int32_t* col_idx,
                               const int32_t* col_ptr_t, const int32_t* row_idx_t, void* dq, void* dk, void* dv,
                               void* ws, int32_t* status, uint64_t timeout_ns, int sms, cudaStream_t stream);

// tensor maps (api.cu)
bool encode_tmap_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner_elems, uint64_t rows,
                         uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows);

}  // namespace ut
