// Block-sparse attention on the CUDA cores in fp32 arithmetic (Sec. 3.3).
//
// This is the path for fp32 inputs (whose tolerance rules out tf32 tensor
// cores) and the generic backward.  One thread owns one query row (forward,
// dQ) or one key row (dK, dV); the partner tile is staged in shared memory in
// chunks of 32 rows and read by broadcast.  Rows of the owned tile are stored
// transposed ([D][b]) so that each thread reads its own column bank-conflict
// free.
//
//   attn_fwd_simt_kernel   online softmax over the listed key blocks; O, LSE.
//   attn_bwd_pre_kernel    D_r = dO_r . O_r.
//   attn_bwd_dq_kernel     dQ_r = scale * sum_k P_rk (dO_r . V_k - D_r) K_k.
//   attn_bwd_dkdv_kernel   per key row over the transposed lists (query
//                          blocks that listed this key block): dV_k = sum_r
//                          P_rk dO_r (pass 0) and dK_k = scale * sum_r dS_rk
//                          Q_r (pass 1).
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kChunkRows = 32;

template <typename T>
UT_DEV float ld_elem(const T* p);
template <>
UT_DEV float ld_elem<float>(const float* p) { return *p; }
template <>
UT_DEV float ld_elem<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <typename T>
UT_DEV void st_elem(T* p, float v);
template <>
UT_DEV void st_elem<float>(float* p, float v) { *p = v; }
template <>
UT_DEV void st_elem<__nv_bfloat16>(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

struct SimtArgs {
  const void* q; const void* k; const void* v; const void* o; const void* dout;
  const float* lse; const float* Dsum;
  const int32_t* ptr; const int32_t* idx;   // CSR (fwd, dq) or CSC (dkdv)
  void* out0; float* out_lse;
  int64_t N, rs; int H, b, nq; float scale;
};

// Stage rows [r0, r0+cnt) of head h into dst[row][D] (fp32), zero beyond cnt.
template <typename T, int D>
UT_DEV void stage_rows(float* dst, const T* src, int64_t r0, int cnt, int rows, int h, int64_t rs) {
  for (int x = threadIdx.x; x < rows * D; x += blockDim.x) {
    int r = x / D, e = x % D;
    dst[x] = r < cnt ? ld_elem<T>(src + (r0 + r) * rs + (int64_t)h * D + e) : 0.f;
  }
}
// Stage rows transposed: dst[e][row] with leading dimension ld.
template <typename T, int D>
UT_DEV void stage_rows_T(float* dst, const T* src, int64_t r0, int cnt, int ld, int h, int64_t rs) {
  for (int x = threadIdx.x; x < ld * D; x += blockDim.x) {
    int r = x / D, e = x % D;
    dst[e * ld + r] = r < cnt ? ld_elem<T>(src + (r0 + r) * rs + (int64_t)h * D + e) : 0.f;
  }
}

template <typename T, int D>
__global__ void attn_fwd_simt_kernel(SimtArgs a) {
  extern __shared__ float sm[];
  const int b = a.b, t = threadIdx.x, i = blockIdx.x, h = blockIdx.y;
  float* qT = sm;                       // [D][b]
  float* ks = qT + D * b;               // [32][D]
  float* vs = ks + kChunkRows * D;      // [32][D]
  const int64_t r0 = (int64_t)i * b;
  const int nvq = (int)min((int64_t)b, a.N - r0);
  const T* Q = static_cast<const T*>(a.q);
  const T* K = static_cast<const T*>(a.k);
  const T* V = static_cast<const T*>(a.v);
  stage_rows_T<T, D>(qT, Q, r0, nvq, b, h, a.rs);
  float o[D];
#pragma unroll
  for (int e = 0; e < D; ++e) o[e] = 0.f;
  float m = -INFINITY, l = 0.f;
  const int row = h * a.nq + i;
  for (int p = a.ptr[row]; p < a.ptr[row + 1]; ++p) {
    const int64_t c0 = (int64_t)a.idx[p] * b;
    const int nvk = (int)min((int64_t)b, a.N - c0);
    for (int cc = 0; cc < nvk; cc += kChunkRows) {
      const int cnt = min(kChunkRows, nvk - cc);
      __syncthreads();
      stage_rows<T, D>(ks, K, c0 + cc, cnt, kChunkRows, h, a.rs);
      stage_rows<T, D>(vs, V, c0 + cc, cnt, kChunkRows, h, a.rs);
      __syncthreads();
      for (int c = 0; c < cnt; ++c) {
        float s = 0.f;
#pragma unroll 16
        for (int e = 0; e < D; ++e) s = fmaf(qT[e * b + t], ks[c * D + e], s);
        s *= a.scale;
        const float mn = fmaxf(m, s);
        const float alpha = expf(m - mn);
        const float pr = expf(s - mn);
        l = l * alpha + pr;
#pragma unroll
        for (int e = 0; e < D; ++e) o[e] = fmaf(o[e], alpha, pr * vs[c * D + e]);
        m = mn;
      }
    }
  }
  if (t < nvq) {
    T* O = static_cast<T*>(a.out0) + (r0 + t) * a.rs + (int64_t)h * D;
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
    for (int e = 0; e < D; ++e) st_elem<T>(O + e, o[e] * inv);
    a.out_lse[(int64_t)h * a.N + r0 + t] = l > 0.f ? m + logf(l) : -INFINITY;
  }
}

template <typename T, int D>
__global__ void attn_bwd_pre_kernel(SimtArgs a) {
  const int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= a.N * a.H) return;
  const int64_t r = x / a.H;
  const int h = (int)(x % a.H);
  const T* O = static_cast<const T*>(a.o) + r * a.rs + (int64_t)h * D;
  const T* dO = static_cast<const T*>(a.dout) + r * a.rs + (int64_t)h * D;
  float s = 0.f;
  for (int e = 0; e < D; ++e) s = fmaf(ld_elem<T>(O + e), ld_elem<T>(dO + e), s);
  const_cast<float*>(a.Dsum)[(int64_t)h * a.N + r] = s;
}

template <typename T, int D>
__global__ void attn_bwd_dq_kernel(SimtArgs a) {
  extern __shared__ float sm[];
  const int b = a.b, t = threadIdx.x, i = blockIdx.x, h = blockIdx.y;
  float* qT = sm;                        // [D][b]
  float* doT = qT + D * b;               // [D][b]
  float* ks = doT + D * b;               // [32][D]
  float* vs = ks + kChunkRows * D;       // [32][D]
  const int64_t r0 = (int64_t)i * b;
  const int nvq = (int)min((int64_t)b, a.N - r0);
  const T* Q = static_cast<const T*>(a.q);
  const T* K = static_cast<const T*>(a.k);
  const T* V = static_cast<const T*>(a.v);
  const T* dO = static_cast<const T*>(a.dout);
  stage_rows_T<T, D>(qT, Q, r0, nvq, b, h, a.rs);
  stage_rows_T<T, D>(doT, dO, r0, nvq, b, h, a.rs);
  const float lse = t < nvq ? a.lse[(int64_t)h * a.N + r0 + t] : 0.f;
  const float Dr = t < nvq ? a.Dsum[(int64_t)h * a.N + r0 + t] : 0.f;
  float dq[D];
#pragma unroll
  for (int e = 0; e < D; ++e) dq[e] = 0.f;
  const int row = h * a.nq + i;
  for (int p = a.ptr[row]; p < a.ptr[row + 1]; ++p) {
    const int64_t c0 = (int64_t)a.idx[p] * b;
    const int nvk = (int)min((int64_t)b, a.N - c0);
    for (int cc = 0; cc < nvk; cc += kChunkRows) {
      const int cnt = min(kChunkRows, nvk - cc);
      __syncthreads();
      stage_rows<T, D>(ks, K, c0 + cc, cnt, kChunkRows, h, a.rs);
      stage_rows<T, D>(vs, V, c0 + cc, cnt, kChunkRows, h, a.rs);
      __syncthreads();
      for (int c = 0; c < cnt; ++c) {
        float s = 0.f, dp = 0.f;
#pragma unroll 16
        for (int e = 0; e < D; ++e) {
          s = fmaf(qT[e * b + t], ks[c * D + e], s);
          dp = fmaf(doT[e * b + t], vs[c * D + e], dp);
        }
        const float pr = expf(s * a.scale - lse);
        const float ds = pr * (dp - Dr) * a.scale;
#pragma unroll
        for (int e = 0; e < D; ++e) dq[e] = fmaf(ds, ks[c * D + e], dq[e]);
      }
    }
  }
  if (t < nvq) {
    T* out = static_cast<T*>(a.out0) + (r0 + t) * a.rs + (int64_t)h * D;
#pragma unroll
    for (int e = 0; e < D; ++e) st_elem<T>(out + e, dq[e]);
  }
}

// PASS 0: dV, PASS 1: dK.  ptr/idx are the transposed lists (per key block).
template <typename T, int D, int PASS>
__global__ void attn_bwd_dkdv_kernel(SimtArgs a) {
  extern __shared__ float sm[];
  const int b = a.b, t = threadIdx.x, j = blockIdx.x, h = blockIdx.y;
  float* kT = sm;                        // [D][b]
  float* vT = kT + D * b;                // [D][b]
  float* qs = vT + D * b;                // [32][D]
  float* dos = qs + kChunkRows * D;      // [32][D]
  float* ls = dos + kChunkRows * D;      // [32]
  float* Ds = ls + kChunkRows;           // [32]
  const int64_t c0 = (int64_t)j * b;
  const int nvk = (int)min((int64_t)b, a.N - c0);
  const T* Q = static_cast<const T*>(a.q);
  const T* K = static_cast<const T*>(a.k);
  const T* V = static_cast<const T*>(a.v);
  const T* dO = static_cast<const T*>(a.dout);
  stage_rows_T<T, D>(kT, K, c0, nvk, b, h, a.rs);
  if (PASS == 1) stage_rows_T<T, D>(vT, V, c0, nvk, b, h, a.rs);
  float acc[D];
#pragma unroll
  for (int e = 0; e < D; ++e) acc[e] = 0.f;
  const int col = h * a.nq + j;
  for (int p = a.ptr[col]; p < a.ptr[col + 1]; ++p) {
    const int64_t q0 = (int64_t)a.idx[p] * b;
    const int nvq = (int)min((int64_t)b, a.N - q0);
    for (int cc = 0; cc < nvq; cc += kChunkRows) {
      const int cnt = min(kChunkRows, nvq - cc);
      __syncthreads();
      stage_rows<T, D>(qs, Q, q0 + cc, cnt, kChunkRows, h, a.rs);
      stage_rows<T, D>(dos, dO, q0 + cc, cnt, kChunkRows, h, a.rs);
      for (int x = threadIdx.x; x < kChunkRows; x += blockDim.x) {
        ls[x] = x < cnt ? a.lse[(int64_t)h * a.N + q0 + cc + x] : 0.f;
        Ds[x] = x < cnt ? a.Dsum[(int64_t)h * a.N + q0 + cc + x] : 0.f;
      }
      __syncthreads();
      for (int r = 0; r < cnt; ++r) {
        float s = 0.f, dp = 0.f;
#pragma unroll 16
        for (int e = 0; e < D; ++e) {
          s = fmaf(qs[r * D + e], kT[e * b + t], s);
          if (PASS == 1) dp = fmaf(dos[r * D + e], vT[e * b + t], dp);
        }
        const float pr = expf(s * a.scale - ls[r]);
        if (PASS == 0) {
#pragma unroll
          for (int e = 0; e < D; ++e) acc[e] = fmaf(pr, dos[r * D + e], acc[e]);
        } else {
          const float ds = pr * (dp - Ds[r]) * a.scale;
#pragma unroll
          for (int e = 0; e < D; ++e) acc[e] = fmaf(ds, qs[r * D + e], acc[e]);
        }
      }
    }
  }
  if (t < nvk) {
    T* out = static_cast<T*>(a.out0) + (c0 + t) * a.rs + (int64_t)h * D;
#pragma unroll
    for (int e = 0; e < D; ++e) st_elem<T>(out + e, acc[e]);
  }
}

// ----------------------------------------------------------------- launchers
template <typename F>
static cudaError_t launch_smem(F kern, dim3 grid, int threads, size_t smem, SimtArgs a, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<grid, threads, smem, s>>>(a);
  return cudaGetLastError();
}

template <typename T, int D>
static cudaError_t fwd_impl(const AttnProblem& p, SimtArgs a, cudaStream_t s) {
  size_t smem = ((size_t)D * p.block + 2 * kChunkRows * D) * sizeof(float);
  return launch_smem(attn_fwd_simt_kernel<T, D>, dim3(p.nq, p.H), p.block, smem, a, s);
}

cudaError_t launch_attn_fwd_simt(const AttnProblem& p, const void* q, const void* k, const void* v,
                                 const int32_t* row_ptr, const int32_t* col_idx, void* o, float* lse,
                                 cudaStream_t stream) {
  if (p.nq == 0) return cudaSuccess;
  SimtArgs a{};
  a.q = q; a.k = k; a.v = v; a.ptr = row_ptr; a.idx = col_idx; a.out0 = o; a.out_lse = lse;
  a.N = p.N; a.rs = p.row_stride; a.H = p.H; a.b = p.block; a.nq = p.nq; a.scale = p.scale;
  if (p.dtype == UT_F32) return p.d == 64 ? fwd_impl<float, 64>(p, a, stream) : fwd_impl<float, 128>(p, a, stream);
  return p.d == 64 ? fwd_impl<__nv_bfloat16, 64>(p, a, stream) : fwd_impl<__nv_bfloat16, 128>(p, a, stream);
}

size_t attn_bwd_simt_ws(const AttnProblem& p) { return (size_t)p.H * p.N * sizeof(float); }

template <typename T, int D>
static cudaError_t bwd_impl(const AttnProblem& p, SimtArgs a, const int32_t* rp, const int32_t* ci,
                            const int32_t* cp, const int32_t* ri, void* dq, void* dk, void* dv, cudaStream_t s) {
  const int64_t NH = p.N * p.H;
  attn_bwd_pre_kernel<T, D><<<(unsigned)((NH + 255) / 256), 256, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  SimtArgs aq = a;
  aq.ptr = rp; aq.idx = ci; aq.out0 = dq;
  size_t smem_q = ((size_t)2 * D * p.block + 2 * kChunkRows * D) * sizeof(float);
  e = launch_smem(attn_bwd_dq_kernel<T, D>, dim3(p.nq, p.H), p.block, smem_q, aq, s);
  if (e != cudaSuccess) return e;
  size_t smem_kv = ((size_t)2 * D * p.block + 2 * kChunkRows * D + 2 * kChunkRows) * sizeof(float);
  SimtArgs av = a;
  av.ptr = cp; av.idx = ri; av.out0 = dv;
  e = launch_smem(attn_bwd_dkdv_kernel<T, D, 0>, dim3(p.nq, p.H), p.block, smem_kv, av, s);
  if (e != cudaSuccess) return e;
  SimtArgs ak = a;
  ak.ptr = cp; ak.idx = ri; ak.out0 = dk;
  return launch_smem(attn_bwd_dkdv_kernel<T, D, 1>, dim3(p.nq, p.H), p.block, smem_kv, ak, s);
}

cudaError_t launch_attn_bwd_simt(const AttnProblem& p, const void* q, const void* k, const void* v, const void* o,
                                 const float* lse, const void* dout, const int32_t* row_ptr, const int32_t* col_idx,
                                 const int32_t* col_ptr_t, const int32_t* row_idx_t, void* dq, void* dk, void* dv,
                                 void* ws, cudaStream_t stream) {
  if (p.nq == 0) return cudaSuccess;
  SimtArgs a{};
  a.q = q; a.k = k; a.v = v; a.o = o; a.dout = dout; a.lse = lse; a.Dsum = static_cast<float*>(ws);
  a.N = p.N; a.rs = p.row_stride; a.H = p.H; a.b = p.block; a.nq = p.nq; a.scale = p.scale;
  if (p.dtype == UT_F32)
    return p.d == 64 ? bwd_impl<float, 64>(p, a, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk, dv, stream)
                     : bwd_impl<float, 128>(p, a, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk, dv, stream);
  return p.d == 64 ? bwd_impl<__nv_bfloat16, 64>(p, a, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk, dv, stream)
                   : bwd_impl<__nv_bfloat16, 128>(p, a, row_ptr, col_idx, col_ptr_t, row_idx_t, dq, dk, dv, stream);
}

}  // namespace ut
