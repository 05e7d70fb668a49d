// Block mask M_c as key-block lists (Sec. 3.3).
//
// Top-K mode:
//   block_pool_kernel    pool(Q) over blocks of b_q rows, pool(K) over blocks
//                        of b_kv rows: fp32 mean over the valid rows of each
//                        block, every head at once (one CTA per block).
//   score_select_kernel  S_c[i, :] = pool(Q)_i . pool(K)_j in fp32 for R query
//                        blocks of one head, then per row an exact radix
//                        select of the K_rho-th largest score (4 passes of 8
//                        bits over order-preserving keys); equal scores go to
//                        the smaller key-block index.  Writes the ascending
//                        list and the dense [H, N_q, N_k] bitmap row.
// Both modes:
//   bitmap_count_kernel  entries per row (or per column for the transpose),
//   scan_kernel          exclusive prefix -> row_ptr / col_ptr,
//   bitmap_fill_kernel   ascending lists by warp ballot.
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kPoolThreads = 256;
constexpr int kSelThreads = 256;
constexpr int kSelMaxRows = 16;

template <typename T>
struct Vec8;
template <>
struct Vec8<__nv_bfloat16> {
  static constexpr int kElems = 8;
  UT_DEV static void load(const __nv_bfloat16* p, float* f) {
    uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float2 x = __bfloat1622float2(h[e]);
      f[2 * e] = x.x;
      f[2 * e + 1] = x.y;
    }
  }
};
template <>
struct Vec8<float> {
  static constexpr int kElems = 4;
  UT_DEV static void load(const float* p, float* f) {
    float4 u = *reinterpret_cast<const float4*>(p);
    f[0] = u.x; f[1] = u.y; f[2] = u.z; f[3] = u.w;
  }
};

// grid (max(nq, nk), 2): blockIdx.y selects Q (0, blocks of bq rows) or K (1,
// blocks of bk rows).  out: pooled Q [H][nq][d], then pooled K [H][nk][d].
template <typename T>
__global__ void __launch_bounds__(kPoolThreads) block_pool_kernel(const T* __restrict__ q, const T* __restrict__ k,
                                                                  int64_t N, int H, int d, int64_t row_stride,
                                                                  int bq, int nq, int bk, int nk,
                                                                  float* __restrict__ out) {
  constexpr int E = Vec8<T>::kElems;
  const bool is_k = blockIdx.y == 1;
  const T* x = is_k ? k : q;
  const int block = is_k ? bk : bq, nb = is_k ? nk : nq;
  const int i = blockIdx.x;
  if (i >= nb) return;
  float* base = is_k ? out + (size_t)H * nq * d : out;
  const int64_t r0 = (int64_t)i * block;
  const int64_t r1 = min(N, r0 + block);
  const int cols = H * d;
  const float inv_cnt = 1.0f / (float)(r1 - r0);
  for (int ch = threadIdx.x; ch * E < cols; ch += kPoolThreads) {
    float acc[E];
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = 0.f;
    for (int64_t r = r0; r < r1; ++r) {
      float f[E];
      Vec8<T>::load(x + r * row_stride + (int64_t)ch * E, f);
#pragma unroll
      for (int e = 0; e < E; ++e) acc[e] += f[e];
    }
    const int c0 = ch * E;
    const int h = c0 / d, e0 = c0 % d;
    float* dst = base + ((int64_t)h * nb + i) * d + e0;
#pragma unroll
    for (int e = 0; e < E; ++e) dst[e] = __fdiv_rn(acc[e], (float)(r1 - r0));
    (void)inv_cnt;
  }
}

UT_DEV uint32_t order_key(float s) {
  s = s + 0.0f;  // -0 -> +0
  uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// grid (H, ceil(nq / R)); dynamic smem: R*d + R*nk floats + 8 warps * 256 ints.
// Rows are query blocks (nq per head), columns key blocks (nk).
__global__ void __launch_bounds__(kSelThreads) score_select_kernel(const float* __restrict__ pooled, int H, int d,
                                                                   int nq, int nk, int R, int k_rho,
                                                                   int32_t* __restrict__ col_idx,
                                                                   uint8_t* __restrict__ bitmap) {
  extern __shared__ float smem[];
  float* pq = smem;                       // [R][d]
  float* sc = smem + R * d;               // [R][nk]
  uint32_t* hist = reinterpret_cast<uint32_t*>(sc + R * nk);  // [8][256]
  const int h = blockIdx.x;
  const int i0 = blockIdx.y * R;
  const int rows = min(R, nq - i0);
  const float* PQ = pooled + ((int64_t)h * nq) * d;
  const float* PK = pooled + (int64_t)H * nq * d + ((int64_t)h * nk) * d;
  for (int t = threadIdx.x; t < rows * d; t += kSelThreads) pq[t] = PQ[(int64_t)i0 * d + t];
  __syncthreads();
  // two key blocks per thread and 16-byte loads of the pooled query rows: one
  // shared load feeds eight FMAs (the sums are accumulated in the same order
  // as one column at a time)
  for (int j0 = threadIdx.x; j0 < nk; j0 += 2 * kSelThreads) {
    const int j1 = j0 + kSelThreads;
    const bool has1 = j1 < nk;
    float acc0[kSelMaxRows], acc1[kSelMaxRows];
#pragma unroll
    for (int r = 0; r < kSelMaxRows; ++r) acc0[r] = acc1[r] = 0.f;
    const float* k0 = PK + (int64_t)j0 * d;
    const float* k1 = PK + (int64_t)(has1 ? j1 : j0) * d;
    for (int e = 0; e < d; e += 4) {
      const float4 a = *reinterpret_cast<const float4*>(k0 + e);
      const float4 b = *reinterpret_cast<const float4*>(k1 + e);
#pragma unroll
      for (int r = 0; r < kSelMaxRows; ++r) {
        if (r < rows) {
          const float4 p = *reinterpret_cast<const float4*>(pq + r * d + e);
          acc0[r] = fmaf(p.x, a.x, acc0[r]);
          acc0[r] = fmaf(p.y, a.y, acc0[r]);
          acc0[r] = fmaf(p.z, a.z, acc0[r]);
          acc0[r] = fmaf(p.w, a.w, acc0[r]);
          acc1[r] = fmaf(p.x, b.x, acc1[r]);
          acc1[r] = fmaf(p.y, b.y, acc1[r]);
          acc1[r] = fmaf(p.z, b.z, acc1[r]);
          acc1[r] = fmaf(p.w, b.w, acc1[r]);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < kSelMaxRows; ++r)
      if (r < rows) {
        sc[r * nk + j0] = acc0[r];
        if (has1) sc[r * nk + j1] = acc1[r];
      }
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t* hw = hist + w * 256;
  const uint32_t lt_mask = (1u << lane) - 1u;
  for (int r = w; r < rows; r += kSelThreads / 32) {
    const float* srow = sc + r * nk;
    uint32_t prefix = 0, pmask = 0;
    int k = k_rho;  // rank still to find among keys matching the prefix
    for (int pass = 3; pass >= 0; --pass) {
      const int shift = pass * 8;
      for (int b = lane; b < 256; b += 32) hw[b] = 0;
      __syncwarp();
      for (int j = lane; j < nk; j += 32) {
        uint32_t u = order_key(srow[j]);
        if ((u & pmask) == prefix) atomicAdd(&hw[(u >> shift) & 255u], 1u);
      }
      __syncwarp();
      // lane l owns bins 255-8l .. 248-8l (descending); find the bin holding rank k.
      uint32_t cnt[8];
      uint32_t local = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        cnt[q] = hw[255 - 8 * lane - q];
        local += cnt[q];
      }
      uint32_t incl = local;
      for (int o = 1; o < 32; o <<= 1) {
        uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const uint32_t before = incl - local;
      const bool here = before < (uint32_t)k && (uint32_t)k <= incl;
      uint32_t digit = 0, above = 0;
      if (here) {
        uint32_t c = before;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (c + cnt[q] >= (uint32_t)k) {
            digit = 255 - 8 * lane - q;
            above = c;
            break;
          }
          c += cnt[q];
        }
      }
      const int src = __ffs(__ballot_sync(0xffffffffu, here)) - 1;
      digit = __shfl_sync(0xffffffffu, digit, src);
      above = __shfl_sync(0xffffffffu, above, src);
      k -= (int)above;
      prefix |= digit << shift;
      pmask |= 0xFFu << shift;
      __syncwarp();
    }
    // prefix = the K_rho-th largest key; take all larger keys and the first k equal ones.
    const int row = h * nq + i0 + r;
    int32_t* out = col_idx + (int64_t)row * k_rho;
    uint8_t* brow = bitmap + (int64_t)row * nk;
    int n_sel = 0, n_eq = 0;
    for (int j0 = 0; j0 < nk; j0 += 32) {
      const int j = j0 + lane;
      uint32_t u = j < nk ? order_key(srow[j]) : 0u;
      const bool valid = j < nk;
      const bool gt = valid && u > prefix;
      const bool eq = valid && u == prefix;
      const uint32_t eqb = __ballot_sync(0xffffffffu, eq);
      const int eq_rank = n_eq + __popc(eqb & lt_mask);
      const bool sel = gt || (eq && eq_rank < k);
      const uint32_t selb = __ballot_sync(0xffffffffu, sel);
      if (sel) out[n_sel + __popc(selb & lt_mask)] = j;
      if (valid) brow[j] = sel ? 1 : 0;
      n_sel += __popc(selb);
      n_eq += __popc(eqb);
    }
  }
}

__global__ void fill_uniform_rowptr_kernel(int32_t* row_ptr, int n_rows, int k) {
  int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r <= n_rows) row_ptr[r] = r * k;
}

// One warp per line.  Line l = (h, a): a row i of [H][nq][nk] (transposed = 0)
// or a column j (transposed = 1).
__global__ void bitmap_count_kernel(const uint8_t* __restrict__ bm, int H, int nq, int nk, int transposed,
                                    int32_t* __restrict__ counts) {
  const int n_lines = transposed ? nk : nq;
  const int line = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (line >= H * n_lines) return;
  const int h = line / n_lines, a = line % n_lines;
  const int len = transposed ? nq : nk;
  const int lane = threadIdx.x & 31;
  int c = 0;
  for (int b = lane; b < len; b += 32) {
    uint8_t v = transposed ? bm[((int64_t)h * nq + b) * nk + a] : bm[((int64_t)h * nq + a) * nk + b];
    c += v != 0;
  }
  for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) counts[line] = c;
}

// Single CTA exclusive scan of n counts into ptr[0..n].
__global__ void __launch_bounds__(1024) scan_kernel(const int32_t* __restrict__ counts, int n,
                                                    int32_t* __restrict__ ptr) {
  __shared__ int64_t warp_tot[32];
  const int tid = threadIdx.x;
  const int per = (n + 1023) / 1024;
  const int a = min(n, tid * per), b = min(n, a + per);
  int64_t local = 0;
  for (int t = a; t < b; ++t) local += counts[t];
  int64_t incl = local;
  const int lane = tid & 31, w = tid >> 5;
  for (int o = 1; o < 32; o <<= 1) {
    int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_tot[w] = incl;
  __syncthreads();
  int64_t wpre = 0;
  for (int i = 0; i < w; ++i) wpre += warp_tot[i];
  int64_t run = wpre + incl - local;
  for (int t = a; t < b; ++t) {
    ptr[t] = (int32_t)run;
    run += counts[t];
  }
  if (tid == 1023) ptr[n] = (int32_t)(wpre + incl);
}

__global__ void bitmap_fill_kernel(const uint8_t* __restrict__ bm, int H, int nq, int nk, int transposed,
                                   const int32_t* __restrict__ ptr, int32_t* __restrict__ out, int64_t cap,
                                   int32_t* status) {
  const int n_lines = transposed ? nk : nq;
  const int line = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (line >= H * n_lines) return;
  const int h = line / n_lines, a = line % n_lines;
  const int len = transposed ? nq : nk;
  const int lane = threadIdx.x & 31;
  const uint32_t lt_mask = (1u << lane) - 1u;
  int64_t pos = ptr[line];
  bool overflow = false;
  for (int b0 = 0; b0 < len; b0 += 32) {
    const int b = b0 + lane;
    bool on = false;
    if (b < len) {
      uint8_t v = transposed ? bm[((int64_t)h * nq + b) * nk + a] : bm[((int64_t)h * nq + a) * nk + b];
      on = v != 0;
    }
    const uint32_t bal = __ballot_sync(0xffffffffu, on);
    if (on) {
      int64_t p = pos + __popc(bal & lt_mask);
      if (p < cap) out[p] = b;
      else overflow = true;
    }
    pos += __popc(bal);
  }
  if (__any_sync(0xffffffffu, overflow) && lane == 0) set_status(status, UT_ERR_CAPACITY);
}

// ----------------------------------------------------------------- launchers
static int select_rows(int nk) {
  int r = (64 * 1024) / (nk * 4);
  r = r < 1 ? 1 : r;
  return r > kSelMaxRows ? kSelMaxRows : r;
}

size_t block_mask_ws(const MaskProblem& p, int mode) {
  const size_t H = p.H, nq = p.nq, nk = p.nk, d = p.d;
  size_t counts = (H * (nq > nk ? nq : nk) + 1) * sizeof(int32_t);
  if (mode == UT_MASK_BITMAP) return counts;
  size_t pooled = H * (nq + nk) * d * sizeof(float);
  size_t bitmap = H * nq * nk;
  return pooled + ((bitmap + 255) / 256) * 256 + counts;
}

static cudaError_t csr_from_bitmap(const uint8_t* bm, int H, int nq, int nk, int transposed, int32_t* ptr,
                                   int32_t* out, int64_t cap, int32_t* counts, int32_t* status,
                                   cudaStream_t stream) {
  const int lines = H * (transposed ? nk : nq);
  const int grid = (lines + 7) / 8;
  if (lines == 0) return cudaSuccess;
  bitmap_count_kernel<<<grid, 256, 0, stream>>>(bm, H, nq, nk, transposed, counts);
  scan_kernel<<<1, 1024, 0, stream>>>(counts, lines, ptr);
  bitmap_fill_kernel<<<grid, 256, 0, stream>>>(bm, H, nq, nk, transposed, ptr, out, cap, status);
  return cudaGetLastError();
}

cudaError_t launch_block_mask_topk(const MaskProblem& p, const void* q, const void* k, int k_rho, int32_t* row_ptr,
                                   int32_t* col_idx, int32_t* col_ptr_t, int32_t* row_idx_t, int64_t col_cap,
                                   void* ws, int32_t* status, int sms, cudaStream_t stream) {
  (void)sms;
  const int H = p.H, nq = p.nq, nk = p.nk, d = p.d;
  float* pooled = static_cast<float*>(ws);
  uint8_t* bitmap = reinterpret_cast<uint8_t*>(pooled + (size_t)H * (nq + nk) * d);
  size_t bm_bytes = (((size_t)H * nq * nk + 255) / 256) * 256;
  int32_t* counts = reinterpret_cast<int32_t*>(bitmap + bm_bytes);
  dim3 pg(nq > nk ? nq : nk, 2);
  if (p.dtype == UT_BF16)
    block_pool_kernel<__nv_bfloat16><<<pg, kPoolThreads, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(k), p.N, H, d, p.row_stride, p.block,
        nq, p.block_k, nk, pooled);
  else
    block_pool_kernel<float><<<pg, kPoolThreads, 0, stream>>>(static_cast<const float*>(q),
                                                              static_cast<const float*>(k), p.N, H, d, p.row_stride,
                                                              p.block, nq, p.block_k, nk, pooled);
  const int R = select_rows(nk);
  size_t smem = ((size_t)R * d + (size_t)R * nk) * sizeof(float) + 8 * 256 * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(score_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 sg(H, (nq + R - 1) / R);
  score_select_kernel<<<sg, kSelThreads, smem, stream>>>(pooled, H, d, nq, nk, R, k_rho, col_idx, bitmap);
  fill_uniform_rowptr_kernel<<<(H * nq + 1 + 255) / 256, 256, 0, stream>>>(row_ptr, H * nq, k_rho);
  if (col_ptr_t && row_idx_t) {
    e = csr_from_bitmap(bitmap, H, nq, nk, 1, col_ptr_t, row_idx_t, col_cap, counts, status, stream);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_block_mask_bitmap(const MaskProblem& p, const uint8_t* bitmap, int32_t* row_ptr, int32_t* col_idx,
                                     int32_t* col_ptr_t, int32_t* row_idx_t, int64_t col_cap, void* ws,
                                     int32_t* status, cudaStream_t stream) {
  int32_t* counts = static_cast<int32_t*>(ws);
  cudaError_t e = csr_from_bitmap(bitmap, p.H, p.nq, p.nk, 0, row_ptr, col_idx, col_cap, counts, status, stream);
  if (e != cudaSuccess) return e;
  if (col_ptr_t && row_idx_t)
    e = csr_from_bitmap(bitmap, p.H, p.nq, p.nk, 1, col_ptr_t, row_idx_t, col_cap, counts, status, stream);
  return e;
}

}  // namespace ut
