// Background Token Dropping (Sec. 3.2) and the scatter back to the canvas.
//
//   fg_count_kernel   per 4096-token chunk: number of foreground tokens.
//   fg_index_kernel   per chunk: exclusive prefix of the chunk counts, then a
//                     block-wide ballot scan writes the ascending canvas
//                     positions idx[n] (the retained tokens' RoPE indices).
//   fg_gather_kernel  Xc[n] = X[idx[n]] for every listed tensor: one warp per
//                     row, 16-byte vector loads/stores, persistent grid.
//   fg_scatter_*      Y[idx[n]] = Xc[n]; background rows kept, zeroed or filled.
//
// All three compaction launches are HBM-bound except the first two, which
// touch only the T-byte mask and the 4N-byte index list.
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kChunk = 4096;          // canvas tokens per count/index CTA
constexpr int kIdxThreads = 256;      // 16 tokens per thread

__global__ void __launch_bounds__(kIdxThreads) fg_count_kernel(const uint8_t* __restrict__ mask, int64_t T,
                                                               int32_t* __restrict__ counts) {
  const int64_t base = (int64_t)blockIdx.x * kChunk + (int64_t)threadIdx.x * 16;
  int c = 0;
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    int64_t t = base + e;
    if (t < T) c += mask[t] != 0;
  }
  __shared__ int red[kIdxThreads / 32];
  for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < kIdxThreads / 32; ++w) s += red[w];
    counts[blockIdx.x] = s;
  }
}

__global__ void __launch_bounds__(kIdxThreads) fg_index_kernel(const uint8_t* __restrict__ mask, int64_t T,
                                                               const int32_t* __restrict__ counts,
                                                               int32_t n_chunks, int32_t* __restrict__ idx,
                                                               int64_t capacity, int32_t* __restrict__ n_out,
                                                               int32_t* status) {
  __shared__ int s_prefix;
  __shared__ int s_total;
  __shared__ int warp_sums[kIdxThreads / 32];
  const int tid = threadIdx.x;
  // Exclusive prefix of the chunk counts before this chunk (and the total).
  {
    int pre = 0, tot = 0;
    for (int c = tid; c < n_chunks; c += kIdxThreads) {
      int v = counts[c];
      tot += v;
      if (c < (int)blockIdx.x) pre += v;
    }
    for (int o = 16; o; o >>= 1) {
      pre += __shfl_xor_sync(0xffffffffu, pre, o);
      tot += __shfl_xor_sync(0xffffffffu, tot, o);
    }
    __shared__ int rp[kIdxThreads / 32], rt[kIdxThreads / 32];
    if ((tid & 31) == 0) { rp[tid >> 5] = pre; rt[tid >> 5] = tot; }
    __syncthreads();
    if (tid == 0) {
      int a = 0, b = 0;
      for (int w = 0; w < kIdxThreads / 32; ++w) { a += rp[w]; b += rt[w]; }
      s_prefix = a;
      s_total = b;
    }
    __syncthreads();
  }
  // This thread's 16 tokens: local count, then a block-wide exclusive scan.
  const int64_t base = (int64_t)blockIdx.x * kChunk + (int64_t)tid * 16;
  uint32_t bits = 0;
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    int64_t t = base + e;
    if (t < T && mask[t] != 0) bits |= 1u << e;
  }
  int mine = __popc(bits);
  int incl = mine;
  const int lane = tid & 31, w = tid >> 5;
  for (int o = 1; o < 32; o <<= 1) {
    int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_sums[w] = incl;
  __syncthreads();
  int wpre = 0;
  for (int i = 0; i < w; ++i) wpre += warp_sums[i];
  int64_t pos = (int64_t)s_prefix + wpre + incl - mine;
  bool overflow = false;
  while (bits) {
    int e = __ffs(bits) - 1;
    bits &= bits - 1;
    if (pos < capacity) idx[pos] = (int32_t)(base + e);
    else overflow = true;
    ++pos;
  }
  if (overflow) set_status(status, UT_ERR_CAPACITY);
  if (blockIdx.x == 0 && tid == 0) *n_out = s_total;
}

struct TensorList {
  const uint8_t* src[8];
  uint8_t* dst[8];
};

// One warp per compacted row; every lane moves 16-byte vectors.  The row's
// loads are all issued before its stores so that each warp keeps
// row_bytes / 16 / 32 vectors in flight.
template <int kVecPerLane>
__global__ void __launch_bounds__(256) fg_gather_kernel(const __grid_constant__ TensorList tl, int n_tensors, const int32_t* __restrict__ idx,
                                                        const int32_t* __restrict__ n_dev, int64_t capacity,
                                                        int64_t row_bytes) {
  const int64_t N = min((int64_t)*n_dev, capacity);
  const int64_t nvec = row_bytes >> 4;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int lane = threadIdx.x & 31;
  for (int64_t n = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); n < N; n += warps) {
    const int64_t t = idx[n];
    for (int ti = 0; ti < n_tensors; ++ti) {
      const uint8_t* s = tl.src[ti] + t * row_bytes;
      uint8_t* d = tl.dst[ti] + n * row_bytes;
      for (int64_t v0 = 0; v0 < nvec; v0 += 32 * kVecPerLane) {
        uint4 r[kVecPerLane];
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) r[u] = ld_nc_v4(s + (v << 4));
        }
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) st_v4(d + (v << 4), r[u]);
        }
      }
    }
  }
}

// KEEP: one warp per compacted row, dst[idx[n]] = src[n].
template <int kVecPerLane>
__global__ void __launch_bounds__(256) fg_scatter_keep_kernel(const __grid_constant__ TensorList tl, int n_tensors,
                                                              const int32_t* __restrict__ idx, int64_t N,
                                                              int64_t row_bytes) {
  const int64_t nvec = row_bytes >> 4;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int lane = threadIdx.x & 31;
  for (int64_t n = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); n < N; n += warps) {
    const int64_t t = idx[n];
    for (int ti = 0; ti < n_tensors; ++ti) {
      const uint8_t* s = tl.src[ti] + n * row_bytes;
      uint8_t* d = tl.dst[ti] + t * row_bytes;
      for (int64_t v0 = 0; v0 < nvec; v0 += 32 * kVecPerLane) {
        uint4 r[kVecPerLane];
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) r[u] = ld_nc_v4(s + (v << 4));
        }
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) st_v4(d + (v << 4), r[u]);
        }
      }
    }
  }
}

// ZERO / FILL: one warp per canvas row; a binary search in the ascending idx
// list tells whether row t is foreground (and which compacted row it is).
template <int kVecPerLane>
__global__ void __launch_bounds__(256) fg_scatter_full_kernel(const __grid_constant__ TensorList tl, int n_tensors,
                                                              const int32_t* __restrict__ idx, int64_t N, int64_t T,
                                                              int64_t row_bytes, const uint8_t* __restrict__ fill) {
  const int64_t nvec = row_bytes >> 4;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int lane = threadIdx.x & 31;
  for (int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); t < T; t += warps) {
    int64_t lo = 0, hi = N;  // first n with idx[n] >= t
    while (lo < hi) {
      int64_t mid = (lo + hi) >> 1;
      if (idx[mid] < t) lo = mid + 1;
      else hi = mid;
    }
    const bool fg = lo < N && idx[lo] == t;
    for (int ti = 0; ti < n_tensors; ++ti) {
      uint8_t* d = tl.dst[ti] + t * row_bytes;
      const uint8_t* s = fg ? tl.src[ti] + lo * row_bytes : fill;
      for (int64_t v0 = 0; v0 < nvec; v0 += 32 * kVecPerLane) {
        uint4 r[kVecPerLane];
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) r[u] = s ? ld_nc_v4(s + (v << 4)) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < kVecPerLane; ++u) {
          int64_t v = v0 + u * 32 + lane;
          if (v < nvec) st_v4(d + (v << 4), r[u]);
        }
      }
    }
  }
}

// ----------------------------------------------------------------- launchers
size_t fg_compact_ws(int64_t T) {
  int64_t chunks = (T + kChunk - 1) / kChunk;
  return (size_t)(chunks > 0 ? chunks : 1) * sizeof(int32_t);
}

static int copy_grid(int64_t rows, int sms) {
  int64_t per_sm = 8;  // 8 CTAs of 8 warps resident per SM
  int64_t want = (rows + 7) / 8;
  int64_t cap = (int64_t)sms * per_sm;
  int64_t g = want < cap ? want : cap;
  return (int)(g > 0 ? g : 1);
}

cudaError_t launch_fg_compact(const uint8_t* mask, int64_t T, int n_tensors, const void* const* src,
                              void* const* dst, int64_t row_bytes, int64_t capacity, int32_t* idx, int32_t* n_out,
                              void* ws, int32_t* status, int sms, cudaStream_t stream) {
  int32_t* counts = static_cast<int32_t*>(ws);
  int n_chunks = (int)((T + kChunk - 1) / kChunk);
  if (n_chunks == 0) return cudaMemsetAsync(n_out, 0, sizeof(int32_t), stream);
  fg_count_kernel<<<n_chunks, kIdxThreads, 0, stream>>>(mask, T, counts);
  fg_index_kernel<<<n_chunks, kIdxThreads, 0, stream>>>(mask, T, counts, n_chunks, idx, capacity, n_out, status);
  TensorList tl{};
  for (int i = 0; i < n_tensors; ++i) {
    tl.src[i] = static_cast<const uint8_t*>(src[i]);
    tl.dst[i] = static_cast<uint8_t*>(dst[i]);
  }
  int64_t rows = T < capacity ? T : capacity;
  int grid = copy_grid(rows, sms);
  if (row_bytes >= 16 * 32 * 12)
    fg_gather_kernel<12><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, n_out, capacity, row_bytes);
  else
    fg_gather_kernel<4><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, n_out, capacity, row_bytes);
  return cudaGetLastError();
}

cudaError_t launch_fg_scatter(const int32_t* idx, int64_t N, int n_tensors, const void* const* src, void* const* dst,
                              int64_t row_bytes, int bg_mode, const void* fill, int64_t T, int sms,
                              cudaStream_t stream) {
  TensorList tl{};
  for (int i = 0; i < n_tensors; ++i) {
    tl.src[i] = static_cast<const uint8_t*>(src[i]);
    tl.dst[i] = static_cast<uint8_t*>(dst[i]);
  }
  const bool big = row_bytes >= 16 * 32 * 12;
  if (bg_mode == UT_BG_KEEP) {
    if (N == 0) return cudaSuccess;
    int grid = copy_grid(N, sms);
    if (big) fg_scatter_keep_kernel<12><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, N, row_bytes);
    else fg_scatter_keep_kernel<4><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, N, row_bytes);
  } else {
    if (T == 0) return cudaSuccess;
    const uint8_t* f = bg_mode == UT_BG_FILL ? static_cast<const uint8_t*>(fill) : nullptr;
    int grid = copy_grid(T, sms);
    if (big) fg_scatter_full_kernel<12><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, N, T, row_bytes, f);
    else fg_scatter_full_kernel<4><<<grid, 256, 0, stream>>>(tl, n_tensors, idx, N, T, row_bytes, f);
  }
  return cudaGetLastError();
}

}  // namespace ut
