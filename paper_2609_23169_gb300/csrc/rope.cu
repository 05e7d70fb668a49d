// Rotary position embedding fused into the compaction gather and the
// gradient scatter (Sec. 3.2: every retained token keeps its original RoPE
// index, i.e. its canvas position).
//
//   canvas position t of images of side S (one after another, raster order,
//   after `prefix` text tokens that stay unrotated)
//     -> (image, y, x) = (t' / S^2, (t' mod S^2) / S, t' mod S), t' = t - prefix;
//   head dimension split into three axes; pair p = (x[2p], x[2p+1]) belongs
//   to axis a(p) and turns by pos_a * freq[p], freq = theta^(-2k/d_a) for the
//   k-th pair of its axis (table computed on the host in double precision).
//
//   rope_kernel<.., kGather>      dst[r] = R(t_r) src[t_r]            (Q, K)
//   rope_kernel<.., kScatterKeep> dst[t_r] = R(t_r)^T src[r]          (dQ, dK)
//   rope_kernel<.., kScatterZero> as KeepScatter, other canvas rows = 0
//
// One warp per row, 16-byte vectors, a lane's loads of a row (up to 12) issued
// before any is used.  A vector holds 4 (bf16) or 2 (fp32)
// pairs of one head; with head_dim * elem / 16 dividing 32, a lane meets the
// same pair slot in every head, so it evaluates its pairs' sin/cos once per
// row (library sincosf on an fp32 angle) and rotates all heads with them.
// The arithmetic is a few FMAs per 16 bytes: the kernels stream at HBM speed
// like the plain gather/scatter, which is the point of the fusion (no extra
// pass over Q and K).
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kRopeThreads = 256;
enum RopeMode { kGather = 0, kScatterKeep = 1, kScatterZero = 2 };

struct RopeParams {
  const uint8_t* src[8];
  uint8_t* dst[8];
  float freq[128];       // per pair: theta^(-2k/d_a)
  uint8_t axis[128];     // per pair: 0 image, 1 y, 2 x
};

template <bool kBf16, int kMode, int kVec>
__global__ void __launch_bounds__(kRopeThreads) rope_kernel(const __grid_constant__ RopeParams prm, int n_tensors,
                                                             const int32_t* __restrict__ idx, int64_t n, int64_t T,
                                                             int side, int prefix, int64_t row_bytes,
                                                             int vec_per_head) {
  constexpr int kPairs = kBf16 ? 4 : 2;  // pairs per 16-byte vector
  constexpr bool kInverse = kMode != kGather;
  const int lane = threadIdx.x & 31;
  const int64_t nvec = row_bytes >> 4;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int64_t rows = kMode == kScatterZero ? T : n;
  const int64_t s2 = (int64_t)side * side;
  const int p0 = (lane % vec_per_head) * kPairs;  // first pair of this lane's slot in every head
  for (int64_t q = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); q < rows; q += warps) {
    int64_t r, t;  // compact row, canvas row
    if (kMode == kScatterZero) {
      t = q;
      int64_t lo = 0, hi = n;  // first r with idx[r] >= t
      while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (idx[mid] < t) lo = mid + 1;
        else hi = mid;
      }
      r = (lo < n && idx[lo] == t) ? lo : -1;
    } else {
      r = q;
      t = idx[q];
      if (t < 0 || t >= T) continue;  // not a canvas row: nothing to read or write
    }
    float cs[kPairs], sn[kPairs];
    for (int ti = 0; ti < n_tensors; ++ti) {
      const uint8_t* s = prm.src[ti] + (kMode == kGather ? t : r) * row_bytes;
      uint8_t* d = prm.dst[ti] + (kMode == kGather ? r : t) * row_bytes;
      for (int64_t v0 = 0; v0 < nvec; v0 += 32 * kVec) {
        // all of this lane's loads of the row in flight before any use
        uint4 w[kVec];
#pragma unroll
        for (int j = 0; j < kVec; ++j) {
          const int64_t v = v0 + j * 32 + lane;
          w[j] = (r >= 0 && v < nvec) ? ld_nc_v4(s + (v << 4)) : make_uint4(0, 0, 0, 0);
        }
        if (ti == 0 && v0 == 0 && r >= 0) {  // this lane's pairs, once per row, while the loads fly
          const int64_t ti = t - prefix;  // text tokens (t < prefix) sit at (0, 0, 0)
          const float pi = ti < 0 ? 0.f : (float)(ti / s2), py = ti < 0 ? 0.f : (float)((ti % s2) / side);
          const float px = ti < 0 ? 0.f : (float)(ti % side);
#pragma unroll
          for (int e = 0; e < kPairs; ++e) {
            const int p = p0 + e;
            const int a = prm.axis[p];
            sincosf((a == 0 ? pi : (a == 1 ? py : px)) * prm.freq[p], &sn[e], &cs[e]);
            if (kInverse) sn[e] = -sn[e];
          }
        }
#pragma unroll
        for (int j = 0; j < kVec; ++j) {
          const int64_t v = v0 + j * 32 + lane;
          if (v >= nvec) continue;
          if (r >= 0) {
            if constexpr (kBf16) {
              uint32_t* u = &w[j].x;
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float x0 = __uint_as_float(u[e] << 16), x1 = __uint_as_float(u[e] & 0xFFFF0000u);
                u[e] = pack_bf16x2(fmaf(x0, cs[e], -x1 * sn[e]), fmaf(x0, sn[e], x1 * cs[e]));
              }
            } else {
              const float a0 = __uint_as_float(w[j].x), a1 = __uint_as_float(w[j].y);
              const float b0 = __uint_as_float(w[j].z), b1 = __uint_as_float(w[j].w);
              w[j].x = __float_as_uint(fmaf(a0, cs[0], -a1 * sn[0]));
              w[j].y = __float_as_uint(fmaf(a0, sn[0], a1 * cs[0]));
              w[j].z = __float_as_uint(fmaf(b0, cs[1], -b1 * sn[1]));
              w[j].w = __float_as_uint(fmaf(b0, sn[1], b1 * cs[1]));
            }
          }
          st_v4(d + (v << 4), w[j]);
        }
      }
    }
  }
}

cudaError_t launch_fg_rope(const int32_t* idx, int64_t n, int n_tensors, const void* const* src, void* const* dst,
                           int heads, int head_dim, bool bf16, int side, int prefix, const int32_t axes[3],
                           float theta, int mode, int64_t T, int sms, cudaStream_t stream) {
  RopeParams prm{};
  for (int i = 0; i < n_tensors; ++i) {
    prm.src[i] = static_cast<const uint8_t*>(src[i]);
    prm.dst[i] = static_cast<uint8_t*>(dst[i]);
  }
  int p = 0;
  for (int a = 0; a < 3; ++a)
    for (int k = 0; k < axes[a] / 2; ++k, ++p) {
      prm.freq[p] = (float)pow((double)theta, -2.0 * k / (double)axes[a]);
      prm.axis[p] = (uint8_t)a;
    }
  const int64_t elem = bf16 ? 2 : 4;
  const int64_t row_bytes = (int64_t)heads * head_dim * elem;
  const int vec_per_head = (int)(head_dim * elem / 16);
  const int64_t rows = mode == kScatterZero ? T : n;
  if (rows == 0) return cudaSuccess;
  int64_t want = (rows + 7) / 8, cap = (int64_t)sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  const bool big = row_bytes >= 16 * 32 * 12;
#define UT_ROPE_LAUNCH(B, M)                                                                                       \
  (big ? rope_kernel<B, M, 12><<<grid, kRopeThreads, 0, stream>>>(prm, n_tensors, idx, n, T, side, prefix,       \
                                                                  row_bytes, vec_per_head)                                  \
       : rope_kernel<B, M, 4><<<grid, kRopeThreads, 0, stream>>>(prm, n_tensors, idx, n, T, side, prefix,        \
                                                                 row_bytes, vec_per_head))
  if (bf16) {
    if (mode == kGather) UT_ROPE_LAUNCH(true, kGather);
    else if (mode == kScatterKeep) UT_ROPE_LAUNCH(true, kScatterKeep);
    else UT_ROPE_LAUNCH(true, kScatterZero);
  } else {
    if (mode == kGather) UT_ROPE_LAUNCH(false, kGather);
    else if (mode == kScatterKeep) UT_ROPE_LAUNCH(false, kScatterKeep);
    else UT_ROPE_LAUNCH(false, kScatterZero);
  }
#undef UT_ROPE_LAUNCH
  return cudaGetLastError();
}

}  // namespace ut
