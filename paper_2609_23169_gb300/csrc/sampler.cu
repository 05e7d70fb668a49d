// Sampler steps on the canvas latent around the foreground-only model call.
//
//   fg_euler_kernel      sparse Euler update (Sec. 3.2, Eq. euler):
//                        z[idx[n]] += dt * v[n], dt = t_prev - t_curr; the
//                        background rows are not touched.  One fused
//                        multiply-add in fp32 per element, rounded once to the
//                        storage type (bf16 or fp32).  Optionally the updated
//                        row is also written to zc[n]: the compacted latent
//                        the next denoising step feeds the model (the gather
//                        of Background Token Dropping fused with the update,
//                        so that step reads z's foreground rows once).
//   fg_composite_kernel  composite latent for decoding (Sec. 3.4,
//                        Eq. mixed_latent): background row t of z takes row
//                        t mod P of the canonical background tile; foreground
//                        rows keep the denoised latent (a plain bit copy).
//
// Both are HBM-bound streams over 16-byte vectors: thread g handles vector
// g % V of row g / V (V = row bytes / 16), grid-stride over a grid of a few
// CTAs per SM.  Euler moves 3 row-bytes per retained token (read v, read and
// write z) plus its 4-byte index; the composite writes the background rows
// and reads the T-byte mask (the tile stays in L2).
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kSamplerThreads = 256;

static int stream_grid(int64_t vectors, int sms) {
  const int64_t need = (vectors + kSamplerThreads - 1) / kSamplerThreads;
  const int64_t cap = (int64_t)sms * 8;
  return (int)(need < cap ? (need > 0 ? need : 1) : cap);
}

UT_DEV float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
UT_DEV float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

UT_DEV uint32_t euler_bf16x2(uint32_t z, uint32_t v, float dt) {
  return pack_bf16x2(fmaf(dt, bf16_lo(v), bf16_lo(z)), fmaf(dt, bf16_hi(v), bf16_hi(z)));
}

template <bool kBf16, typename I>
__global__ void __launch_bounds__(kSamplerThreads) fg_euler_kernel(const int32_t* __restrict__ idx, int64_t n,
                                                                   uint8_t* __restrict__ z,
                                                                   const uint8_t* __restrict__ v, int64_t T,
                                                                   int64_t row_bytes, float dt, int32_t* status,
                                                                   uint8_t* __restrict__ zc) {
  // I: the index type of the vector count (32-bit division when it fits)
  const I V = (I)(row_bytes >> 4);
  const I total = (I)n * V;
  for (I g = (I)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += (I)gridDim.x * blockDim.x) {
    const I r = g / V, c = g - r * V;
    const int64_t t = idx[r];
    if (t < 0 || t >= T) {  // an index outside the canvas: skip the row, report it
      if (c == 0) set_status(status, UT_ERR_INVALID_ARG);
      continue;
    }
    const uint4 vv = ld_nc_v4(v + r * row_bytes + (c << 4));
    uint8_t* zp = z + t * row_bytes + (c << 4);
    uint4 zz = *reinterpret_cast<const uint4*>(zp);
    if (kBf16) {
      zz.x = euler_bf16x2(zz.x, vv.x, dt);
      zz.y = euler_bf16x2(zz.y, vv.y, dt);
      zz.z = euler_bf16x2(zz.z, vv.z, dt);
      zz.w = euler_bf16x2(zz.w, vv.w, dt);
    } else {
      zz.x = __float_as_uint(fmaf(dt, __uint_as_float(vv.x), __uint_as_float(zz.x)));
      zz.y = __float_as_uint(fmaf(dt, __uint_as_float(vv.y), __uint_as_float(zz.y)));
      zz.z = __float_as_uint(fmaf(dt, __uint_as_float(vv.z), __uint_as_float(zz.z)));
      zz.w = __float_as_uint(fmaf(dt, __uint_as_float(vv.w), __uint_as_float(zz.w)));
    }
    st_v4(zp, zz);
    if (zc) st_v4(zc + (int64_t)r * row_bytes + ((int64_t)c << 4), zz);
  }
}

__global__ void __launch_bounds__(kSamplerThreads) fg_composite_kernel(const uint8_t* __restrict__ mask, int64_t T,
                                                                       uint8_t* __restrict__ z,
                                                                       const uint8_t* __restrict__ tile,
                                                                       int64_t period, int64_t row_bytes) {
  const int64_t V = row_bytes >> 4;
  const int64_t total = T * V;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
    const int64_t t = g / V, c = g - t * V;
    if (mask[t]) continue;
    const uint4 b = *reinterpret_cast<const uint4*>(tile + (t % period) * row_bytes + (c << 4));
    st_v4(z + t * row_bytes + (c << 4), b);
  }
}

cudaError_t launch_fg_euler(const int32_t* idx, int64_t n, void* z, const void* v, int64_t T, int64_t row_bytes,
                            bool bf16, float dt, int32_t* status, void* zc, int sms, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  const int64_t vectors = n * (row_bytes >> 4);
  const int grid = stream_grid(vectors, sms);
  uint8_t* zb = static_cast<uint8_t*>(z);
  const uint8_t* vb = static_cast<const uint8_t*>(v);
  uint8_t* zcb = static_cast<uint8_t*>(zc);
  // the grid-stride index stays below vectors + grid * threads
  const bool small = vectors + (int64_t)grid * kSamplerThreads < ((int64_t)1 << 31);
  if (bf16) {
    if (small)
      fg_euler_kernel<true, int32_t><<<grid, kSamplerThreads, 0, stream>>>(idx, n, zb, vb, T, row_bytes, dt, status, zcb);
    else
      fg_euler_kernel<true, int64_t><<<grid, kSamplerThreads, 0, stream>>>(idx, n, zb, vb, T, row_bytes, dt, status, zcb);
  } else {
    if (small)
      fg_euler_kernel<false, int32_t><<<grid, kSamplerThreads, 0, stream>>>(idx, n, zb, vb, T, row_bytes, dt, status, zcb);
    else
      fg_euler_kernel<false, int64_t><<<grid, kSamplerThreads, 0, stream>>>(idx, n, zb, vb, T, row_bytes, dt, status, zcb);
  }
  return cudaGetLastError();
}

cudaError_t launch_fg_composite(const uint8_t* mask, int64_t T, void* z, const void* tile, int64_t period,
                                int64_t row_bytes, int sms, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const int grid = stream_grid(T * (row_bytes >> 4), sms);
  fg_composite_kernel<<<grid, kSamplerThreads, 0, stream>>>(mask, T, static_cast<uint8_t*>(z),
                                                            static_cast<const uint8_t*>(tile), period, row_bytes);
  return cudaGetLastError();
}

}  // namespace ut
