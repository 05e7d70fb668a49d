// Canvas mask from alpha channels (Sec. 3.2, mask construction): a token is
// foreground when some alpha pixel of its factor x factor block exceeds the
// threshold (the 1/16 downsampling), then the token mask is dilated by a
// square of radius r; the view masks serve the targets and the conditions,
// the reference image has its own.
//
//   alpha_mask_kernel  one CTA per 16 x 16 token tile of one image (a thread
//                      per token of the tile and its halo): pool the
//                      tile plus an r-token halo into shared memory (16-byte
//                      loads of the alpha rows, per-byte compares), then
//                      dilate from shared memory and write the token to its
//                      target and condition slots (views) or the reference
//                      slot of the canvas.
//
// HBM-bound: the alpha images are read once (the halo re-reads hit L2) and the
// canvas mask (one byte per token) is written once.
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kMaskTile = 16;     // tokens per tile side
constexpr int kMaskMaxRadius = 16;

__global__ void __launch_bounds__(1024) alpha_mask_kernel(
    const uint8_t* __restrict__ alpha, int n_views, int height, int width, int factor, int radius, int threshold,
    bool vec16, uint8_t* __restrict__ canvas) {
  __shared__ uint8_t pooled[(kMaskTile + 2 * kMaskMaxRadius) * (kMaskTile + 2 * kMaskMaxRadius)];
  const int img = blockIdx.z;
  const int th = height / factor, tw = width / factor;  // tokens per image side
  const int y0 = blockIdx.y * kMaskTile - radius, x0 = blockIdx.x * kMaskTile - radius;
  const int hs = kMaskTile + 2 * radius;                 // halo tile side
  const uint8_t* a = alpha + (int64_t)img * height * width;
  const uint32_t thr4 = 0x01010101u * (uint32_t)threshold;
  for (int s = threadIdx.x; s < hs * hs; s += blockDim.x) {
    const int ty = y0 + s / hs, tx = x0 + s % hs;
    uint8_t fg = 0;
    if (ty >= 0 && ty < th && tx >= 0 && tx < tw) {
      const uint8_t* blk = a + (int64_t)ty * factor * width + (int64_t)tx * factor;
      if (vec16) {
        // 16 pixel rows per batch, all loads issued before the compares (no
        // early exit inside a batch: it would serialise the loads)
        uint32_t any = 0;
        for (int py0 = 0; py0 < factor && !any; py0 += 16)
          for (int px = 0; px < factor; px += 16) {
            uint4 w[16];
#pragma unroll
            for (int r = 0; r < 16; ++r) w[r] = ld_nc_v4(blk + (int64_t)(py0 + r) * width + px);
#pragma unroll
            for (int r = 0; r < 16; ++r)
              any |= __vcmpgtu4(w[r].x, thr4) | __vcmpgtu4(w[r].y, thr4) | __vcmpgtu4(w[r].z, thr4) |
                     __vcmpgtu4(w[r].w, thr4);
          }
        fg = any != 0;
      } else {
        for (int py = 0; py < factor && !fg; ++py)
          for (int px = 0; px < factor; ++px)
            if (blk[(int64_t)py * width + px] > threshold) {
              fg = 1;
              break;
            }
      }
    }
    pooled[s] = fg;
  }
  __syncthreads();
  if (threadIdx.x >= kMaskTile * kMaskTile) return;
  const int ly = threadIdx.x / kMaskTile, lx = threadIdx.x % kMaskTile;
  const int ty = blockIdx.y * kMaskTile + ly, tx = blockIdx.x * kMaskTile + lx;
  if (ty >= th || tx >= tw) return;
  uint8_t m = 0;
  for (int dy = 0; dy <= 2 * radius && !m; ++dy)
    for (int dx = 0; dx <= 2 * radius; ++dx) m |= pooled[(ly + dy) * hs + lx + dx];
  const int64_t per_img = (int64_t)th * tw, pos = (int64_t)ty * tw + tx;
  if (img < n_views) {
    canvas[img * per_img + pos] = m;                 // noisy target view
    canvas[(n_views + img) * per_img + pos] = m;     // its condition image shares the mask
  } else {
    canvas[2 * (int64_t)n_views * per_img + pos] = m;  // reference image
  }
}

cudaError_t launch_mask_from_alpha(const uint8_t* alpha, int n_views, int height, int width, int factor,
                                   int radius, int threshold, uint8_t* canvas, cudaStream_t stream) {
  const int th = height / factor, tw = width / factor;
  if (th == 0 || tw == 0) return cudaSuccess;
  const bool vec16 = factor % 16 == 0 && width % 16 == 0 && (reinterpret_cast<uintptr_t>(alpha) & 15) == 0;
  dim3 grid((tw + kMaskTile - 1) / kMaskTile, (th + kMaskTile - 1) / kMaskTile, n_views + 1);
  // one thread per token of the tile plus its halo (a single round of loads)
  // up to 1024 threads; at least one per token of the tile for the dilation
  const int hs = kMaskTile + 2 * radius;
  int threads = ((hs * hs + 31) / 32) * 32;
  if (threads > 1024) threads = 1024;
  alpha_mask_kernel<<<grid, threads, 0, stream>>>(alpha, n_views, height, width, factor, radius,
                                                                 threshold, vec16, canvas);
  return cudaGetLastError();
}

}  // namespace ut
