// Block-sparse attention backward on the tcgen05 tensor cores.
//
// With P = exp(S - LSE) recomputed from the forward's row normalisers and
// D_r = dO_r . O_r:
//   dV = P^T dO,   dS = P o (dO V^T - D),   dQ = scale * dS K,   dK = scale * dS^T Q
// over the retained block pairs only:
//
//   bwd_pre_kernel          D_r and LSE_r * log2(e) per (head, row) into a
//                           padded [H, N_t*128] workspace (padding rows: D = 0,
//                           LSE = +inf so that they contribute P = 0).
//   bwd_fused_kernel        item (h, 128-row key tile j) over the transposed
//                           lists: S^T and dP^T once per pair, dK and dV
//                           accumulated in TMEM, dQ^T partials added into an
//                           fp32 accumulator (below).
//   bwd_dq_finalize_kernel  dQ = scale * accumulator, bf16.
//
// Blocks of 64 rows (b_q or b_kv) are served by the same 128 x 128 tiles:
//   b_q = 64:   two listed 64-row query blocks fill one 128-row query tile
//               (Q and dO loaded as two 64-row TMA boxes, PairList):
//               consecutive entries of the key block's list for b_kv = 128
//               (nothing discarded), the two 64-row key blocks' lists in
//               lockstep for b_kv = 64 (key rows 0-63 see the low half of the
//               query tile, key rows 64-127 the high half); the dQ^T drain
//               adds each half into its own query block;
//   b_q = 128, b_kv = 64:  the item's two lists are merged into 128-row query
//               tiles with a mask of the listed 64 x 64 sub-blocks (TileList).
// P of the sub-blocks a key row does not see is zero.
// All waits are bounded (UT_ERR_TIMEOUT on expiry, then drain and return).
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kTile = 128;
constexpr uint32_t kChunk = 128 * 128;  // one 128-row x 128-byte swizzled sub-tile

// ------------------------------------------------------------- preprocess
// One warp per (padded) row r; a half-warp per head (8 bf16 per lane).
__global__ void __launch_bounds__(256) bwd_pre_kernel(const __nv_bfloat16* __restrict__ o,
                                                      const __nv_bfloat16* __restrict__ dout,
                                                      const float* __restrict__ lse, int64_t N, int64_t Np, int H,
                                                      int d, int64_t rs, float* __restrict__ lse2,
                                                      float* __restrict__ dsum) {
  const int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (r >= Np) return;
  const int lane = threadIdx.x & 31;
  const int lanes_per_head = d / 8;           // 16 (d=128) or 8 (d=64)
  const int heads_per_iter = 32 / lanes_per_head;
  for (int h0 = 0; h0 < H; h0 += heads_per_iter) {
    const int h = h0 + lane / lanes_per_head;
    float s = 0.f;
    if (r < N && h < H) {
      const int64_t off = r * rs + (int64_t)h * d + (lane % lanes_per_head) * 8;
      uint4 a = *reinterpret_cast<const uint4*>(o + off);
      uint4 b = *reinterpret_cast<const uint4*>(dout + off);
      const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
      const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float2 x = __bfloat1622float2(pa[e]);
        float2 y = __bfloat1622float2(pb[e]);
        s = fmaf(x.x, y.x, s);
        s = fmaf(x.y, y.y, s);
      }
    }
    for (int off = lanes_per_head / 2; off; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if ((lane % lanes_per_head) == 0 && h < H) {
      dsum[(int64_t)h * Np + r] = r < N ? s : 0.f;
      lse2[(int64_t)h * Np + r] = r < N ? lse[(int64_t)h * N + r] * 1.4426950408889634f : INFINITY;
    }
  }
}

struct BwdParams {
  const int32_t* ptr;   // transposed fine lists: per (head, key block) the query blocks
  const int32_t* idx;
  const float* lse2;    // [H, Np]  LSE * log2(e)
  const float* dsum;    // [H, Np]  D
  __nv_bfloat16* out0;  // dv
  __nv_bfloat16* out1;  // dk
  int32_t* status;
  int64_t N, Np, rs;
  int H, nq, n_items;   // nq: 128-row tiles per head (items = H * nq key tiles)
  int nk_fine;          // key blocks per head in the transposed lists
  int k_rows_per_tile;  // 1 (b_kv = 128) or 2 (b_kv = 64)
  int list_shift;       // 0 (b_q = 128) or 1 (b_q = 64)
  float scale, scale_log2;
  uint64_t timeout_ns;
  int32_t* item_counter;  // next item to hand out (zeroed before the launch)
};

// 64 consecutive TMEM columns of this warp's 32 lanes, one wait.
UT_DEV void tmem_ld64(uint32_t taddr, uint32_t* r) {
  tmem_ld32(taddr, *reinterpret_cast<uint32_t(*)[32]>(r));
  tmem_ld32(taddr + 32, *reinterpret_cast<uint32_t(*)[32]>(r + 32));
  tmem_wait_ld();
}

// =========================================================================
//                       fused dK, dV and dQ (one kernel)
// =========================================================================
// Item = (head h, key block j); the pairs are the query blocks i of the
// transposed list.  Per pair, with the 128 key rows as TMEM lanes:
//   S^T  = K Q_i^T         -> TMEM R0            (A = K, B = Q_i; smem)
//   P^T  = exp2(S^T c - LSE_i log2 e)   -> bf16, shared tile PT
//   dP^T = V dO_i^T        -> TMEM R0 (after S^T was read)
//   dV  += P^T dO_i        (A = PT, B = dO_i)
//   dS^T = P^T o (dP^T - D_i)           -> bf16, shared tile DST
//   dK  += dS^T Q_i        (A = DST, B = Q_i)
//   dQ_i^T = K^T dS^T      -> TMEM RQ            (A = K read d-major, B = DST)
// and four drain warps add dQ_i^T into an fp32 [H, N_q*128, d] accumulator
// with coalesced reductions (lane = d, one 128-byte row segment per query
// row), off the elementwise warps' path; S and dP are computed once per pair.
// A final kernel scales the accumulator by the softmax scale and writes dQ in
// bf16.  Roles (512 threads, four warpgroups; the register file is rebalanced
// with setmaxnreg): warpgroup 0 = warp 0 TMA, warp 1 TMEM owner + MMA issuer
// (warps 2-3 idle); warpgroups 1-2 = 8 elementwise warps; warpgroup 3 = 4 dQ
// drain warps.
// TMEM columns: R0 [0,128), RQ [128,256), dV [256,256+d), dK [384,384+d).
// For d = 64 the A operand K^T of the dQ product is padded to 128 rows with a
// zero sub-tile placed right after K, and the padding rows of RQ are ignored.
constexpr int kFuThreads = 512;
// registers per thread after setmaxnreg, per warpgroup; the sum equals the
// launch allocation (4 x 128) so that every increase is covered by decreases
constexpr int kFuRegLaunch = 128, kFuRegCtl = 96, kFuRegEw = 168, kFuRegDrain = 80;
static_assert(kFuRegCtl + 2 * kFuRegEw + kFuRegDrain == 4 * kFuRegLaunch, "setmaxnreg split must match the launch");
// Ring depths: Q is held from S^T to dK (late in the pair), dO only from dP^T
// to dV (early), so dO gets one stage and its 32 KB buy separate P^T and
// dS^T tiles: P^T of the next pair never waits for this pair's dK and dQ.
constexpr int kFuQStages = 2, kFuDoStages = 1;
constexpr uint32_t kColR0 = 0, kColRQ = 128, kColFuDv = 256, kColFuDk = 384;

// Items are handed out dynamically (the transposed lists differ in length:
// 36-153 query blocks per key block at the 2048 canvas, so a static
// round-robin leaves the busiest CTA ~5% above the mean), still in head-major
// order, so that the CTAs in flight share one head's Q, dO and dQ accumulator
// in L2.  kItemConsumers: TMA lane 1, the MMA warp, 8 elementwise warps, 4
// drain warps.
constexpr int kItemSlots = 4, kItemConsumers = 14;

template <int D>
struct FusedSmem {
  static constexpr int kC = D / 64;
  static constexpr uint32_t kTileBytes = kTile * D * 2;
  alignas(1024) uint8_t k[2 * kChunk];        // K (d/64 sub-tiles), then zeros up to 128 d-rows
  alignas(1024) uint8_t v[kTileBytes];
  alignas(1024) uint8_t pt[kTile * kTile * 2];   // P^T of the current pair
  alignas(1024) uint8_t dst[kTile * kTile * 2];  // dS^T of the current pair
  alignas(1024) uint8_t q[kFuQStages][kTileBytes];
  alignas(1024) uint8_t dout[kFuDoStages][kTileBytes];
  alignas(16) float lse2[2][kTile];
  alignas(16) float dsum[2][kTile];
  uint64_t kv_full, kv_empty;
  uint64_t q_full[kFuQStages], q_empty[kFuQStages], do_full[kFuDoStages], do_empty[kFuDoStages];
  uint64_t s_full, s_empty, dp_full, dp_empty, pt_full, pt_done, dst_full, ds_done, dq_empty;
  uint64_t acc_full, acc_empty, mma_done;
  uint64_t rowvec_full[2];
  // the CTA's item sequence: TMA lane 0 takes the next item from the global
  // counter and publishes it here; every other role reads the slots in order
  int32_t item[kItemSlots];
  uint64_t item_full[kItemSlots], item_empty[kItemSlots];
  uint32_t tmem_base;
  int abort_flag;
};

UT_DEV void red_add_f32(float* p, float v) {
  asm volatile("red.relaxed.gpu.global.add.f32 [%0], %1;" ::"l"(p), "f"(v) : "memory");
}

template <int D, int kMode>
__global__ void __launch_bounds__(kFuThreads, 1)
    bwd_fused_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
                     const __grid_constant__ CUtensorMap tm_q64, const __grid_constant__ CUtensorMap tm_do64,
                     const BwdParams prm, float* __restrict__ dq_acc) {
  constexpr bool kSub = kMode != 0;  // 64-row blocks on at least one side
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  FusedSmem<D>& sm = *reinterpret_cast<FusedSmem<D>*>(smem_raw);
  constexpr int C = FusedSmem<D>::kC;
  constexpr uint32_t TB = FusedSmem<D>::kTileBytes;
  const uint32_t warp = warp_id(), lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;
  if ((smem_u32(smem_raw) & 1023u) != 0) {
    if (threadIdx.x == 0) set_status(prm.status, UT_ERR_INVALID_ARG);
    return;
  }
  if (D == 64) {  // zero padding sub-tile of K^T (rows d = 64..127 of the dQ product)
    uint4* z = reinterpret_cast<uint4*>(sm.k + kChunk);
    for (uint32_t x = threadIdx.x; x < kChunk / 16; x += blockDim.x) z[x] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
  }
  if (threadIdx.x == 0) {
    mbar_init(&sm.kv_full, 1);
    mbar_init(&sm.kv_empty, 1);
    for (int s = 0; s < kFuQStages; ++s) {
      mbar_init(&sm.q_full[s], 1);
      mbar_init(&sm.q_empty[s], 1);
    }
    for (int s = 0; s < kFuDoStages; ++s) {
      mbar_init(&sm.do_full[s], 1);
      mbar_init(&sm.do_empty[s], 1);
    }
    mbar_init(&sm.s_full, 1);
    mbar_init(&sm.s_empty, 8);
    mbar_init(&sm.dp_full, 1);
    mbar_init(&sm.dp_empty, 8);
    mbar_init(&sm.pt_full, 8);
    mbar_init(&sm.pt_done, 1);
    mbar_init(&sm.dst_full, 8);
    mbar_init(&sm.ds_done, 1);
    mbar_init(&sm.dq_empty, 4);
    mbar_init(&sm.acc_full, 1);
    mbar_init(&sm.acc_empty, 8);
    mbar_init(&sm.mma_done, 1);
    mbar_init(&sm.rowvec_full[0], 256);
    mbar_init(&sm.rowvec_full[1], 256);
    for (int s = 0; s < kItemSlots; ++s) {
      mbar_init(&sm.item_full[s], 1);
      mbar_init(&sm.item_empty[s], kItemConsumers);
    }
    sm.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t wg = warp >> 2;
  // next item of this CTA's sequence (-1: none left); whole warp (converged)
  // or, with one = true, a single thread.  Returns false on timeout / abort.
  auto next_item = [&](uint32_t& kk, int& w, bool one) -> bool {
    const uint32_t s = kk % kItemSlots, n = kk / kItemSlots;
    const bool got = one ? mbar_wait(&sm.item_full[s], n & 1, abort_flag, prm.status, prm.timeout_ns)
                         : warp_wait(&sm.item_full[s], n & 1, abort_flag, prm.status, prm.timeout_ns);
    if (!got) return false;
    w = *reinterpret_cast<volatile int32_t*>(&sm.item[s]);
    if (one) {
      mbar_arrive(&sm.item_empty[s]);
    } else {
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.item_empty[s]);
    }
    ++kk;
    return true;
  };
  if (wg == 0) {
    setmaxnreg_dec<kFuRegCtl>();
    if (warp == 0) {
      // lane 0: K, V of the item and the Q ring (Q is freed after dK += dS^T Q);
      // lane 1: the dO ring (dO is freed after dV += P^T dO).
      if (lane < 2) {
        const bool is_q = lane == 0;
        if (is_q) {
          tma_prefetch_desc(&tm_q);
          tma_prefetch_desc(&tm_k);
          tma_prefetch_desc(&tm_v);
          if (kMode >= 2) tma_prefetch_desc(&tm_q64);
        } else {
          tma_prefetch_desc(&tm_do);
          if (kMode >= 2) tma_prefetch_desc(&tm_do64);
        }
        const uint64_t pol_qd = policy_evict_last(), pol_kv = policy_evict_first();
        uint64_t* full = is_q ? sm.q_full : sm.do_full;
        uint64_t* empty = is_q ? sm.q_empty : sm.do_empty;
        uint8_t* ring = is_q ? &sm.q[0][0] : &sm.dout[0][0];
        const void* tmap = is_q ? static_cast<const void*>(&tm_q) : static_cast<const void*>(&tm_do);
        const void* tmap64 = is_q ? static_cast<const void*>(&tm_q64) : static_cast<const void*>(&tm_do64);
        const uint32_t nst = is_q ? kFuQStages : kFuDoStages;
        uint32_t ki = 0, qd = 0, kk = 0;
        bool ok = true;
        for (;;) {
          int w;
          if (is_q) {  // take the next item and publish it to the other roles
            const uint32_t s = kk % kItemSlots, n = kk / kItemSlots;
            if (!(ok = mbar_wait(&sm.item_empty[s], (n & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
            w = atomicAdd(prm.item_counter, 1);
            if (w >= prm.n_items) w = -1;
            *reinterpret_cast<volatile int32_t*>(&sm.item[s]) = w;
            mbar_arrive(&sm.item_full[s]);
            ++kk;
          } else if (!(ok = next_item(kk, w, true))) {
            break;
          }
          if (w < 0) break;
          const int h = w / prm.nq, j = w % prm.nq;
          BlockSteps<kMode> tl;
          tl.init(prm.ptr, prm.idx, h, j, prm.nk_fine, prm.k_rows_per_tile, prm.list_shift);
          if (tl.empty()) continue;
          if (is_q) {
            if (!(ok = mbar_wait(&sm.kv_empty, (ki & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
            mbar_expect_tx(&sm.kv_full, 2 * TB);
            for (int c = 0; c < C; ++c) {
              tma_load_2d(sm.k + c * kChunk, &tm_k, &sm.kv_full, h * D + c * 64, j * kTile, pol_kv);
              tma_load_2d(sm.v + c * kChunk, &tm_v, &sm.kv_full, h * D + c * 64, j * kTile, pol_kv);
            }
            ++ki;
          }
          int i, ih;
          uint32_t bits;
          for (; tl.next(i, ih, bits); ++qd) {
            const uint32_t st = qd % nst, n = qd / nst;
            if (!(ok = mbar_wait(&empty[st], (n & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
            mbar_expect_tx(&full[st], TB);
            uint8_t* dst = ring + st * TB;
            if (tl.pair) {  // two 64-row boxes: rows 0-63 and 64-127 of each 128-row sub-tile
              const int b0 = PairList::load_lo(i, ih), b1 = PairList::load_hi(i, ih);
              for (int c = 0; c < C; ++c) {
                tma_load_2d(dst + c * kChunk, tmap64, &full[st], h * D + c * 64, b0 * 64, pol_qd);
                tma_load_2d(dst + c * kChunk + 64 * 128, tmap64, &full[st], h * D + c * 64, b1 * 64, pol_qd);
              }
            } else {
              for (int c = 0; c < C; ++c)
                tma_load_2d(dst + c * kChunk, tmap, &full[st], h * D + c * 64, i * kTile, pol_qd);
            }
          }
          if (!ok) break;
        }
        auto drain = [&](uint64_t* bar, uint32_t parity) {
          if (!mbar_drain(bar, parity, kDrainTimeoutNs)) set_status(prm.status, UT_ERR_TIMEOUT);
        };
        if (ki > 0) drain(&sm.kv_full, (ki - 1) & 1);
        for (uint32_t u = (qd >= nst ? qd - nst : 0); u < qd; ++u) drain(&full[u % nst], (u / nst) & 1);
      }
    } else if (warp == 1) {
      // whole warp, converged: waits are warp-uniform, MMAs/commits elect one lane.
      // Per pair t: dP^T_t, dV_t, S^T_{t+1}, dK_t, dQ_t^T.
      {
        constexpr uint32_t idesc_s = idesc_bf16_f32(kTile, kTile, false, false);
        constexpr uint32_t idesc_acc = idesc_bf16_f32(kTile, D, false, true);
        constexpr uint32_t idesc_dq = idesc_bf16_f32(kTile, kTile, true, true);
        const uint32_t k_addr = smem_u32(sm.k), v_addr = smem_u32(sm.v);
      const uint32_t pt_addr = smem_u32(sm.pt), dst_addr = smem_u32(sm.dst);
        uint32_t ki = 0, qd0 = 0, kk = 0;
        bool ok = true;
        for (;;) {
          int w;
          if (!(ok = next_item(kk, w, false)) || w < 0) break;
          BlockSteps<kMode> tl;
          tl.init(prm.ptr, prm.idx, w / prm.nq, w % prm.nq, prm.nk_fine, prm.k_rows_per_tile, prm.list_shift);
          const int L = tl.count_warp();
          if (L <= 0) continue;
          if (!(ok = warp_wait(&sm.kv_full, ki & 1, abort_flag, prm.status, prm.timeout_ns))) break;
          auto issue_st = [&](int t) -> bool {  // S^T_t = K Q_t^T into R0
            const uint32_t qd = qd0 + t, st = qd % kFuQStages, n = qd / kFuQStages;
            if (!warp_wait(&sm.q_full[st], n & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
            if (!warp_wait(&sm.dp_empty, (qd & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)) return false;
            tc_fence_after();
            const uint32_t q_addr = smem_u32(sm.q[st]);
  #pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t off = (kk >> 2) * kChunk + (kk & 3) * 32;
              mma_bf16_ss_w(tmem + kColR0, sdesc_sw128(k_addr + off, 16, 1024), sdesc_sw128(q_addr + off, 16, 1024),
                            idesc_s, kk > 0);
            }
            mma_commit_w(&sm.s_full);
            return true;
          };
          if (!(ok = issue_st(0))) break;
          for (int t = 0; t < L && ok; ++t) {
            const uint32_t qd = qd0 + t, sq = qd % kFuQStages, sd = qd % kFuDoStages, nd = qd / kFuDoStages;
            const uint32_t do_addr = smem_u32(sm.dout[sd]), q_addr = smem_u32(sm.q[sq]);
            // dP^T_t = V dO_t^T into R0 once S^T_t has been read
            if (!(ok = warp_wait(&sm.do_full[sd], nd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
            if (!(ok = warp_wait(&sm.s_empty, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
            tc_fence_after();
  #pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t off = (kk >> 2) * kChunk + (kk & 3) * 32;
              mma_bf16_ss_w(tmem + kColR0, sdesc_sw128(v_addr + off, 16, 1024), sdesc_sw128(do_addr + off, 16, 1024),
                            idesc_s, kk > 0);
            }
            mma_commit_w(&sm.dp_full);
            // dV += P^T_t dO_t
            if (!(ok = warp_wait(&sm.pt_full, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
            if (t == 0 && !(ok = warp_wait(&sm.acc_empty, (ki & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)))
              break;
            tc_fence_after();
  #pragma unroll
            for (int kk = 0; kk < kTile / 16; ++kk) {
              const uint32_t aoff = (kk >> 2) * kChunk + (kk & 3) * 32;
              mma_bf16_ss_w(tmem + kColFuDv, sdesc_sw128(pt_addr + aoff, 16, 1024),
                            sdesc_sw128(do_addr + kk * 2048, kChunk, 1024), idesc_acc, (t > 0 || kk > 0));
            }
            mma_commit_w(&sm.pt_done);
            mma_commit_w(&sm.do_empty[sd]);
            // S^T_{t+1} once dP^T_t has been read
            if (t + 1 < L && !(ok = issue_st(t + 1))) break;
            // dK += dS^T_t Q_t
            if (!(ok = warp_wait(&sm.dst_full, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
            tc_fence_after();
  #pragma unroll
            for (int kk = 0; kk < kTile / 16; ++kk) {
              const uint32_t aoff = (kk >> 2) * kChunk + (kk & 3) * 32;
              mma_bf16_ss_w(tmem + kColFuDk, sdesc_sw128(dst_addr + aoff, 16, 1024),
                            sdesc_sw128(q_addr + kk * 2048, kChunk, 1024), idesc_acc, (t > 0 || kk > 0));
            }
            mma_commit_w(&sm.q_empty[sq]);
            // dQ_t^T = K^T dS^T_t into RQ once the previous pair's dQ^T was drained
            if (!(ok = warp_wait(&sm.dq_empty, (qd & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
            tc_fence_after();
  #pragma unroll
            for (int kk = 0; kk < kTile / 16; ++kk)
              mma_bf16_ss_w(tmem + kColRQ, sdesc_sw128(k_addr + kk * 2048, kChunk, 1024),
                            sdesc_sw128(dst_addr + kk * 2048, kChunk, 1024), idesc_dq, kk > 0);
            mma_commit_w(&sm.ds_done);
            if (t == L - 1) mma_commit_w(&sm.kv_empty);
          }
          if (!ok) break;
          mma_commit_w(&sm.acc_full);
          qd0 += L;
          ++ki;
        }
        mma_commit_w(&sm.mma_done);
        if (!mbar_drain(&sm.mma_done, 0, kDrainTimeoutNs)) set_status(prm.status, UT_ERR_TIMEOUT);
      }
  }
  } else if (wg == 1 || wg == 2) {
    setmaxnreg_inc<kFuRegEw>();
    // 8 elementwise warps: warps w and w+4 share TMEM lane quarter (w & 3),
    // i.e. the same 32 key rows, and split the 128 query columns (and the D
    // output columns) into halves.  A half is exactly one 128-byte swizzle
    // sub-tile of the shared P^T / dS^T tile.
    const uint32_t quarter = warp & 3;
    const uint32_t half = (warp - 4) >> 2;
    const uint32_t krow = quarter * 32 + lane;  // key row of the tile = TMEM lane (d index for dQ^T)
    const uint32_t tid = threadIdx.x - 128;     // 0..255 within the elementwise group
    const uint32_t lane_base = (quarter * 32) << 16;
    constexpr int HC = kTile / 2;               // query columns per half
    constexpr int HD = D / 2;                   // output columns per half
    const float c = prm.scale_log2;
    const uint32_t pt_row = smem_u32(sm.pt) + half * kChunk + krow * 128;
    const uint32_t dst_row = smem_u32(sm.dst) + half * kChunk + krow * 128;
    uint32_t qd0 = 0, ki = 0, kk = 0;
    bool ok = true;
    const uint32_t kh = krow >> 6;  // which 64-row half of the key tile
    for (;;) {
      int w;
      if (!(ok = next_item(kk, w, false)) || w < 0) break;
      const int h = w / prm.nq, j = w % prm.nq;
      BlockSteps<kMode> tl;
      tl.init(prm.ptr, prm.idx, h, j, prm.nk_fine, prm.k_rows_per_tile, prm.list_shift);
      const int L = tl.count_warp();
      const int64_t gk = (int64_t)j * kTile + krow;
      const bool row_ok = gk < prm.N;
      __nv_bfloat16* dv_row = prm.out0 + gk * prm.rs + (int64_t)h * D + half * HD;
      __nv_bfloat16* dk_row = prm.out1 + gk * prm.rs + (int64_t)h * D + half * HD;
      if (L <= 0) {
        if (row_ok)
          for (int e = 0; e < HD; e += 8) {
            *reinterpret_cast<uint4*>(dv_row + e) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(dk_row + e) = make_uint4(0, 0, 0, 0);
          }
        continue;
      }
      // this thread's element of the query-row vectors (LSE*log2e for threads
      // 0-127, D for 128-255) is loaded one pair ahead: query column
      // tid mod 128 of the tile, in its 64-row half
      const uint32_t qcol = tid & (kTile - 1), qhalf = qcol >> 6;
      const float* rv_src = (tid < kTile ? prm.lse2 : prm.dsum) + (int64_t)h * prm.Np + (qcol & 63);
      auto rv_row = [&](int lo, int hi) -> int64_t {  // first row of this thread's 64-row query half
        if (tl.pair) return 64 * (int64_t)(qhalf ? PairList::load_hi(lo, hi) : PairList::load_lo(lo, hi));
        return (int64_t)lo * kTile + 64 * qhalf;
      };
      int i_next, ih_next;
      uint32_t bits_next;
      tl.next(i_next, ih_next, bits_next);
      float rv = rv_src[rv_row(i_next, ih_next)];
      for (int t = 0; t < L; ++t) {
        const uint32_t qd = qd0 + t;
        // this half's 64 query columns and this thread's 64 key rows form one
        // 64 x 64 sub-block of the tile pair: listed or not
        const bool listed = !kSub || ((bits_next >> (2 * kh + half)) & 1u);
        // this pair's query-row LSE*log2e and D into the shared double buffer
        // (buffer qd&1 was last read in pair qd-2, which every thread finished
        //  before arriving for pair qd-1)
        if (tid < kTile) sm.lse2[qd & 1][tid] = rv;
        else sm.dsum[qd & 1][tid - kTile] = rv;
        mbar_arrive(&sm.rowvec_full[qd & 1]);
        if (t + 1 < L && tl.next(i_next, ih_next, bits_next)) rv = rv_src[rv_row(i_next, ih_next)];
        if (!(ok = warp_wait(&sm.rowvec_full[qd & 1], (qd >> 1) & 1, abort_flag, prm.status, prm.timeout_ns)))
          break;
        const float* ls = sm.lse2[qd & 1] + half * HC;
        const float* ds_v = sm.dsum[qd & 1] + half * HC;
        if (!(ok = warp_wait(&sm.s_full, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
        tc_fence_after();
        float p[HC];
        {
          uint32_t r[HC];
          tmem_ld64(tmem + lane_base + kColR0 + half * HC, r);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.s_empty);
          if (listed) {
#pragma unroll
            for (int x = 0; x < HC; x += 4) {
              const float4 l4 = *reinterpret_cast<const float4*>(ls + x);
              p[x + 0] = ex2_approx(fmaf(__uint_as_float(r[x + 0]), c, -l4.x));
              p[x + 1] = ex2_approx(fmaf(__uint_as_float(r[x + 1]), c, -l4.y));
              p[x + 2] = ex2_approx(fmaf(__uint_as_float(r[x + 2]), c, -l4.z));
              p[x + 3] = ex2_approx(fmaf(__uint_as_float(r[x + 3]), c, -l4.w));
            }
          } else {
#pragma unroll
            for (int x = 0; x < HC; ++x) p[x] = 0.f;
          }
        }
        // the P^T tile is free once the previous pair's dV MMA finished
        if (!(ok = warp_wait(&sm.pt_done, (qd & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
#pragma unroll
        for (int u = 0; u < HC / 8; ++u)
          st_shared_v4(pt_row + ((u ^ (krow & 7)) << 4), pack_bf16x2(p[8 * u], p[8 * u + 1]),
                       pack_bf16x2(p[8 * u + 2], p[8 * u + 3]), pack_bf16x2(p[8 * u + 4], p[8 * u + 5]),
                       pack_bf16x2(p[8 * u + 6], p[8 * u + 7]));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.pt_full);
        if (!(ok = warp_wait(&sm.dp_full, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
        tc_fence_after();
        // dS^T in two 32-column steps (fewer live registers); the dS^T tile is
        // free once the previous pair's dK and dQ^T MMAs finished
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_base + kColR0 + half * HC + hh * 32, r);
          tmem_wait_ld();
          if (hh == 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.dp_empty);
          }
          uint32_t dsk[16];
#pragma unroll
          for (int x = 0; x < 32; x += 4) {
            const float4 d4 = *reinterpret_cast<const float4*>(ds_v + hh * 32 + x);
            const float* pp = p + hh * 32 + x;
            dsk[x / 2] = pack_bf16x2(pp[0] * (__uint_as_float(r[x]) - d4.x), pp[1] * (__uint_as_float(r[x + 1]) - d4.y));
            dsk[x / 2 + 1] =
                pack_bf16x2(pp[2] * (__uint_as_float(r[x + 2]) - d4.z), pp[3] * (__uint_as_float(r[x + 3]) - d4.w));
          }
          if (hh == 0 && !(ok = warp_wait(&sm.ds_done, (qd & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)))
            break;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int uu = hh * 4 + u;
            st_shared_v4(dst_row + ((uu ^ (krow & 7)) << 4), dsk[4 * u], dsk[4 * u + 1], dsk[4 * u + 2],
                         dsk[4 * u + 3]);
          }
        }
        if (!ok) break;
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.dst_full);
      }
      if (!ok) break;
      if (!(ok = warp_wait(&sm.acc_full, ki & 1, abort_flag, prm.status, prm.timeout_ns))) break;
      tc_fence_after();
#pragma unroll
      for (int part = 0; part < 2; ++part) {
        __nv_bfloat16* dst = part == 0 ? dv_row : dk_row;
        const float f = part == 0 ? 1.0f : prm.scale;
#pragma unroll
        for (int g = 0; g < HD / 32; ++g) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_base + (part == 0 ? kColFuDv : kColFuDk) + half * HD + g * 32, r);
          tmem_wait_ld();
          if (row_ok) {
#pragma unroll
            for (int x = 0; x < 32; x += 8) {
              uint4 v;
              v.x = pack_bf16x2(__uint_as_float(r[x + 0]) * f, __uint_as_float(r[x + 1]) * f);
              v.y = pack_bf16x2(__uint_as_float(r[x + 2]) * f, __uint_as_float(r[x + 3]) * f);
              v.z = pack_bf16x2(__uint_as_float(r[x + 4]) * f, __uint_as_float(r[x + 5]) * f);
              v.w = pack_bf16x2(__uint_as_float(r[x + 6]) * f, __uint_as_float(r[x + 7]) * f);
              *reinterpret_cast<uint4*>(dst + g * 32 + x) = v;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acc_empty);
      qd0 += L;
      ++ki;
    }
  } else {
    setmaxnreg_dec<kFuRegDrain>();
    // 4 dQ drain warps, one per TMEM lane quarter: for dQ_i^T the TMEM lane is
    // the d index.  Each thread adds its d of all 128 query rows of block i,
    // one fp32 reduction per row; the warp covers 32 consecutive d of a row
    // (one 128-byte segment).  RQ is released once both halves are read.
    const uint32_t quarter = warp & 3;
    const uint32_t dcol = quarter * 32 + lane;
    const uint32_t lane_base = (quarter * 32) << 16;
    uint32_t qd0 = 0, kk = 0;
    bool ok = true;
    for (;;) {
      int w;
      if (!(ok = next_item(kk, w, false)) || w < 0) break;
      const int h = w / prm.nq;
      BlockSteps<kMode> tl;
      tl.init(prm.ptr, prm.idx, h, w % prm.nq, prm.nk_fine, prm.k_rows_per_tile, prm.list_shift);
      const int L = tl.count_warp();
      if (L <= 0) continue;
      for (int t = 0; t < L; ++t) {
        const uint32_t qd = qd0 + t;
        int i, ih;
        uint32_t bits;
        tl.next(i, ih, bits);
        if (!(ok = warp_wait(&sm.ds_done, qd & 1, abort_flag, prm.status, prm.timeout_ns))) break;
        tc_fence_after();
#pragma unroll
        for (int g = 0; g < 2; ++g) {
          // query half g of the tile: rows of 64-row block lo / hi (paired), or
          // rows g * 64 .. of the 128-row query block; a missing block (-1)
          // has dS^T = 0 there and is not added
          const int blk = tl.pair ? (g ? ih : i) : 0;
          const int64_t row0 = tl.pair ? 64 * (int64_t)blk : (int64_t)i * kTile + 64 * g;
          float* dst = dq_acc + (((int64_t)h * prm.Np + row0) * D + dcol);
          uint32_t r[64];
          tmem_ld64(tmem + lane_base + kColRQ + g * 64, r);
          if (g == 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.dq_empty);
          }
          if (dcol < (uint32_t)D && blk >= 0) {
#pragma unroll
            for (int x = 0; x < 64; ++x) red_add_f32(dst + (int64_t)x * D, __uint_as_float(r[x]));
          }
        }
      }
      if (!ok) break;
      qd0 += L;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// dQ = scale * accumulator, bf16, rows < N: thread = 8 consecutive d of one (row, head)
__global__ void __launch_bounds__(256) bwd_dq_finalize_kernel(const float* __restrict__ acc, int64_t N, int64_t Np,
                                                              int H, int d, int64_t rs, float scale,
                                                              __nv_bfloat16* __restrict__ dq) {
  const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int per_row = H * d / 8;
  if (g >= N * per_row) return;
  const int64_t r = g / per_row;
  const int e = (int)(g % per_row) * 8;
  const int h = e / d, c = e % d;
  const float4* src = reinterpret_cast<const float4*>(acc + ((int64_t)h * Np + r) * d + c);
  const float4 a = src[0], b = src[1];
  uint4 v;
  v.x = pack_bf16x2(a.x * scale, a.y * scale);
  v.y = pack_bf16x2(a.z * scale, a.w * scale);
  v.z = pack_bf16x2(b.x * scale, b.y * scale);
  v.w = pack_bf16x2(b.z * scale, b.w * scale);
  *reinterpret_cast<uint4*>(dq + r * rs + e) = v;
}

// ----------------------------------------------------------------- launcher
size_t attn_bwd_tc_ws(const AttnProblem& p) {
  const size_t Np = (size_t)((p.N + kTile - 1) / kTile) * kTile;
  return 2 * (size_t)p.H * Np * sizeof(float) + (size_t)p.H * Np * p.d * sizeof(float) + 16;  // + item counter
}

constexpr size_t kMaxDynSmem = 232448;  // 227 KB opt-in per block on sm_100/sm_103
static_assert(sizeof(FusedSmem<128>) <= kMaxDynSmem, "fused backward shared layout exceeds the per-block limit");

template <int D, int kMode>
static cudaError_t launch_bwd_fused(const AttnProblem& p, const CUtensorMap* tm, BwdParams prm, float* dq_acc,
                                   __nv_bfloat16* dq, int sms, cudaStream_t s) {
  const int n_items = prm.n_items;
  const int grid = n_items < sms ? n_items : sms;
  const size_t smem = sizeof(FusedSmem<D>);
  cudaError_t e =
      cudaFuncSetAttribute(bwd_fused_kernel<D, kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  // the setmaxnreg split assumes exactly kFuRegLaunch registers per thread at
  // launch: with fewer, the increases would wait for registers that never come
  cudaFuncAttributes fa;
  e = cudaFuncGetAttributes(&fa, bwd_fused_kernel<D, kMode>);
  if (e != cudaSuccess) return e;
  if (fa.numRegs != kFuRegLaunch) return cudaErrorInvalidConfiguration;
  bwd_fused_kernel<D, kMode><<<grid, kFuThreads, smem, s>>>(tm[0], tm[1], tm[2], tm[3], tm[4], tm[5], prm, dq_acc);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t n8 = p.N * p.H * D / 8;
  bwd_dq_finalize_kernel<<<(unsigned)((n8 + 255) / 256), 256, 0, s>>>(dq_acc, p.N, prm.Np, p.H, D, p.row_stride,
                                                                      p.scale, dq);
  return cudaGetLastError();
}

cudaError_t launch_attn_bwd_tc(const AttnProblem& p, const void* q, const void* k, const void* v, const void* o,
                               const float* lse, const void* dout, const int32_t* row_ptr, const int32_t* col_idx,
                               const int32_t* col_ptr_t, const int32_t* row_idx_t, void* dq, void* dk, void* dv,
                               void* ws, int32_t* status, uint64_t timeout_ns, int sms, cudaStream_t stream) {
  (void)row_ptr;
  (void)col_idx;  // the fused kernel walks the transposed lists only
  const int nt = (int)((p.N + kTile - 1) / kTile);  // 128-row tiles
  if (nt == 0) return cudaSuccess;
  const int64_t Np = (int64_t)nt * kTile;
  float* lse2 = static_cast<float*>(ws);
  float* dsum = lse2 + (size_t)p.H * Np;
  float* dq_acc = dsum + (size_t)p.H * Np;
  int32_t* item_counter = reinterpret_cast<int32_t*>(dq_acc + (size_t)p.H * Np * p.d);
  // one clear for the dQ accumulator and the item counter right after it
  cudaError_t e = cudaMemsetAsync(dq_acc, 0, (size_t)p.H * Np * p.d * sizeof(float) + 16, stream);
  if (e != cudaSuccess) return e;
  bwd_pre_kernel<<<(unsigned)((Np + 7) / 8), 256, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(o), static_cast<const __nv_bfloat16*>(dout), lse, p.N, Np, p.H, p.d,
      p.row_stride, lse2, dsum);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // 0: 128-row blocks on both sides; 1: 128-row query blocks, 64-row key
  // blocks (merged lists); 2: 64-row query blocks, 128-row key blocks, paired
  // into 128-row tiles; 3: 64-row blocks on both sides, merged or paired per item
  const int mode = p.block == 128 ? (p.block_k == 128 ? 0 : 1) : (p.block_k == 128 ? 2 : 3);
  CUtensorMap tm[6];  // Q, K, V, dO as 128-row boxes, then Q and dO as 64-row boxes
  const uint64_t inner = (uint64_t)p.H * p.d, stride = (uint64_t)p.row_stride * 2;
  const void* bases[6] = {q, k, v, dout, q, dout};
  for (int x = 0; x < 6; ++x)
    if (!encode_tmap_2d_bf16(&tm[x], bases[x], inner, p.N, stride, 64, x < 4 ? kTile : 64))
      return cudaErrorInvalidValue;
  BwdParams a{};
  a.ptr = col_ptr_t;
  a.idx = row_idx_t;
  a.lse2 = lse2;
  a.dsum = dsum;
  a.out0 = static_cast<__nv_bfloat16*>(dv);
  a.out1 = static_cast<__nv_bfloat16*>(dk);
  a.status = status;
  a.N = p.N;
  a.Np = Np;
  a.rs = p.row_stride;
  a.H = p.H;
  a.nq = nt;
  a.n_items = p.H * nt;
  a.nk_fine = p.nk;
  a.k_rows_per_tile = p.block_k == 64 ? 2 : 1;
  a.list_shift = p.block == 64 ? 1 : 0;
  a.scale = p.scale;
  a.scale_log2 = p.scale * 1.4426950408889634f;
  a.timeout_ns = timeout_ns;
  a.item_counter = item_counter;
  __nv_bfloat16* dqb = static_cast<__nv_bfloat16*>(dq);
#define UT_BWD_LAUNCH(DD, MM) launch_bwd_fused<DD, MM>(p, tm, a, dq_acc, dqb, sms, stream)
#define UT_BWD_MODES(DD)                                                                    \
  (mode == 0 ? UT_BWD_LAUNCH(DD, 0)                                                         \
             : (mode == 1 ? UT_BWD_LAUNCH(DD, 1) : (mode == 2 ? UT_BWD_LAUNCH(DD, 2) : UT_BWD_LAUNCH(DD, 3))))
  if (p.d == 64) return UT_BWD_MODES(64);
  return UT_BWD_MODES(128);
#undef UT_BWD_MODES
#undef UT_BWD_LAUNCH
}

}  // namespace ut
