// Block-sparse attention forward on the 5th-generation tensor cores (Sec. 3.3):
//   O_i = softmax(Q_i K_{S_i}^T * scale) V_{S_i}
// for every (head, query block i), iterating only the listed key blocks.
//
// Persistent kernel, one CTA per SM, work items (h, i) in head-major order so
// that the CTAs in flight share one head's K/V in L2.  Roles (192 threads):
//   warp 0      TMA producers: lane 0 streams the item's Q tile and the K tiles,
//               lane 1 the V tiles, each into its own 3-stage ring of
//               128B-swizzled shared tiles.  A K stage is released by the MMA
//               that consumed it (S = Q K^T), a V stage by O += P V.
//   warp 1      TMEM owner and MMA issuer (one elected thread):
//               S_t = Q K_t^T with Q read from TMEM (only K from shared
//               memory) into one of two TMEM S buffers, two key blocks ahead
//               of O += P_u V_u with P also read from TMEM (only V from shared
//               memory).
//   warps 2-5   softmax: thread = query row = TMEM lane.  At the start of an
//               item they copy its Q tile from shared memory into TMEM (the A
//               operand of S), then finish the previous item (normalise O,
//               write O in bf16 and LSE in fp32, natural log) while the tensor
//               core already computes the new item's first S blocks.  Per key
//               block: read S_t from TMEM, mask the ragged last key block, keep
//               a running row maximum (rescaling O in TMEM only when the
//               maximum grew by more than 2^8, so the exponentials stay
//               bounded), write P_t as bf16 pairs into the TMEM P buffer.
// Reading Q from TMEM halves the shared-memory operand traffic of S = Q K^T;
// per key block the shared memory then serves K and V to the tensor core and
// their TMA writes (128 KB), about what the two 128 x 128 x 128 products take.
// TMEM columns: S0 [0,128), S1 [128,256), O [256,256+D), P [384,448),
// Q [448,448+D/2).
// Blocks of 64 rows (b_q or b_kv) are served by the same 128 x 128 tiles:
//   b_kv = 64:  two listed 64-row key blocks fill one 128-row key tile (two
//               TMA boxes per operand, PairList): consecutive entries of the
//               list for b_q = 128 (nothing discarded), the two 64-row query
//               blocks' lists in lockstep for b_q = 64 (rows 0-63 see the low
//               half of the tile, rows 64-127 the high half);
//   b_q = 64, b_kv = 128:  the item's two lists are merged into 128-row key
//               tiles with a mask of the listed 64 x 64 sub-blocks (TileList).
// The softmax sets the scores of sub-blocks a row does not see to -inf.  Rows
// that see no key end with O = 0 and LSE = -inf.
// Every wait is bounded; on expiry the kernel records UT_ERR_TIMEOUT,
// drains its own copies and MMAs, frees TMEM and returns.
#include "common.cuh"
#include "kernels.h"

namespace ut {

constexpr int kBM = 128;  // query rows per tile
constexpr int kBN = 128;  // key rows per tile
constexpr int kFwdThreads = 192;
constexpr int kStages = 3;                       // K and V ring depth
constexpr uint32_t kTileChunkBytes = 128 * 128;  // 128 rows x 128 bytes (64 bf16)
constexpr uint32_t kColO = 256, kColP = 384, kColQ = 448;  // TMEM column bases

template <int D>
struct FwdSmem {
  static constexpr int kChunks = D / 64;
  static constexpr uint32_t kQBytes = kBM * D * 2;
  static constexpr uint32_t kKVBytes = kBN * D * 2;
  alignas(1024) uint8_t q[kQBytes];
  alignas(1024) uint8_t k[kStages][kKVBytes];
  alignas(1024) uint8_t v[kStages][kKVBytes];
  uint64_t q_full, q_empty;    // shared Q tile: TMA landed / copied into TMEM
  uint64_t qt_full, qt_empty;  // TMEM Q: written by the softmax warps / last S of the item done
  uint64_t k_full[kStages], v_full[kStages], k_empty[kStages], v_empty[kStages];
  uint64_t s_full[2], s_empty[2];
  uint64_t p_full, pv_done;    // one TMEM P buffer
  uint64_t o_empty, mma_done;
  uint32_t tmem_base;
  int abort_flag;
};

struct FwdParams {
  const int32_t* row_ptr;   // fine lists: nq_fine rows per head
  const int32_t* col_idx;
  int nq_fine;              // query blocks per head in the lists
  int q_rows_per_tile;      // 1 (b_q = 128) or 2 (b_q = 64)
  int list_shift;           // 0 (b_kv = 128) or 1 (b_kv = 64)
  __nv_bfloat16* o;
  float* lse;
  int32_t* status;
  int64_t N;
  int64_t rs;  // elements between tokens
  int H, nq;         // nq: 128-row query tiles per head
  int n_items;
  float scale_log2;  // softmax scale * log2(e)
  uint64_t timeout_ns;
};

template <int D, int kMode>
__global__ void __launch_bounds__(kFwdThreads, 1)
    attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_k64,
                       const __grid_constant__ CUtensorMap tm_v64, const FwdParams prm) {
  constexpr bool kSub = kMode != 0;  // 64-row blocks on at least one side
  extern __shared__ uint8_t smem_raw[];
  FwdSmem<D>& sm = *reinterpret_cast<FwdSmem<D>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int C = FwdSmem<D>::kChunks;
  const uint32_t warp = warp_id();
  const uint32_t lane = lane_id();
  volatile int* abort_flag = &sm.abort_flag;

  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    mbar_init(&sm.q_empty, 4);
    mbar_init(&sm.qt_full, 4);
    mbar_init(&sm.qt_empty, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.k_full[s], 1);
      mbar_init(&sm.v_full[s], 1);
      mbar_init(&sm.k_empty[s], 1);
      mbar_init(&sm.v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_empty[s], 4);
    }
    mbar_init(&sm.p_full, 4);
    mbar_init(&sm.pv_done, 1);
    mbar_init(&sm.o_empty, 4);
    mbar_init(&sm.mma_done, 1);
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

  const int G = gridDim.x;
  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // lane 0 streams Q and K, lane 1 streams V: each ring is released by the
    // MMA that consumes it (K after S = Q K^T, V after O += P V), so neither
    // waits for the other.
    if (lane < 2) {
      const bool is_k = lane == 0;
      if (is_k) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
        if (kMode >= 2) tma_prefetch_desc(&tm_k64);
      } else {
        tma_prefetch_desc(&tm_v);
        if (kMode >= 2) tma_prefetch_desc(&tm_v64);
      }
      const uint64_t pol_kv = policy_evict_last();
      const uint64_t pol_q = policy_evict_first();
      uint64_t* full = is_k ? sm.k_full : sm.v_full;
      uint64_t* empty = is_k ? sm.k_empty : sm.v_empty;
      uint8_t* ring = is_k ? &sm.k[0][0] : &sm.v[0][0];
      const void* tmap = is_k ? static_cast<const void*>(&tm_k) : static_cast<const void*>(&tm_v);
      const void* tmap64 = is_k ? static_cast<const void*>(&tm_k64) : static_cast<const void*>(&tm_v64);
      uint32_t qi = 0, kv = 0;
      bool ok = true;
      for (int w = blockIdx.x; w < prm.n_items && ok; w += G) {
        const int h = w / prm.nq, i = w % prm.nq;
        BlockSteps<kMode> tl;
        tl.init(prm.row_ptr, prm.col_idx, h, i, prm.nq_fine, prm.q_rows_per_tile, prm.list_shift);
        if (tl.empty()) continue;
        if (is_k) {
          if (!(ok = mbar_wait(&sm.q_empty, (qi & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
          mbar_expect_tx(&sm.q_full, FwdSmem<D>::kQBytes);
          for (int c = 0; c < C; ++c)
            tma_load_2d(sm.q + c * kTileChunkBytes, &tm_q, &sm.q_full, h * D + c * 64, i * kBM, pol_q);
          ++qi;
        }
        int j, jh;
        uint32_t bits;
        for (; tl.next(j, jh, bits); ++kv) {
          const uint32_t st = kv % kStages, n = kv / kStages;
          if (!(ok = mbar_wait(&empty[st], (n & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
          mbar_expect_tx(&full[st], FwdSmem<D>::kKVBytes);
          uint8_t* dst = ring + st * FwdSmem<D>::kKVBytes;
          if (tl.pair) {  // two 64-row boxes: rows 0-63 and 64-127 of each 128-row sub-tile
            const int b0 = PairList::load_lo(j, jh), b1 = PairList::load_hi(j, jh);
            for (int c = 0; c < C; ++c) {
              tma_load_2d(dst + c * kTileChunkBytes, tmap64, &full[st], h * D + c * 64, b0 * 64, pol_kv);
              tma_load_2d(dst + c * kTileChunkBytes + 64 * 128, tmap64, &full[st], h * D + c * 64, b1 * 64, pol_kv);
            }
          } else {
            for (int c = 0; c < C; ++c)
              tma_load_2d(dst + c * kTileChunkBytes, tmap, &full[st], h * D + c * 64, j * kBN, pol_kv);
          }
        }
      }
      // Drain: every copy this lane issued has landed before the CTA may exit.
      auto drain = [&](uint64_t* bar, uint32_t parity) {
        if (!mbar_drain(bar, parity, kDrainTimeoutNs)) set_status(prm.status, UT_ERR_TIMEOUT);
      };
      if (qi > 0) drain(&sm.q_full, (qi - 1) & 1);
      for (uint32_t u = (kv >= kStages ? kv - kStages : 0); u < kv; ++u)
        drain(&full[u % kStages], (u / kStages) & 1);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------- MMA issuer
    // The whole warp runs this loop converged; every MMA and commit is issued
    // by one elected lane (see mma_bf16_ss_w), waits are warp-uniform.
    {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t idesc_o = idesc_bf16_f32(kBM, D, false, true);
      uint32_t qi = 0, oi = 0, kv0 = 0, sc0 = 0;
      bool ok = true;
      for (int w = blockIdx.x; w < prm.n_items && ok; w += G) {
        BlockSteps<kMode> tl;
        tl.init(prm.row_ptr, prm.col_idx, w / prm.nq, w % prm.nq, prm.nq_fine, prm.q_rows_per_tile, prm.list_shift);
        const int L = tl.count_warp();
        if (L <= 0) continue;
        // Q of this item in TMEM (the softmax warps copied it there)
        if (!(ok = warp_wait(&sm.qt_full, qi & 1, abort_flag, prm.status, prm.timeout_ns))) break;
        // S runs two key blocks ahead of P V: S_{u+2} goes into the S buffer
        // that softmax u has just read, so the tensor core computes it while
        // the softmax works, and PV_u follows as soon as P_u is in TMEM.
        auto issue_s = [&](int t) -> bool {
          const uint32_t kv = kv0 + t, st = kv % kStages, n = kv / kStages;
          const uint32_t sc = sc0 + t, sb = sc & 1, ns = sc >> 1;
          if (!warp_wait(&sm.k_full[st], n & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
          if (!warp_wait(&sm.s_empty[sb], (ns & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)) return false;
          tc_fence_after();
          const uint32_t k_addr = smem_u32(sm.k[st]);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk >> 2) * kTileChunkBytes + (kk & 3) * 32;
            mma_bf16_ts_w(tmem + sb * 128, tmem + kColQ + kk * 8, sdesc_sw128(k_addr + off, 16, 1024), idesc_s,
                          kk > 0);
          }
          mma_commit_w(&sm.s_full[sb]);
          mma_commit_w(&sm.k_empty[st]);
          if (t == L - 1) mma_commit_w(&sm.qt_empty);  // Q's TMEM columns are free once these S are done
          return true;
        };
        auto issue_pv = [&](int u) -> bool {
          const uint32_t kv = kv0 + u, st = kv % kStages, n = kv / kStages;
          const uint32_t sc = sc0 + u;
          if (!warp_wait(&sm.p_full, sc & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
          if (!warp_wait(&sm.v_full[st], n & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
          if (u == 0 && !warp_wait(&sm.o_empty, (oi & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)) return false;
          tc_fence_after();
          const uint32_t v_addr = smem_u32(sm.v[st]);
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)
            mma_bf16_ts_w(tmem + kColO, tmem + kColP + kk * 8, sdesc_sw128(v_addr + kk * 2048, kTileChunkBytes, 1024),
                          idesc_o, (u > 0 || kk > 0));
          mma_commit_w(&sm.pv_done);
          mma_commit_w(&sm.v_empty[st]);
          return true;
        };
        ok = issue_s(0) && (L < 2 || issue_s(1));
        for (int u = 0; u < L && ok; ++u) {
          if (u + 2 < L && !(ok = issue_s(u + 2))) break;
          ok = issue_pv(u);
        }
        kv0 += L;
        sc0 += L;
        ++qi;
        ++oi;
      }
      // Drain: all MMAs issued by this warp complete before TMEM is freed.
      mma_commit_w(&sm.mma_done);
      if (!mbar_drain(&sm.mma_done, 0, kDrainTimeoutNs)) set_status(prm.status, UT_ERR_TIMEOUT);
    }
  } else {
    // ------------------------------------------------------------- softmax
    const uint32_t quarter = warp & 3;
    const uint32_t row = quarter * 32 + lane;
    const uint32_t lane_base = (quarter * 32) << 16;
    const float c = prm.scale_log2;
    uint32_t sc0 = 0, qi = 0;
    bool ok = true;
    const uint32_t rh = row >> 6;  // which 64-row half of the query tile
    // Q tile of the next item: shared memory (128B-swizzled, as TMA wrote it)
    // -> registers -> TMEM, this thread's row, bf16 pairs (element 2u in the
    // low half of column u), the A-operand layout of S = Q K^T.
    auto load_q = [&]() -> bool {
      if (!warp_wait(&sm.q_full, qi & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
      if (!warp_wait(&sm.qt_empty, (qi & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns)) return false;
      tc_fence_after();
#pragma unroll
      for (int cc = 0; cc < C; ++cc) {
        uint32_t qv[32];
        const uint32_t base = smem_u32(sm.q) + cc * kTileChunkBytes + row * 128;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                       : "=r"(qv[4 * u]), "=r"(qv[4 * u + 1]), "=r"(qv[4 * u + 2]), "=r"(qv[4 * u + 3])
                       : "r"(base + ((u ^ (row & 7)) << 4)));
        tmem_st32(tmem + lane_base + kColQ + cc * 32, qv);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&sm.qt_full);
        mbar_arrive(&sm.q_empty);
      }
      ++qi;
      return true;
    };
    // The previous item's epilogue (O / l -> bf16, LSE) runs after the next
    // item's Q is in TMEM, so the tensor core computes the next S blocks
    // meanwhile.
    bool pend = false;
    float e_m = 0.f, e_l = 0.f;
    uint32_t e_last = 0;
    int64_t e_grow = 0;
    int e_h = 0;
    auto epilogue = [&]() -> bool {
      if (!warp_wait(&sm.pv_done, e_last & 1, abort_flag, prm.status, prm.timeout_ns)) return false;
      tc_fence_after();
      const bool row_ok = e_grow < prm.N;
      __nv_bfloat16* orow = prm.o + e_grow * prm.rs + (int64_t)e_h * D;
      const float inv = (!kSub || e_l > 0.f) ? 1.0f / e_l : 0.f;  // a row that saw no key: O = 0, LSE = -inf
#pragma unroll
      for (int g = 0; g < D / 32; ++g) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_base + kColO + g * 32, r);
        tmem_wait_ld();
        if (row_ok) {
#pragma unroll
          for (int x = 0; x < 32; x += 8) {
            uint4 v;
            v.x = pack_bf16x2(__uint_as_float(r[x + 0]) * inv, __uint_as_float(r[x + 1]) * inv);
            v.y = pack_bf16x2(__uint_as_float(r[x + 2]) * inv, __uint_as_float(r[x + 3]) * inv);
            v.z = pack_bf16x2(__uint_as_float(r[x + 4]) * inv, __uint_as_float(r[x + 5]) * inv);
            v.w = pack_bf16x2(__uint_as_float(r[x + 6]) * inv, __uint_as_float(r[x + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + g * 32 + x) = v;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.o_empty);
      if (row_ok)
        prm.lse[(int64_t)e_h * prm.N + e_grow] =
            (!kSub || e_l > 0.f) ? (e_m + log2f(e_l)) * 0.69314718055994531f : -INFINITY;
      return true;
    };
    for (int w = blockIdx.x; w < prm.n_items && ok; w += G) {
      const int h = w / prm.nq, i = w % prm.nq;
      BlockSteps<kMode> tl;
      tl.init(prm.row_ptr, prm.col_idx, h, i, prm.nq_fine, prm.q_rows_per_tile, prm.list_shift);
      const int L = tl.count_warp();
      const int64_t grow = (int64_t)i * kBM + row;
      if (L <= 0) {
        if (grow < prm.N) {
          __nv_bfloat16* orow = prm.o + grow * prm.rs + (int64_t)h * D;
          for (int e = 0; e < D; e += 8) *reinterpret_cast<uint4*>(orow + e) = make_uint4(0, 0, 0, 0);
          prm.lse[(int64_t)h * prm.N + grow] = -INFINITY;
        }
        continue;
      }
      if (!(ok = load_q())) break;
      if (pend && !(ok = epilogue())) break;
      pend = false;
      float m_used = 0.f, l = 0.f;
      int j_next = 0, jh_next = -1;
      uint32_t bits_next = 0;
      tl.next(j_next, jh_next, bits_next);
      for (int t = 0; t < L; ++t) {
        const int j = j_next, jh = jh_next;
        const uint32_t bits = bits_next;
        if (t + 1 < L) tl.next(j_next, jh_next, bits_next);  // the next tile's blocks, fetched a tile ahead
        const uint32_t sc = sc0 + t, sb = sc & 1, ns = sc >> 1;
        if (!(ok = warp_wait(&sm.s_full[sb], ns & 1, abort_flag, prm.status, prm.timeout_ns))) break;
        tc_fence_after();
        // all four 32-column loads in flight before one wait
        uint32_t r[kBN];
#pragma unroll
        for (int g = 0; g < kBN / 32; ++g)
          tmem_ld32(tmem + lane_base + sb * 128 + g * 32, *reinterpret_cast<uint32_t(*)[32]>(&r[g * 32]));
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.s_empty[sb]);
        float s[kBN];
#pragma unroll
        for (int x = 0; x < kBN; ++x) s[x] = __uint_as_float(r[x]);
        // ragged last key block: columns past N do not exist; 64-column
        // halves of the tile not listed for this row's half are masked
        const uint32_t cols = kSub ? (bits >> (2 * rh)) & 3u : 3u;
        if (tl.pair) {  // each half holds its own 64-row key block
          const int64_t nv0 = prm.N - 64 * (int64_t)PairList::load_lo(j, jh);
          const int64_t nv1 = prm.N - 64 * (int64_t)PairList::load_hi(j, jh);
          if (nv0 < 64) {
#pragma unroll
            for (int x = 0; x < 64; ++x)
              if (x >= nv0) s[x] = -INFINITY;
          }
          if (nv1 < 64) {
#pragma unroll
            for (int x = 64; x < kBN; ++x)
              if (x - 64 >= nv1) s[x] = -INFINITY;
          }
        } else {
          const int64_t nv = prm.N - (int64_t)j * kBN;
          if (nv < kBN) {
#pragma unroll
            for (int x = 0; x < kBN; ++x)
              if (x >= nv) s[x] = -INFINITY;
          }
        }
        if (kSub) {  // a masked half is the same for the whole warp (rh is per warp)
          if (!(cols & 1u)) {
#pragma unroll
            for (int x = 0; x < kBN / 2; ++x) s[x] = -INFINITY;
          }
          if (!(cols & 2u)) {
#pragma unroll
            for (int x = kBN / 2; x < kBN; ++x) s[x] = -INFINITY;
          }
        }
        // row maximum as a tree (8 independent chains) rather than one long chain
        float m8[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) m8[q] = s[q];
#pragma unroll
        for (int x = 8; x < kBN; ++x) m8[x & 7] = fmaxf(m8[x & 7], s[x]);
        float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                         fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
        // a row may see nothing in this tile: keep the reference maximum
        // finite so that exp2(-inf - m) stays 0 (not NaN)
        mx = kSub ? fmaxf(mx * c, -1e30f) : mx * c;
        if (t == 0) {
          m_used = mx;
        } else {
          const bool need = mx > m_used + 8.0f;
          if (__any_sync(0xffffffffu, need)) {
            // O holds P V up to the previous key block once that MMA finished
            if (!(ok = warp_wait(&sm.pv_done, (sc & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
            tc_fence_after();
            const float alpha = need ? ex2_approx(m_used - mx) : 1.0f;
#pragma unroll
            for (int g = 0; g < D / 32; ++g) {
              uint32_t r[32];
              tmem_ld32(tmem + lane_base + kColO + g * 32, r);
              tmem_wait_ld();
#pragma unroll
              for (int x = 0; x < 32; ++x) r[x] = __float_as_uint(__uint_as_float(r[x]) * alpha);
              tmem_st32(tmem + lane_base + kColO + g * 32, r);
            }
            tmem_wait_st();
            if (need) {
              l *= alpha;
              m_used = mx;
            }
          }
        }
        // P = exp2(s * c - m_used), rounded to bf16 for the P V MMA
        uint32_t pk[kBN / 2];
        float l8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int hc = 0; hc < 2; ++hc) {
          if (kSub && !((cols >> hc) & 1u)) {  // a masked half: P = 0 without the exponentials
#pragma unroll
            for (int x = hc * (kBN / 2); x < (hc + 1) * (kBN / 2); x += 2) pk[x / 2] = 0u;
            continue;
          }
#pragma unroll
          for (int x = hc * (kBN / 2); x < (hc + 1) * (kBN / 2); x += 2) {
            const float p0 = ex2_approx(fmaf(s[x], c, -m_used));
            const float p1 = ex2_approx(fmaf(s[x + 1], c, -m_used));
            l8[(x >> 1) & 7] += p0 + p1;
            pk[x / 2] = pack_bf16x2(p0, p1);
          }
        }
        l += ((l8[0] + l8[1]) + (l8[2] + l8[3])) + ((l8[4] + l8[5]) + (l8[6] + l8[7]));
        // the TMEM P buffer is free once the previous key block's P V finished
        if (!(ok = warp_wait(&sm.pv_done, (sc & 1) ^ 1, abort_flag, prm.status, prm.timeout_ns))) break;
        tc_fence_after();
        tmem_st32(tmem + lane_base + kColP, *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
        tmem_st32(tmem + lane_base + kColP + 32, *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.p_full);
      }
      if (!ok) break;
      pend = true;
      e_m = m_used;
      e_l = l;
      e_last = sc0 + L - 1;
      e_grow = grow;
      e_h = h;
      sc0 += L;
    }
    if (ok && pend) ok = epilogue();
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

static_assert(sizeof(FwdSmem<128>) + 1024 <= 232448, "forward shared layout exceeds the per-block limit");

template <int D, int kMode>
static cudaError_t launch_d(const AttnProblem& p, const CUtensorMap& tq, const CUtensorMap& tk,
                            const CUtensorMap& tv, const CUtensorMap& tk64, const CUtensorMap& tv64,
                            const FwdParams& prm, int grid, cudaStream_t stream) {
  const size_t smem = sizeof(FwdSmem<D>) + 1024;
  cudaError_t e =
      cudaFuncSetAttribute(attn_fwd_tc_kernel<D, kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  attn_fwd_tc_kernel<D, kMode><<<grid, kFwdThreads, smem, stream>>>(tq, tk, tv, tk64, tv64, prm);
  return cudaGetLastError();
}

cudaError_t launch_attn_fwd_tc(const AttnProblem& p, const void* q, const void* k, const void* v,
                               const int32_t* row_ptr, const int32_t* col_idx, void* o, float* lse, int32_t* status,
                               uint64_t timeout_ns, int sms, cudaStream_t stream) {
  const int nt = (int)((p.N + kBM - 1) / kBM);  // 128-row tiles
  const int n_items = p.H * nt;
  if (n_items == 0) return cudaSuccess;
  // 0: 128-row blocks on both sides; 1: 64-row query blocks, 128-row key
  // blocks (merged lists); 2: 128-row query blocks, 64-row key blocks paired
  // into 128-row tiles; 3: 64-row blocks on both sides, merged or paired per item
  const int mode = p.block == 128 ? (p.block_k == 128 ? 0 : 2) : (p.block_k == 128 ? 1 : 3);
  CUtensorMap tq, tk, tv, tk64, tv64;  // K / V as 128-row and as 64-row boxes
  const uint64_t inner = (uint64_t)p.H * p.d;
  const uint64_t stride = (uint64_t)p.row_stride * 2;
  if (!encode_tmap_2d_bf16(&tq, q, inner, p.N, stride, 64, kBM) ||
      !encode_tmap_2d_bf16(&tk, k, inner, p.N, stride, 64, kBN) ||
      !encode_tmap_2d_bf16(&tv, v, inner, p.N, stride, 64, kBN) ||
      !encode_tmap_2d_bf16(&tk64, k, inner, p.N, stride, 64, 64) ||
      !encode_tmap_2d_bf16(&tv64, v, inner, p.N, stride, 64, 64))
    return cudaErrorInvalidValue;
  FwdParams prm{};
  prm.row_ptr = row_ptr;
  prm.col_idx = col_idx;
  prm.o = static_cast<__nv_bfloat16*>(o);
  prm.lse = lse;
  prm.status = status;
  prm.N = p.N;
  prm.rs = p.row_stride;
  prm.H = p.H;
  prm.nq = nt;
  prm.nq_fine = p.nq;
  prm.q_rows_per_tile = p.block == 64 ? 2 : 1;
  prm.list_shift = p.block_k == 64 ? 1 : 0;
  prm.n_items = n_items;
  prm.scale_log2 = p.scale * 1.4426950408889634f;
  prm.timeout_ns = timeout_ns;
  const int grid = n_items < sms ? n_items : sms;
#define UT_FWD_LAUNCH(DD, MM) launch_d<DD, MM>(p, tq, tk, tv, tk64, tv64, prm, grid, stream)
#define UT_FWD_MODES(DD)                                                                    \
  (mode == 0 ? UT_FWD_LAUNCH(DD, 0)                                                         \
             : (mode == 1 ? UT_FWD_LAUNCH(DD, 1) : (mode == 2 ? UT_FWD_LAUNCH(DD, 2) : UT_FWD_LAUNCH(DD, 3))))
  if (p.d == 64) return UT_FWD_MODES(64);
  return UT_FWD_MODES(128);
#undef UT_FWD_MODES
#undef UT_FWD_LAUNCH
}

}  // namespace ut
