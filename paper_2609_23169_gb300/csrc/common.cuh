// Device helpers shared by the kernels: status word, bounded mbarrier waits,
// TMA loads, tcgen05 (TMEM alloc, MMA, commit, ld/st) and descriptors.
// Everything is hand-written inline PTX for sm_103a.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ultratex.h"

#define UT_DEV __device__ __forceinline__

namespace ut {

// Limit for the drains on the way out of a kernel (its own in-flight TMA copies
// and MMAs must land before the CTA frees TMEM and exits).  Independent of the
// per-call wait limit, so that a tiny wait limit can never skip a drain.
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;

// ------------------------------------------------------------------ status
UT_DEV void set_status(int32_t* status, int32_t code) {
  if (status) atomicCAS(status, 0, code);
}

UT_DEV uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

UT_DEV uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

UT_DEV uint32_t lane_id() { return threadIdx.x & 31; }
UT_DEV uint32_t warp_id() { return __shfl_sync(0xffffffffu, threadIdx.x >> 5, 0); }

// ---------------------------------------------------------------- mbarrier
UT_DEV void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
UT_DEV void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
UT_DEV void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
UT_DEV void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
UT_DEV bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and records UT_ERR_TIMEOUT, raises the CTA's
// abort flag) if the phase with this parity has not completed within
// timeout_ns, or if another role of the CTA has already aborted.  A limit of 0
// gives up at the first wait that is not already satisfied (diagnostics).
// The spin loop lives inside one asm block: a loop written in C++ around the
// wait, placed between tcgen05.mma groups, keeps the tensor pipe from
// streaming consecutive MMAs (measured: ~2x fewer MMAs per cycle).
UT_DEV bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int32_t* status,
                      uint64_t timeout_ns) {
  uint32_t r;  // 1 = phase complete, 0 = timed out, 2 = CTA already aborted
  asm volatile(
      "{\n\t"
      ".reg .pred p, q;\n\t"
      ".reg .u64 t0, t1;\n\t"
      ".reg .u32 ab;\n\t"
      "mov.u32 %0, 1;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "@p bra UT_WAIT_DONE;\n\t"
      "setp.eq.u64 q, %4, 0;\n\t"
      "@q bra UT_WAIT_TIMEOUT;\n\t"
      "mov.u64 t0, %%globaltimer;\n\t"
      "UT_WAIT_LOOP:\n\t"
      "ld.volatile.shared.u32 ab, [%3];\n\t"
      "setp.ne.u32 q, ab, 0;\n\t"
      "@q bra UT_WAIT_ABORT;\n\t"
      "mov.u64 t1, %%globaltimer;\n\t"
      "sub.u64 t1, t1, t0;\n\t"
      "setp.gt.u64 q, t1, %4;\n\t"
      "@q bra UT_WAIT_TIMEOUT;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "@!p bra UT_WAIT_LOOP;\n\t"
      "bra UT_WAIT_DONE;\n\t"
      "UT_WAIT_ABORT:\n\t"
      "mov.u32 %0, 2;\n\t"
      "bra UT_WAIT_DONE;\n\t"
      "UT_WAIT_TIMEOUT:\n\t"
      "mov.u32 %0, 0;\n\t"
      "UT_WAIT_DONE:\n\t"
      "}"
      : "=r"(r)
      : "r"(smem_u32(bar)), "r"(parity), "r"(smem_u32(const_cast<int*>(abort_flag))), "l"(timeout_ns)
      : "memory");
  if (r == 1) return true;
  if (r == 0) {
    set_status(status, UT_ERR_TIMEOUT);
    *abort_flag = 1;
  }
  return false;
}

// Unbounded-count but time-bounded drain wait (no abort check): used on the way
// out of a kernel for the CTA's own copies and MMAs.
UT_DEV bool mbar_drain(uint64_t* bar, uint32_t parity, uint64_t timeout_ns) {
  uint32_t r;
  asm volatile(
      "{\n\t"
      ".reg .pred p, q;\n\t"
      ".reg .u64 t0, t1;\n\t"
      "mov.u32 %0, 1;\n\t"
      "mov.u64 t0, %%globaltimer;\n\t"
      "UT_DRAIN_LOOP:\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "@p bra UT_DRAIN_DONE;\n\t"
      "mov.u64 t1, %%globaltimer;\n\t"
      "sub.u64 t1, t1, t0;\n\t"
      "setp.gt.u64 q, t1, %3;\n\t"
      "@!q bra UT_DRAIN_LOOP;\n\t"
      "mov.u32 %0, 0;\n\t"
      "UT_DRAIN_DONE:\n\t"
      "}"
      : "=r"(r)
      : "r"(smem_u32(bar)), "r"(parity), "l"(timeout_ns)
      : "memory");
  return r == 1;
}

// Warp-collective form: every lane waits, and the warp agrees on the outcome
// (a timeout seen by any lane aborts all 32, keeping later .sync.aligned
// tcgen05 instructions convergent).
UT_DEV bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int32_t* status,
                      uint64_t timeout_ns) {
  bool r = mbar_wait(bar, parity, abort_flag, status, timeout_ns);
  return __all_sync(0xffffffffu, r);
}

// -------------------------------------------------------------------- TMA
UT_DEV void tma_prefetch_desc(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(tmap) : "memory");
}

// 2D tiled load, completion signalled on `bar` (complete_tx bytes).
UT_DEV void tma_load_2d(void* smem_dst, const void* tmap, uint64_t* bar, int32_t x, int32_t y,
                        uint64_t cache_policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(tmap), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(cache_policy)
      : "memory");
}

UT_DEV uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
UT_DEV uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

UT_DEV void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Warpgroup register reallocation (all four warps of a warpgroup execute it).
template <int N>
UT_DEV void setmaxnreg_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}
template <int N>
UT_DEV void setmaxnreg_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

// ------------------------------------------------------------ tile lists
// The tensor-core kernels work on 128-row tiles; the block lists may be at a
// 64-row granularity on either side (b_q, b_kv in {64, 128}).  An item (one
// 128-row tile of the listing side) then owns one or two fine list rows, and
// a listed 64-row block falls in tile j >> 1.  TileList merges the item's
// fine lists into ascending 128-row tiles and, per tile, a 2 x 2 mask of the
// 64 x 64 sub-blocks that are listed:
//   bit (2 * r + c): rows r * 64 .. r * 64 + 63 of the item's tile may see
//   columns c * 64 .. c * 64 + 63 of the listed tile.
// With 128-row blocks on both sides every listed tile has all four bits.
template <bool kSub>  // kSub: 64-row blocks on at least one side
struct TileList {
  const int32_t* a;   // fine list of the item's first (or only) row block
  const int32_t* b;   // fine list of its second 64-row block, if any
  int na, nb, pa, pb;
  int shift;          // 1 when the listed blocks have 64 rows
  bool split;         // the item holds two 64-row blocks (a: rows 0-63, b: rows 64-127)

  // item = (row-block tile t of head h); ptr/idx the fine lists with nfine
  // rows per head; rows_per_tile = 2 for 64-row blocks on the listing side.
  UT_DEV void init(const int32_t* ptr, const int32_t* idx, int h, int t, int nfine, int rows_per_tile,
                   int list_shift) {
    const int r0 = kSub ? t * rows_per_tile : t;
    const int64_t base = (int64_t)h * nfine;
    const int s0 = ptr[base + r0];
    a = idx + s0;
    na = ptr[base + r0 + 1] - s0;
    pa = pb = 0;
    b = a;
    nb = 0;
    split = false;
    shift = 0;
    if (kSub) {
      split = rows_per_tile == 2;
      shift = list_shift;
      if (split && r0 + 1 < nfine) {
        const int s1 = ptr[base + r0 + 1];
        b = idx + s1;
        nb = ptr[base + r0 + 2] - s1;
      }
    }
  }
  // next listed tile and its sub-block mask; false at the end
  UT_DEV bool next(int& tile, uint32_t& bits) {
    if (!kSub) {  // 128-row blocks on both sides: the list itself, every sub-block
      if (pa >= na) return false;
      tile = a[pa++];
      bits = 15u;
      return true;
    }
    const int ta = pa < na ? (a[pa] >> shift) : 0x7fffffff;
    const int tb = pb < nb ? (b[pb] >> shift) : 0x7fffffff;
    tile = ta < tb ? ta : tb;
    if (tile == 0x7fffffff) return false;
    const uint32_t rows_a = split ? 1u : 3u;
    bits = 0;
    while (pa < na && (a[pa] >> shift) == tile) {
      const uint32_t cols = shift ? (1u << (a[pa] & 1)) : 3u;
      bits |= ((rows_a & 1u) ? cols : 0u) | ((rows_a & 2u) ? cols << 2 : 0u);
      ++pa;
    }
    while (pb < nb && (b[pb] >> shift) == tile) {
      const uint32_t cols = shift ? (1u << (b[pb] & 1)) : 3u;
      bits |= cols << 2;
      ++pb;
    }
    return true;
  }
  UT_DEV bool empty() const { return na == 0 && nb == 0; }

  // number of listed tiles; the whole warp calls it (converged): the distinct
  // tiles of each list are counted 32 entries at a time with ballots, and a
  // tile listed by both lists is found by a binary search in the other one
  UT_DEV int count_warp() const {
    if (!kSub) return na;
    const uint32_t lane = threadIdx.x & 31u;
    int total = 0;
    for (int which = 0; which < 2; ++which) {
      const int32_t* x = which ? b : a;
      const int nx = which ? nb : na;
      const int32_t* y = which ? a : b;  // the other list (for shared tiles)
      const int ny = which ? na : nb;
      for (int i0 = 0; i0 < nx; i0 += 32) {
        const int i = i0 + (int)lane;
        bool fresh = false, shared = false;
        if (i < nx) {
          const int t = x[i] >> shift;
          fresh = i == 0 || (x[i - 1] >> shift) != t;
          if (fresh && which == 0 && ny > 0) {  // count a tile both lists hold once
            int lo = 0, hi = ny;                // first y entry with (y >> shift) >= t
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if ((y[mid] >> shift) < t) lo = mid + 1;
              else hi = mid;
            }
            shared = lo < ny && (y[lo] >> shift) == t;
          }
        }
        total += __popc(__ballot_sync(0xffffffffu, fresh)) - __popc(__ballot_sync(0xffffffffu, shared));
      }
    }
    return total;
  }
};

// 64-row blocks paired into 128-row tiles.  The tensor cores run 128 x 128
// tiles at full rate (an N = 64 product costs 44 cycles against 64 for
// N = 128, and M = 64 runs at the rate of M = 128), so a listed 64-row block
// of the listed side is loaded as one half of a 128-row operand tile (two
// 64-row TMA boxes) and paired with another one:
//   one list  (the item is one block of the listing side, 128 rows): step t
//             takes the consecutive entries (L[2t], L[2t+1]); every row of
//             the item sees both halves (no work is discarded);
//   two lists (the item holds two 64-row blocks a, b of the listing side):
//             step t takes (a[t], b[t]); rows 0-63 of the item see the low
//             half, rows 64-127 the high half.
// A missing entry is -1: that half is masked, and the loader fills it with
// the other half's block so that it holds finite values.
// bits: bit (2 * r + c) = rows r * 64 .. r * 64 + 63 of the item see columns
// c * 64 .. c * 64 + 63 of the tile (the encoding TileList uses).
struct PairList {
  const int32_t* a;
  const int32_t* b;
  int na, nb, t;
  bool two;

  // item = block t of head h on the listing side: one list (two = false) or
  // the two 64-row blocks 2 * item and 2 * item + 1 (two = true); nfine list
  // rows per head.
  UT_DEV void init(const int32_t* ptr, const int32_t* idx, int h, int item, int nfine, bool item_has_two) {
    const int64_t base = (int64_t)h * nfine;
    two = item_has_two;
    const int r0 = two ? 2 * item : item;
    const int s0 = ptr[base + r0];
    a = idx + s0;
    na = ptr[base + r0 + 1] - s0;
    b = a;
    nb = 0;
    if (two && r0 + 1 < nfine) {
      const int s1 = ptr[base + r0 + 1];
      b = idx + s1;
      nb = ptr[base + r0 + 2] - s1;
    }
    t = 0;
  }
  UT_DEV int count() const { return two ? (na > nb ? na : nb) : (na + 1) / 2; }
  UT_DEV bool empty() const { return na == 0 && nb == 0; }
  // next pair: the 64-row blocks of the low and high halves (never both -1)
  // and the visibility bits
  // step t of two lists in lockstep (also used on a TileList's own lists)
  UT_DEV static bool step_two(const int32_t* a, const int32_t* b, int na, int nb, int& t, int& lo, int& hi,
                              uint32_t& bits) {
    if (t >= (na > nb ? na : nb)) return false;
    lo = t < na ? a[t] : -1;
    hi = t < nb ? b[t] : -1;
    bits = (lo >= 0 ? 1u : 0u) | (hi >= 0 ? 8u : 0u);
    ++t;
    return true;
  }
  UT_DEV bool next(int& lo, int& hi, uint32_t& bits) {
    if (two) return step_two(a, b, na, nb, t, lo, hi, bits);
    if (t >= count()) return false;
    {
      lo = a[2 * t];
      hi = 2 * t + 1 < na ? a[2 * t + 1] : -1;
      bits = hi >= 0 ? 15u : 5u;
    }
    ++t;
    return true;
  }
  // the blocks the loader puts into the two halves (a missing one repeats the other)
  UT_DEV static int load_lo(int lo, int hi) { return lo >= 0 ? lo : hi; }
  UT_DEV static int load_hi(int lo, int hi) { return hi >= 0 ? hi : lo; }
};

// With 64-row blocks on both sides an item can merge its two lists into
// 128-row tiles (TileList) or step through them in lockstep (the two-list
// form of PairList, run on the TileList's own lists); each step costs one
// 128 x 128 tile.  Pairing takes max(na, nb) steps.  Merging takes the number
// of distinct tiles, at most the entry count and at most the tiles spanned
// between the first and the last entry: few for dense or clustered lists,
// about na + nb for sparse scattered ones.  Pairing is chosen when it takes
// fewer steps than that bound.  Only the lists' first and last entries are
// read, so every role takes the same choice at the cost of four loads.
UT_DEV bool pairing_is_shorter(const TileList<true>& tl) {
  if (tl.na + tl.nb == 0) return false;
  int first = 0x7fffffff, last = -1;
  if (tl.na > 0) {
    first = tl.a[0];
    last = tl.a[tl.na - 1];
  }
  if (tl.nb > 0) {
    first = tl.b[0] < first ? tl.b[0] : first;
    last = tl.b[tl.nb - 1] > last ? tl.b[tl.nb - 1] : last;
  }
  const int spanned = (last >> tl.shift) - (first >> tl.shift) + 1;
  const int entries = tl.na + tl.nb;
  const int paired = tl.na > tl.nb ? tl.na : tl.nb;
  return paired < (spanned < entries ? spanned : entries);
}

// The steps of an item over the listed side.  kMode 0: 128-row blocks on both
// sides (the list itself); 1: 64-row blocks on the item's side, 128-row
// blocks listed (the item's two lists merged, TileList); 2: 64-row blocks
// listed, 128-row item blocks (consecutive entries paired, PairList); 3:
// 64-row blocks on both sides, per item whichever of the merged tiles and the
// two lists in lockstep takes fewer steps (pairing_is_shorter, decided in
// init() from the lists' first and last entries, the same in every role).
// next() gives the tile's listed blocks (paired: the 64-row blocks of the low
// and high halves, -1 if missing; merged or plain: lo = the 128-row tile) and
// the visibility bits.
template <int kMode>
struct BlockSteps {
  TileList<kMode == 1 || kMode == 3> tl;
  PairList pl;
  bool pair;
  // item = 128-row block t of head h on the item's side; ptr/idx the fine
  // lists with nfine rows per head; rows_per_tile = 2 for 64-row blocks on the
  // item's side; list_shift = 1 for 64-row listed blocks
  UT_DEV void init(const int32_t* ptr, const int32_t* idx, int h, int t, int nfine, int rows_per_tile,
                   int list_shift) {
    if (kMode != 2) tl.init(ptr, idx, h, t, nfine, rows_per_tile, list_shift);
    if (kMode == 2) pl.init(ptr, idx, h, t, nfine, rows_per_tile == 2);
    pair = kMode == 2;
    if constexpr (kMode == 3) pair = pairing_is_shorter(tl);
  }
  UT_DEV int count_warp() const {
    if (kMode == 3 && pair) return tl.na > tl.nb ? tl.na : tl.nb;
    return kMode == 2 ? pl.count() : tl.count_warp();
  }
  UT_DEV bool empty() const { return kMode == 2 ? pl.empty() : tl.empty(); }
  UT_DEV bool next(int& lo, int& hi, uint32_t& bits) {
    if (kMode == 2) return pl.next(lo, hi, bits);
    if (kMode == 3 && pair) return PairList::step_two(tl.a, tl.b, tl.na, tl.nb, tl.pa, lo, hi, bits);
    hi = -1;
    return tl.next(lo, bits);
  }
};

// ---------------------------------------------------------------- tcgen05
UT_DEV void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
UT_DEV void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
UT_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
UT_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
UT_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem desc] * B[smem desc]; kind::f16 (bf16 in, fp32 accumulate).
UT_DEV void mma_bf16_ss(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem desc]; A is M x K in TMEM (lane = row, two bf16
// per 32-bit column, K-step of 16 = 8 columns), B as above.
UT_DEV void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Warp-collective forms: the whole (converged) warp executes them and the
// instruction is issued by one elected lane (always the same lane while the
// warp is fully active, so commits track that lane's MMAs).
UT_DEV void mma_bf16_ss_w(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred e, p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
UT_DEV void mma_bf16_ts_w(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred e, p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
UT_DEV void mma_commit_w(uint64_t* bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(
          smem_u32(bar))
      : "memory");
}

// Arrive on `bar` once every tcgen05.mma issued so far by this thread completed.
UT_DEV void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// Instruction descriptor, kind::f16: D fp32, A/B bf16, dense.
//   bits 4-5 D format (1 = f32), 7-9 A format (1 = bf16), 10-12 B format (1 = bf16),
//   15 A major (0 = K), 16 B major (0 = K, 1 = MN), 17-22 N>>3, 24-28 M>>4.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N, bool a_mn_major, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn_major ? 1u : 0u) << 15) | ((b_mn_major ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Shared-memory matrix descriptor, 128-byte swizzle (layout type 2), version 1.
//   bits 0-13 start>>4, 16-29 LBO>>4, 32-45 SBO>>4, 46-47 version=1, 61-63 layout.
UT_DEV uint64_t sdesc_sw128(uint32_t smem_addr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// 32 lanes x 32 bit, 32 consecutive columns per thread.
UT_DEV void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]),
        "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
        "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
UT_DEV void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
UT_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
UT_DEV void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// ------------------------------------------------------------------ misc
UT_DEV uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

UT_DEV float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

UT_DEV void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}

UT_DEV uint4 ld_nc_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}
UT_DEV void st_v4(void* p, uint4 v) {
  asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

}  // namespace ut
