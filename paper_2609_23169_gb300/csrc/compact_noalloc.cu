// ut_fg_compact_noalloc: Background Token Dropping for callers that cannot
// allocate device memory.
//
// ut_fg_compact needs a small caller-provided workspace (one int32 count per
// 4096 canvas tokens).  Some callers have no way to provide one: a plugin or
// inference host that owns every device allocation and hands the library only
// its input and output buffers, a real-time loop that must never enter the
// allocator, or code that sits behind a C interface with no allocator handle.
// This variant keeps that workspace in a fixed device array inside the
// library instead, so the call needs nothing beyond its inputs and outputs.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it (4 KiB) until the process exits.  In host code its name
// is only a host-side stand-in, so its device address is looked up with
// cudaGetSymbolAddress once per CUDA context, on the first call made while
// that context is current, and cached under the context's unique id: a
// context created later (after cudaDeviceReset, or a separate driver-API
// context) never reuses an address looked up for another one.  That first
// call may also make the CUDA runtime load the library's device code into the
// context (lazy loading), and loading code allocates device memory inside the
// driver; this file itself calls no allocating routine.  Make the first call
// in each context before any stream capture.  All calls in one context share
// the one array, so calls that overlap on the GPU (different streams, or
// different host threads without ordering) race on it; serialise them.  The
// counts are fully rewritten by every call (nothing in the array has to start
// at zero).
#include <mutex>

#include "../../include/ultratex.h"
#include "common.cuh"
#include "kernels.h"

namespace ut {

// Largest canvas this variant accepts: one count per 4096 tokens, 1024 counts.
constexpr int64_t kNoAllocMaxTokens = 4096ll * 1024ll;
constexpr int kNoAllocCounts = 1024;

static __device__ __align__(256) int32_t g_compact_scratch[kNoAllocCounts];

namespace {
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Driver entry points, resolved once through the runtime (the library links
// the static runtime only).
template <typename F>
F driver_fn(const char* name) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPoint(name, &p, cudaEnableDefault, &q) != cudaSuccess || q != cudaDriverEntryPointSuccess)
    return nullptr;
  return reinterpret_cast<F>(p);
}

constexpr int kMaxContexts = 64;
struct ScratchEntry {
  unsigned long long ctx_id;  // 0 = unused (driver context ids start at 1)
  void* addr;
};
std::mutex g_setup_mutex;
ScratchEntry g_scratch[kMaxContexts] = {};

// Id of the current context; 0 if none is current or the query fails.
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
  static CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
  if (!get_current || !get_id) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of g_compact_scratch in the current context.
cudaError_t scratch_address(void** out) {
  unsigned long long id = current_context_id();
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (id != 0) {
    for (const ScratchEntry& e : g_scratch)
      if (e.ctx_id == id) {
        *out = e.addr;
        return cudaSuccess;
      }
  }
  // first call in this context (the lookup also makes the runtime bind its
  // context when none was current yet, so the id is taken again afterwards)
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_compact_scratch);
  if (e != cudaSuccess) return e;
  if (id == 0) id = current_context_id();
  if (id != 0) {
    for (ScratchEntry& s : g_scratch)
      if (s.ctx_id == 0) {
        s.ctx_id = id;
        s.addr = p;
        break;
      }  // a full table only means later calls in this context look up again
  }
  *out = p;
  return cudaSuccess;
}
}  // namespace

}  // namespace ut

extern "C" ut_status ut_fg_compact_noalloc(const uint8_t* mask, int64_t T, int32_t n_tensors,
                                           const void* const* h_src, void* const* h_dst, int64_t row_bytes,
                                           int64_t capacity, int32_t* idx_out, int32_t* n_out, int32_t* dev_status,
                                           void* stream) {
  using namespace ut;
  if (T > kNoAllocMaxTokens) return UT_ERR_UNSUPPORTED;  // beyond the fixed scratch array
  if (T < 0 || capacity < 0 || n_tensors < 1 || n_tensors > 8 || !n_out) return UT_ERR_INVALID_ARG;
  if (row_bytes <= 0 || row_bytes % 16 != 0) return UT_ERR_INVALID_ARG;
  if (!h_src || !h_dst) return UT_ERR_INVALID_ARG;
  if (T > 0) {
    if (!mask) return UT_ERR_INVALID_ARG;
    if (capacity > 0 && !idx_out) return UT_ERR_INVALID_ARG;
    for (int i = 0; i < n_tensors; ++i) {
      if (!h_src[i] || (reinterpret_cast<uintptr_t>(h_src[i]) & 15u)) return UT_ERR_INVALID_ARG;
      if (capacity > 0 && (!h_dst[i] || (reinterpret_cast<uintptr_t>(h_dst[i]) & 15u))) return UT_ERR_INVALID_ARG;
    }
  }
  void* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return UT_ERR_CUDA;
  int dev = 0, sms = 1;
  if (cudaGetDevice(&dev) != cudaSuccess) return UT_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return UT_ERR_CUDA;
  cudaError_t e = launch_fg_compact(mask, T, n_tensors, h_src, h_dst, row_bytes, capacity, idx_out, n_out, scratch,
                                    dev_status, sms, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? UT_OK : UT_ERR_CUDA;
}
