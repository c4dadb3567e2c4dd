// prunekv_score_static: token scoring (the same kernels as prunekv_score) for
// callers that cannot allocate device memory: code running inside a memory
// pool or allocator hook (a cudaMalloc there would re-enter the allocator),
// a host that replays frozen CUDA graphs (a fresh allocation is not part of
// the captured memory), or an embedding runtime that hands out no workspace.
// Its scratch (status word, plan tables and the per-row log-sum-exp of the
// first pass) lives in one fixed device array owned by this library instead
// of a caller workspace.
//
// The array is a file-scope __device__ variable of kStaticScratchBytes; every
// GPU that loads the library holds it until the process exits.  Host code
// cannot use the symbol's name as a device address, so the device address is
// looked up with cudaGetSymbolAddress on the first call made in a CUDA
// context (with that context's device current) and cached together with the
// context's id.  A later call in another context -- after cudaDeviceReset, or
// after the primary context was released and created again, when the module
// is loaded anew and the array may sit elsewhere -- sees a different id and
// looks the address up again.
//
// All calls on a device share the array and it keeps the last call's
// contents.  Nothing in it needs to start at zero: each call rewrites the
// status word and the tables before its kernels read them, and the first
// pass overwrites every log-sum-exp value the second pass reads.  Calls whose
// kernels overlap on the GPU (different streams, or different host threads)
// race on the array and must be serialised by the caller.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <mutex>

#include "viscache.h"

namespace {

constexpr size_t kStaticScratchBytes = VC_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_score_scratch[kStaticScratchBytes];

struct Slot {
  unsigned long long ctx_id;   // id of the context the address belongs to
  void* addr;                  // nullptr: not looked up yet
};

std::mutex g_mu;
Slot g_slot[kMaxDevices] = {};

// Id of the calling thread's current CUDA context; false if there is none or
// the driver does not offer the query.
bool current_context_id(unsigned long long* id) {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  if (!get_current || !get_id) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// Device address of g_score_scratch in the current context (nullptr on failure).
void* scratch_address() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  unsigned long long id = 0;
  const bool have_id = current_context_id(&id);
  std::lock_guard<std::mutex> lock(g_mu);
  Slot& s = g_slot[dev];
  if (have_id && s.addr && s.ctx_id == id) return s.addr;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_score_scratch) != cudaSuccess) return nullptr;
  // the lookup makes the primary context current if none was; cache only
  // when the context can be identified, else look the address up every call
  unsigned long long id2 = 0;
  if (current_context_id(&id2)) {
    s.ctx_id = id2;
    s.addr = p;
  } else {
    s.addr = nullptr;
  }
  return p;
}

}  // namespace

extern "C" size_t prunekv_score_static_capacity(void) { return kStaticScratchBytes; }

extern "C" int prunekv_score_static(const void* Qw, const void* K, int dtype, int32_t L,
                                    int32_t Hq, int32_t Hkv, int32_t d, int32_t n_vis, int32_t W,
                                    float scale, int rank_mode, const float* row_lse,
                                    float* scores, void* stream) {
  if (L < 1 || L > 256 || Hq < 1 || W < 1) return VC_ERR_INVALID_ARG;
  // reject problems whose scratch does not fit before touching the device
  const size_t need = prunekv_score_workspace_size(L, Hq, W);
  if (need == 0) return VC_ERR_INVALID_ARG;
  if (need > kStaticScratchBytes) return VC_ERR_WORKSPACE;
  void* ws = scratch_address();
  if (!ws) return VC_ERR_CUDA;
  return prunekv_score(Qw, K, dtype, L, Hq, Hkv, d, n_vis, W, scale, rank_mode, row_lse, scores,
                       ws, kStaticScratchBytes, stream);
}

// The status word is the first 4 bytes of the scratch (the workspace layout
// puts it at offset 0); it is read straight from the symbol, no address needed.
extern "C" int prunekv_score_static_status(void* stream) {
  int32_t s = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyFromSymbolAsync(&s, g_score_scratch, sizeof(s), 0, cudaMemcpyDeviceToHost, st) !=
      cudaSuccess)
    return VC_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return VC_ERR_CUDA;
  return s;
}
