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
// looked up once per device with cudaGetSymbolAddress (on the first call made
// on that device, with that device current) and cached.
//
// All calls on a device share the array and it keeps the last call's
// contents.  Nothing in it needs to start at zero: each call rewrites the
// status word and the tables before its kernels read them, and the first
// pass overwrites every log-sum-exp value the second pass reads.  Calls whose
// kernels overlap on the GPU (different streams, or different host threads)
// race on the array and must be serialised by the caller.
#include <cuda_runtime.h>

#include <mutex>

#include "viscache.h"

namespace {

constexpr size_t kStaticScratchBytes = VC_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_score_scratch[kStaticScratchBytes];

std::mutex g_mu;
void* g_addr[kMaxDevices] = {};

// Device address of g_score_scratch on the current device (nullptr on failure).
void* scratch_address() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_score_scratch) != cudaSuccess) return nullptr;
    g_addr[dev] = p;
  }
  return g_addr[dev];
}

}  // namespace

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
