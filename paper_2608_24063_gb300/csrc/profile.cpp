// Optional per-kernel timing: when enabled, every kernel launch of the library
// is bracketed by a pair of CUDA events on its stream; viscache_profile_read
// sums the elapsed times per kernel name.  Off by default (no events, no cost).
// Not thread-safe: meant for one benchmarking thread.
#include <cuda_runtime.h>
#include <string.h>

#include <mutex>
#include <string>
#include <vector>

#include "profile.h"
#include "viscache.h"

namespace vc {
namespace {

struct Slot {
  const char* name;
  cudaEvent_t start, stop;
};

struct Profiler {
  bool on = false;
  std::vector<Slot> slots;      // recorded this window
  std::vector<cudaEvent_t> pool;
  size_t used = 0;
  std::mutex mu;

  cudaEvent_t take() {
    if (used == pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[used++];
  }
};

Profiler& prof() {
  static Profiler p;
  return p;
}

}  // namespace

ProfileScope::ProfileScope(const char* name, cudaStream_t st) : name_(name), st_(st) {
  Profiler& p = prof();
  if (!p.on) return;
  std::lock_guard<std::mutex> g(p.mu);
  start_ = p.take();
  if (start_) cudaEventRecord(start_, st_);
}

ProfileScope::~ProfileScope() {
  Profiler& p = prof();
  if (!p.on || !start_) return;
  std::lock_guard<std::mutex> g(p.mu);
  cudaEvent_t stop = p.take();
  if (!stop) return;
  cudaEventRecord(stop, st_);
  p.slots.push_back(Slot{name_, start_, stop});
}

}  // namespace vc

extern "C" int viscache_profile_enable(int on) {
  vc::Profiler& p = vc::prof();
  std::lock_guard<std::mutex> g(p.mu);
  p.on = on != 0;
  p.slots.clear();
  p.used = 0;
  return VC_OK;
}

extern "C" int viscache_profile_read(char* names, int name_bytes, float* total_ms, int* launches,
                                     int max_kernels) {
  vc::Profiler& p = vc::prof();
  std::lock_guard<std::mutex> g(p.mu);
  std::vector<std::string> keys;
  std::vector<float> ms;
  std::vector<int> cnt;
  for (const vc::Slot& s : p.slots) {
    if (cudaEventSynchronize(s.stop) != cudaSuccess) return -VC_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, s.start, s.stop) != cudaSuccess) return -VC_ERR_CUDA;
    size_t k = 0;
    while (k < keys.size() && keys[k] != s.name) ++k;
    if (k == keys.size()) { keys.push_back(s.name); ms.push_back(0.f); cnt.push_back(0); }
    ms[k] += t;
    cnt[k] += 1;
  }
  const int nk = (int)keys.size() < max_kernels ? (int)keys.size() : max_kernels;
  std::string joined;
  for (int k = 0; k < nk; ++k) {
    if (total_ms) total_ms[k] = ms[k];
    if (launches) launches[k] = cnt[k];
    joined += keys[k];
    joined += '\n';
  }
  if (names && name_bytes > 0) {
    strncpy(names, joined.c_str(), name_bytes - 1);
    names[name_bytes - 1] = '\0';
  }
  p.slots.clear();
  p.used = 0;
  return nk;
}
