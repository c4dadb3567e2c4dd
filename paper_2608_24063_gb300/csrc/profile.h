// Per-kernel CUDA-event timing used by viscache_profile_enable / _read.
#pragma once

#include <cuda_runtime.h>

namespace vc {

// Records an event pair around the launches made during its lifetime when
// profiling is enabled; does nothing otherwise.
class ProfileScope {
 public:
  ProfileScope(const char* name, cudaStream_t st);
  ~ProfileScope();
  ProfileScope(const ProfileScope&) = delete;
  ProfileScope& operator=(const ProfileScope&) = delete;

 private:
  const char* name_;
  cudaStream_t st_;
  cudaEvent_t start_ = nullptr;
};

}  // namespace vc
