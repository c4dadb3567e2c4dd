// Copies a plan-table image (a kernel parameter) into the caller workspace and
// clears the status word.
#include "kernels.h"
#include "profile.h"

namespace vc {
namespace {

__global__ void upload_kernel(const __grid_constant__ TableImage im, uint32_t bytes, uint8_t* dst,
                              int32_t* status) {
  // launched fully serialised after everything before it on the stream; the
  // kernels after it wait for it before they read the tables
  dep_launch();
  const uint4* src = reinterpret_cast<const uint4*>(im.bytes);
  uint4* d = reinterpret_cast<uint4*>(dst);
  for (uint32_t i = threadIdx.x; i < bytes / 16; i += blockDim.x) d[i] = src[i];
  for (uint32_t i = (bytes / 16) * 16 + threadIdx.x; i < bytes; i += blockDim.x) dst[i] = im.bytes[i];
  if (threadIdx.x == 0) *status = VC_OK;
}

}  // namespace

cudaError_t launch_upload(const TableImage& im, uint32_t bytes, uint8_t* dst, int32_t* status,
                          cudaStream_t st) {
  ProfileScope ps("upload_tables", st);
  upload_kernel<<<1, 256, 0, st>>>(im, bytes, dst, status);
  return cudaGetLastError();
}

}  // namespace vc
