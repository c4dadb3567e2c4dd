// Ranking and keep/drop sets, Algorithm 1 steps 1 and 3.
//
// A sort problem is (request, KV head) in the shared mode, (request, layer, KV
// head) in the layer-specific mode.  Scores become 32-bit keys whose ascending
// order is descending score; rank[v] = position of token v in the order
// "descending score, lower index first on exact ties".
//
// chunk_sort_kernel + chunk_rank_kernel: sorted 1024-key chunks, then each
// element's rank by counting (binary search) in every other chunk of its
// problem; many CTAs per problem, ranks exact and schedule-independent.
//
// compact_kernel: one CTA per (request, layer <= h, KV head) with B_l > 0.  A
// block-wide scan over tokens in ascending position (segments of 8192
// consecutive tokens, 8 per thread) emits keep = {rank < B_l} and drop =
// {B_l <= rank < Nq}, so both lists come out ascending and the result does
// not depend on thread scheduling.
#include <algorithm>
#include <climits>

#include "vc_common.cuh"
#include "kernels.h"
#include "profile.h"

namespace vc {
namespace {

__device__ __forceinline__ uint32_t desc_key(float s) {
  // monotone map float -> uint32 (ascending), then invert for descending order
  uint32_t u = __float_as_uint(s);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~u;
}

// chunk_sort_kernel: CTA (chunk c, problem p) forms the composite keys
// (desc_key(score) << 32 | token) of tokens c*1024 ... c*1024+1023 (missing
// tokens: all ones) and sorts them ascending with a bitonic network in shared
// memory; composite keys are unique, so "ascending composite" is exactly
// "descending score, lower index first on exact ties".
// chunk_rank_kernel: CTA (c, p) holds its sorted chunk, one element per thread,
// and streams every other chunk of the problem through shared memory; a
// binary search counts that chunk's elements below the thread's element.  The
// element's rank is its position in its own chunk plus those counts: the
// number of elements of the whole problem below it.

// Ranking problem p: its request, score offset and chunk base; false when
// the problem's layer is not scored (per-layer ranking of an evicted layer in
// the fused pass), so the CTA has nothing to do.
__device__ __forceinline__ bool problem_of(const Shape& sh, const Tables& tb, int p, Req& rq,
                                           int64_t& off, int64_t& chunk_base, int& nchunks) {
  const bool per_layer = sh.rank_mode == VC_RANK_PER_LAYER;
  const int per_req = per_layer ? sh.L * sh.Hkv : sh.Hkv;
  const int r = p / per_req, k = p % per_req;
  rq = tb.req[r];
  nchunks = (rq.n + kSortChunk - 1) / kSortChunk;
  off = rq.s_off + (int64_t)k * rq.n;
  chunk_base = ((int64_t)rq.chunk0 + (int64_t)k * nchunks) * kSortChunk;
  return !per_layer || k / sh.Hkv < rq.Ls;
}

// Compare-exchange of the bitonic network between lanes t and t ^ j of a
// warp (j < 32): the lower lane keeps min/max as the direction bit says.
__device__ __forceinline__ uint64_t bitonic_lane(uint64_t a, int t, int j, int k) {
  const uint64_t b = __shfl_xor_sync(0xffffffffu, a, j);
  const bool up = (t & k) == 0;
  const bool lower = (t & j) == 0;
  return (lower == up) ? (a < b ? a : b) : (a < b ? b : a);
}

__global__ void __launch_bounds__(kSortChunk) chunk_sort_kernel(Shape sh, Tables tb,
                                                                const float* __restrict__ scores,
                                                                uint64_t* __restrict__ chunks) {
  __shared__ uint64_t e[kSortChunk];
  dep_wait();                                      // the scores
  if (threadIdx.x == 0) dep_launch();
  Req rq;
  int64_t off, base;
  int nchunks;
  const bool scored = problem_of(sh, tb, blockIdx.y, rq, off, base, nchunks);
  const int c = blockIdx.x;
  if (c >= nchunks || !scored) return;
  const int t = threadIdx.x;
  const int v = c * kSortChunk + t;
  uint64_t a = v < rq.n ? ((uint64_t)desc_key(scores[off + v]) << 32) | (uint32_t)v : ~0ull;
  // strides below 32 stay in the warp (shuffles), larger ones go through
  // shared memory with a block barrier
  for (int k = 2; k <= kSortChunk; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      if (j >= 32) {
        e[t] = a;
        __syncthreads();
        const uint64_t b = e[t ^ j];
        const bool up = (t & k) == 0;
        const bool lower = (t & j) == 0;
        a = (lower == up) ? (a < b ? a : b) : (a < b ? b : a);
        __syncthreads();
      } else {
        a = bitonic_lane(a, t, j, k);
      }
    }
  }
  chunks[base + (int64_t)c * kSortChunk + t] = a;
}

// Other chunks are staged kRankGroup at a time (8 KB each) so a group costs
// one barrier pair; each thread then runs its binary searches back to back.
constexpr int kRankGroup = 12;

__global__ void __launch_bounds__(kSortChunk) chunk_rank_kernel(Shape sh, Tables tb,
                                                                const uint64_t* __restrict__ chunks,
                                                                int32_t* __restrict__ rank) {
  extern __shared__ uint64_t other[];               // [kRankGroup][kSortChunk]
  dep_wait();                                      // the sorted chunks
  if (threadIdx.x == 0) dep_launch();
  Req rq;
  int64_t off, base;
  int nchunks;
  const bool scored = problem_of(sh, tb, blockIdx.y, rq, off, base, nchunks);
  const int c = blockIdx.x;
  if (c >= nchunks || !scored) return;
  const int t = threadIdx.x;
  const uint64_t mine = chunks[base + (int64_t)c * kSortChunk + t];
  int count = t;                                   // elements of its own chunk below it
  for (int g0 = 0; g0 < nchunks; g0 += kRankGroup) {
    const int gn = min(kRankGroup, nchunks - g0);
    __syncthreads();
    for (int i = 0; i < gn; ++i)
      other[i * kSortChunk + t] = chunks[base + (int64_t)(g0 + i) * kSortChunk + t];
    __syncthreads();
    for (int i = 0; i < gn; ++i) {
      if (g0 + i == c) continue;
      const uint64_t* o = other + i * kSortChunk;
      int pos = 0;                                 // elements of chunk g0 + i below `mine`
#pragma unroll
      for (int s = kSortChunk; s > 0; s >>= 1)
        if (pos + s <= kSortChunk && o[pos + s - 1] < mine) pos += s;
      count += pos;
    }
  }
  if (mine != ~0ull) {
    const uint32_t v = (uint32_t)mine;
    if (v < (uint32_t)rq.n && count < rq.n) rank[off + v] = count;
    else set_status(tb.status, VC_ERR_DEVICE_INDEX);
  }
}

// One CTA per (request, layer, KV head); layers with B_l == 0 exit at once.
constexpr int kScanThreads = 1024;
constexpr int kScanPer = 8;                  // tokens per thread per segment

__global__ void __launch_bounds__(kScanThreads) compact_kernel(Shape sh, Tables tb,
                                                               const int32_t* __restrict__ rank,
                                                               int32_t* __restrict__ keep_idx,
                                                               int32_t* __restrict__ drop_idx) {
  constexpr int kWarps = kScanThreads / 32;
  __shared__ int32_t wk[kWarps], wd[kWarps], tot[2];
  dep_wait();                                // the ranks (at once when launched ordinarily)
  if (threadIdx.x == 0) dep_launch();        // the gather may be scheduled
  const int g = blockIdx.y;
  const int rl = blockIdx.x;                 // request * L + layer
  const int r = rl / sh.L, l = rl % sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  if (ly.B <= 0) return;
  const int n = rq.n;
  const int32_t* rk = rank + rq.s_off + (sh.rank_mode == VC_RANK_PER_LAYER
                                             ? ((int64_t)l * sh.Hkv + g) * n
                                             : (int64_t)g * n);
  int32_t* ko = keep_idx + rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B;
  int32_t* dro = drop_idx + rq.drop_row0 + (int64_t)sh.Hkv * ly.Qd + (int64_t)g * ly.D;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // segments of kScanThreads * kScanPer consecutive tokens: thread t looks at
  // tokens s + t*kScanPer ..., the block counts the keep/drop tokens before
  // them (warp scans, warp totals through shared memory) and the thread
  // writes its own at the running offsets, so both lists come out in
  // ascending position
  int base_k = 0, base_d = 0;
  for (int s0 = 0; s0 < n; s0 += kScanThreads * kScanPer) {
    const int v0 = s0 + (int)threadIdx.x * kScanPer;
    int xs[kScanPer];
#pragma unroll
    for (int k = 0; k < kScanPer; ++k) xs[k] = v0 + k < n ? rk[v0 + k] : INT_MAX;
    int ck = 0, cd = 0;
#pragma unroll
    for (int k = 0; k < kScanPer; ++k) {
      ck += xs[k] < ly.B;
      cd += (xs[k] >= ly.B) & (xs[k] < rq.Nq);
    }
    int ik = ck, id = cd;                    // inclusive warp scan
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int a = __shfl_up_sync(0xffffffffu, ik, off);
      const int b = __shfl_up_sync(0xffffffffu, id, off);
      if (lane >= off) { ik += a; id += b; }
    }
    if (lane == 31) { wk[warp] = ik; wd[warp] = id; }
    __syncthreads();
    if (warp == 0) {                         // exclusive scan of the warp totals, and the block total
      const int a = lane < kWarps ? wk[lane] : 0, b = lane < kWarps ? wd[lane] : 0;
      int ia = a, ib = b;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, ia, off);
        const int y = __shfl_up_sync(0xffffffffu, ib, off);
        if (lane >= off) { ia += x; ib += y; }
      }
      if (lane < kWarps) { wk[lane] = ia - a; wd[lane] = ib - b; }
      if (lane == 31) { tot[0] = ia; tot[1] = ib; }
    }
    __syncthreads();
    int pk = base_k + wk[warp] + ik - ck, pd = base_d + wd[warp] + id - cd;
#pragma unroll
    for (int k = 0; k < kScanPer; ++k) {
      const int x = xs[k], v = v0 + k;
      if (x < ly.B) {
        if (pk < ly.B) ko[pk] = v; else set_status(tb.status, VC_ERR_DEVICE_INDEX);
        ++pk;
      } else if (x < rq.Nq) {
        if (pd < ly.D) dro[pd] = v; else set_status(tb.status, VC_ERR_DEVICE_INDEX);
        ++pd;
      }
    }
    base_k += tot[0];
    base_d += tot[1];
    __syncthreads();                         // shared totals are rewritten next segment
  }
}

}  // namespace

cudaError_t launch_select(const Shape& sh, const Tables& tb, int n_problems, int max_chunks,
                          const float* scores, int32_t* rank, uint64_t* chunks, int32_t* keep_idx,
                          int32_t* drop_idx, cudaStream_t st) {
  const dim3 grid((unsigned)max_chunks, (unsigned)n_problems);
  {
    ProfileScope ps("chunk_sort", st);
    cudaError_t el = launch_dep(chunk_sort_kernel, grid, dim3(kSortChunk), 0, st, sh, tb, scores, chunks);
    if (el != cudaSuccess) return el;
  }
  cudaError_t e0 = cudaGetLastError();
  if (e0 != cudaSuccess) return e0;
  {
    const size_t smem = sizeof(uint64_t) * kSortChunk * (size_t)std::min(kRankGroup, std::max(max_chunks, 1));
    cudaError_t ea = cudaFuncSetAttribute(chunk_rank_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (ea != cudaSuccess) return ea;
    ProfileScope ps("chunk_rank", st);
    cudaError_t el = launch_dep(chunk_rank_kernel, grid, dim3(kSortChunk), smem, st, sh, tb,
                                static_cast<const uint64_t*>(chunks), rank);
    if (el != cudaSuccess) return el;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  {
    ProfileScope ps("compact_keep_drop", st);
    // an ordinary launch: it starts once the ranks are complete.  Measured on
    // the ragged 8-request batch, the chain of dependent launches from the
    // column sums through the gather cost ~60 us per call when every link
    // of it was dependent, and nothing when any one of them was not; here
    // the break costs nothing on the single-request workloads.
    compact_kernel<<<dim3(sh.n_req * sh.L, sh.Hkv), kScanThreads, 0, st>>>(sh, tb, rank, keep_idx,
                                                                           drop_idx);
  }
  return cudaGetLastError();
}

}  // namespace vc
