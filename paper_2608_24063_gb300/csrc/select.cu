// Ranking and keep/drop sets, Algorithm 1 steps 1 and 3.
//
// rank_sort_kernel: one CTA per sort problem ((request, KV head) in the shared
// mode, (request, layer, KV head) in the layer-specific mode).  Scores become
// 32-bit keys whose ascending order is descending score; a stable LSD radix
// sort (four 8-bit digits) over (key, token) pairs that start in ascending
// token order then yields the order "descending score, lower index first on
// exact ties".  rank[v] = position of token v.  The ping-pong buffers live in
// the workspace (L2-resident at these sizes).
//
// compact_kernel: one CTA per (request, layer <= h, KV head) with B_l > 0.  A
// block-wide scan over tokens in ascending position emits keep = {rank < B_l}
// and drop = {B_l <= rank < Nq}, so both lists come out ascending and the
// result does not depend on thread scheduling.
#include "vc_common.cuh"
#include "kernels.h"
#include "profile.h"

namespace vc {
namespace {

constexpr int kSortThreads = 1024;
constexpr int kSortWarps = kSortThreads / 32;

// Lanes of the warp holding the same 8-bit digit (and the same validity),
// built from nine ballots.
__device__ __forceinline__ uint32_t digit_peers(uint32_t dig, bool ok) {
  const uint32_t okm = __ballot_sync(0xffffffffu, ok);
  uint32_t peers = ok ? okm : ~okm;
#pragma unroll
  for (int b = 0; b < 8; ++b) {
    const uint32_t bit = (dig >> b) & 1u;
    const uint32_t m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return peers;
}

__device__ __forceinline__ uint32_t desc_key(float s) {
  // monotone map float -> uint32 (ascending), then invert for descending order
  uint32_t u = __float_as_uint(s);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~u;
}

struct SortProblem {
  const float* s;      // scores of this problem [n]
  int32_t* rank;       // rank output [n]
  uint32_t* k0; uint32_t* k1;   // key ping-pong [n]
  int32_t* v0; int32_t* v1;     // token ping-pong [n]
  int n;
};

__device__ __forceinline__ SortProblem sort_problem(const Shape& sh, const Tables& tb,
                                                    const float* scores, int32_t* rank,
                                                    uint32_t* keys, int32_t* vals,
                                                    int64_t sort_stride_elems) {
  SortProblem p;
  const int per_req = sh.rank_mode == VC_RANK_PER_LAYER ? sh.L * sh.Hkv : sh.Hkv;
  const int r = blockIdx.x / per_req, k = blockIdx.x % per_req;
  const Req rq = tb.req[r];
  const int64_t off = rq.s_off + (int64_t)k * rq.n;
  p.s = scores + off;
  p.rank = rank + off;
  p.k0 = keys + off;
  p.k1 = keys + sort_stride_elems + off;
  p.v0 = vals + off;
  p.v1 = vals + sort_stride_elems + off;
  p.n = rq.n;
  return p;
}

__global__ void __launch_bounds__(kSortThreads) rank_sort_kernel(Shape sh, Tables tb,
                                                                 const float* __restrict__ scores,
                                                                 int32_t* __restrict__ rank,
                                                                 uint32_t* keys, int32_t* vals,
                                                                 int64_t sort_stride_elems) {
  __shared__ uint32_t hist[kSortWarps][256];
  __shared__ uint32_t digit_base[256];
  SortProblem p = sort_problem(sh, tb, scores, rank, keys, vals, sort_stride_elems);
  const int n = p.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t lt_mask = (1u << lane) - 1u;
  // contiguous segment per warp, a multiple of 32 long
  const int seg = ((n + kSortWarps * 32 - 1) / (kSortWarps * 32)) * 32;
  const int s0 = warp * seg;

  for (int e = threadIdx.x; e < n; e += kSortThreads) {
    p.k0[e] = desc_key(p.s[e]);
    p.v0[e] = e;
  }
  uint32_t* kin = p.k0; uint32_t* kout = p.k1;
  int32_t* vin = p.v0; int32_t* vout = p.v1;
  __syncthreads();

  for (int shift = 0; shift < 32; shift += 8) {
    for (int d = lane; d < 256; d += 32) hist[warp][d] = 0;
    __syncwarp();
    // phase 1: per-warp digit histogram
    for (int c = 0; c < seg; c += 32) {
      const int e = s0 + c + lane;
      const bool ok = e < n;
      const uint32_t dig = ok ? (kin[e] >> shift) & 0xffu : 0x100u + lane;
      const uint32_t peers = digit_peers(dig, ok);
      if (ok && (peers & lt_mask) == 0) hist[warp][dig] += __popc(peers);
      __syncwarp();
    }
    __syncthreads();
    // phase 2: exclusive offsets, digit-major then warp order
    if (threadIdx.x < 256) {
      const int d = threadIdx.x;
      uint32_t run = 0;
      for (int w = 0; w < kSortWarps; ++w) {
        const uint32_t c = hist[w][d];
        hist[w][d] = run;
        run += c;
      }
      digit_base[d] = run;   // total count of digit d for now
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // exclusive scan of 256 digit totals by one warp (8 per lane)
      uint32_t v[8], sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) { v[i] = digit_base[lane * 8 + i]; sum += v[i]; }
      uint32_t incl = sum;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t o = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += o;
      }
      uint32_t run = incl - sum;
#pragma unroll
      for (int i = 0; i < 8; ++i) { digit_base[lane * 8 + i] = run; run += v[i]; }
    }
    __syncthreads();
    // phase 3: stable scatter
    for (int c = 0; c < seg; c += 32) {
      const int e = s0 + c + lane;
      const bool ok = e < n;
      const uint32_t key = ok ? kin[e] : 0u;
      const uint32_t dig = ok ? (key >> shift) & 0xffu : 0x100u + lane;
      const uint32_t peers = digit_peers(dig, ok);
      uint32_t pos = 0;
      if (ok) pos = digit_base[dig] + hist[warp][dig] + __popc(peers & lt_mask);
      __syncwarp();
      if (ok && (peers & lt_mask) == 0) hist[warp][dig] += __popc(peers);
      if (ok) {
        if (pos < (uint32_t)n) { kout[pos] = key; vout[pos] = vin[e]; }
        else set_status(tb.status, VC_ERR_DEVICE_INDEX);
      }
      __syncwarp();
    }
    __syncthreads();
    uint32_t* tk = kin; kin = kout; kout = tk;
    int32_t* tv = vin; vin = vout; vout = tv;
  }
  // after four passes the sorted order is back in (k0, v0)
  for (int e = threadIdx.x; e < n; e += kSortThreads) {
    const int v = vin[e];
    if (v >= 0 && v < n) p.rank[v] = e;
  }
}

// Shared-memory variant for n <= kSmemSortMax: keys, token ids and the
// per-warp histograms stay on chip; only the scores are read and the ranks
// written.  Same stable LSD passes as rank_sort_kernel.
constexpr int kSmemSortMax = 16384;

__global__ void __launch_bounds__(kSortThreads) rank_sort_smem_kernel(Shape sh, Tables tb,
                                                                      const float* __restrict__ scores,
                                                                      int32_t* __restrict__ rank) {
  extern __shared__ uint4 smem_u4[];
  uint32_t* k0 = reinterpret_cast<uint32_t*>(smem_u4);
  uint32_t* k1 = k0 + kSmemSortMax;
  uint16_t* v0 = reinterpret_cast<uint16_t*>(k1 + kSmemSortMax);
  uint16_t* v1 = v0 + kSmemSortMax;
  uint16_t (*hist)[256] = reinterpret_cast<uint16_t (*)[256]>(v1 + kSmemSortMax);
  __shared__ uint32_t digit_base[256];
  const int per_req = sh.rank_mode == VC_RANK_PER_LAYER ? sh.L * sh.Hkv : sh.Hkv;
  const int r = blockIdx.x / per_req, kprob = blockIdx.x % per_req;
  const Req rq = tb.req[r];
  const int64_t off = rq.s_off + (int64_t)kprob * rq.n;
  const int n = rq.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t lt_mask = (1u << lane) - 1u;
  const int seg = ((n + kSortWarps * 32 - 1) / (kSortWarps * 32)) * 32;
  const int s0 = warp * seg;
  for (int e = threadIdx.x; e < n; e += kSortThreads) {
    k0[e] = desc_key(scores[off + e]);
    v0[e] = (uint16_t)e;
  }
  uint32_t* kin = k0; uint32_t* kout = k1;
  uint16_t* vin = v0; uint16_t* vout = v1;
  __syncthreads();
  for (int shift = 0; shift < 32; shift += 8) {
    for (int d = lane; d < 256; d += 32) hist[warp][d] = 0;
    __syncwarp();
    for (int c = 0; c < seg; c += 32) {
      const int e = s0 + c + lane;
      const bool ok = e < n;
      const uint32_t dig = ok ? (kin[e] >> shift) & 0xffu : 0x100u + lane;
      const uint32_t peers = digit_peers(dig, ok);
      if (ok && (peers & lt_mask) == 0) hist[warp][dig] += (uint16_t)__popc(peers);
      __syncwarp();
    }
    __syncthreads();
    if (threadIdx.x < 256) {
      const int d = threadIdx.x;
      uint32_t run = 0;
      for (int w = 0; w < kSortWarps; ++w) {
        const uint32_t cnt = hist[w][d];
        hist[w][d] = (uint16_t)run;
        run += cnt;
      }
      digit_base[d] = run;
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      uint32_t v[8], sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) { v[i] = digit_base[lane * 8 + i]; sum += v[i]; }
      uint32_t incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      uint32_t run = incl - sum;
#pragma unroll
      for (int i = 0; i < 8; ++i) { digit_base[lane * 8 + i] = run; run += v[i]; }
    }
    __syncthreads();
    for (int c = 0; c < seg; c += 32) {
      const int e = s0 + c + lane;
      const bool ok = e < n;
      const uint32_t key = ok ? kin[e] : 0u;
      const uint32_t dig = ok ? (key >> shift) & 0xffu : 0x100u + lane;
      const uint32_t peers = digit_peers(dig, ok);
      uint32_t pos = 0;
      if (ok) pos = digit_base[dig] + hist[warp][dig] + __popc(peers & lt_mask);
      __syncwarp();
      if (ok && (peers & lt_mask) == 0) hist[warp][dig] += (uint16_t)__popc(peers);
      if (ok) {
        if (pos < (uint32_t)n) { kout[pos] = key; vout[pos] = vin[e]; }
        else set_status(tb.status, VC_ERR_DEVICE_INDEX);
      }
      __syncwarp();
    }
    __syncthreads();
    uint32_t* tk = kin; kin = kout; kout = tk;
    uint16_t* tv = vin; vin = vout; vout = tv;
  }
  int32_t* rk = rank + off;
  for (int e = threadIdx.x; e < n; e += kSortThreads) rk[vin[e]] = e;
}

// One CTA per (request, layer, KV head); layers with B_l == 0 exit at once.
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads) compact_kernel(Shape sh, Tables tb,
                                                               const int32_t* __restrict__ rank,
                                                               int32_t* __restrict__ keep_idx,
                                                               int32_t* __restrict__ drop_idx) {
  __shared__ int32_t wk[32], wd[32];
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
  const int per = (n + kScanThreads - 1) / kScanThreads;
  const int t0 = threadIdx.x * per;
  const int t1 = min(n, t0 + per);
  int ck = 0, cd = 0;
  for (int v = t0; v < t1; ++v) {
    const int x = rk[v];
    ck += x < ly.B;
    cd += (x >= ly.B) & (x < rq.Nq);
  }
  // block exclusive scan of (ck, cd)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int ik = ck, id = cd;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int a = __shfl_up_sync(0xffffffffu, ik, off);
    const int b = __shfl_up_sync(0xffffffffu, id, off);
    if (lane >= off) { ik += a; id += b; }
  }
  if (lane == 31) { wk[warp] = ik; wd[warp] = id; }
  __syncthreads();
  if (warp == 0) {
    int a = wk[lane], b = wd[lane];
    int ia = a, ib = b;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int x = __shfl_up_sync(0xffffffffu, ia, off);
      const int y = __shfl_up_sync(0xffffffffu, ib, off);
      if (lane >= off) { ia += x; ib += y; }
    }
    wk[lane] = ia - a;
    wd[lane] = ib - b;
  }
  __syncthreads();
  int pk = wk[warp] + ik - ck, pd = wd[warp] + id - cd;
  for (int v = t0; v < t1; ++v) {
    const int x = rk[v];
    if (x < ly.B) {
      if (pk < ly.B) ko[pk] = v; else set_status(tb.status, VC_ERR_DEVICE_INDEX);
      ++pk;
    } else if (x < rq.Nq) {
      if (pd < ly.D) dro[pd] = v; else set_status(tb.status, VC_ERR_DEVICE_INDEX);
      ++pd;
    }
  }
}

}  // namespace

cudaError_t launch_select(const Shape& sh, const Tables& tb, int n_problems, int max_n,
                          const float* scores, int32_t* rank, uint32_t* keys, int32_t* vals,
                          int64_t sort_stride, int32_t* keep_idx, int32_t* drop_idx,
                          cudaStream_t st) {
  if (max_n <= kSmemSortMax) {
    const size_t smem = (size_t)kSmemSortMax * (2 * 4 + 2 * 2) + (size_t)kSortWarps * 256 * 2;
    cudaError_t e = cudaFuncSetAttribute(rank_sort_smem_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    ProfileScope ps("rank_sort", st);
    rank_sort_smem_kernel<<<n_problems, kSortThreads, smem, st>>>(sh, tb, scores, rank);
  } else {
    ProfileScope ps("rank_sort", st);
    rank_sort_kernel<<<n_problems, kSortThreads, 0, st>>>(sh, tb, scores, rank, keys, vals,
                                                          sort_stride);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  {
    ProfileScope ps("compact_keep_drop", st);
    compact_kernel<<<dim3(sh.n_req * sh.L, sh.Hkv), kScanThreads, 0, st>>>(sh, tb, rank, keep_idx,
                                                                           drop_idx);
  }
  return cudaGetLastError();
}

}  // namespace vc
