// Scout keyframe selection, Eq. (mmr) (Sec. 3.1): for each video, frame
// embeddings h_f and a prompt embedding h_t; frames join the selected set
// Omega greedily by
//     lambda * sim(h_f, h_t) - (1 - lambda) * max_{f' in Omega} sim(h_f, h_f')
// (cosine similarity) until k = ceil(p * F) frames are chosen.  Readings: the
// redundancy term is 0 while Omega is empty, ties go to the lower frame index,
// a zero vector has similarity 0 with everything.
//
// Three kernels, fp32 arithmetic:
//   scout_norm_kernel  one warp per frame / prompt row: the row scaled to unit
//                      length (zero rows stay zero);
//   scout_sim_kernel   per video the F x F cosine matrix S = Hn Hn^T, 64 x 64
//                      tiles (CUDA cores: the matrix is small and every later
//                      pick compares entries of it, so it is kept in fp32);
//   scout_mmr_kernel   one 1024-thread CTA per video runs the greedy loop:
//                      each thread holds up to four frames' relevance and
//                      running redundancy in registers, a block-wide argmax of
//                      (score, -index) picks the frame, and the picked frame's
//                      row of S updates the redundancies.  The picks are
//                      written in selection order, then (a block scan over the
//                      frame flags) in ascending frame order.
// Videos are independent: the batch is the data-parallel axis (one CTA each).
//
// Short videos (F <= 128 frames whose rows and S fit in 224 KB: the paper's 64 CLIP frames of
// width 512) take one fused kernel instead, scout_small_kernel: one CTA per
// video keeps the raw rows (d-major; dot products are scaled by the two
// inverse norms afterwards) and S in shared memory, builds S
// from 4 x 4 tiles of its upper triangle (four lanes per tile, each summing a
// quarter of the width with packed fmas, parts added in a fixed order), and
// runs the greedy loop inside one warp (up to four frames per lane; the warp
// argmax is a max reduction of the score key and a min reduction of the
// frame index; no block barriers).  Each video takes one path by its own size,
// so a batch returns what its videos return one by one.
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "profile.h"
#include "viscache.h"

namespace vc {
namespace {

constexpr int kScoutMaxReq = 64;
constexpr int kScoutMaxFrames = 4096;
constexpr int kMmrThreads = 1024;
constexpr int kFpt = kScoutMaxFrames / kMmrThreads;   // frames per thread
constexpr int kSimTile = 64;
constexpr int kSimChunk = 32;
constexpr size_t kWsAlign = 256;

struct ScoutTable {            // kernel parameter: per-video sizes and offsets
  int32_t n_req, D;
  float lam;
  int32_t F[kScoutMaxReq];     // frames
  int32_t k[kScoutMaxReq];     // keyframes
  int32_t k_off[kScoutMaxReq]; // first output row
  int64_t h_off[kScoutMaxReq]; // first frame row of H
  int64_t s_off[kScoutMaxReq]; // first element of the video's F x F matrix
};

constexpr int kSmallMaxFrames = 128;
constexpr int kSmallMaxFloats = 56000;       // shared memory of the fused kernel, in floats
constexpr int kSmallThreads = 1024;

// d-major row stride of the fused kernel's unit rows: F rounded up to 4 plus 4
// (16-byte aligned; the padding spreads a warp's transposed writes over banks)
__host__ __device__ __forceinline__ int small_ld(int F) { return ((F + 3) & ~3) + 4; }
__host__ __device__ __forceinline__ int64_t small_floats(int F, int D) {
  return (int64_t)D * small_ld(F) + (int64_t)F * F + D + F;
}
// A video small enough for the fused kernel (the paper's 64 frames of width 512 are).
__host__ __device__ __forceinline__ bool small_video(int F, int D) {
  return F <= kSmallMaxFrames && small_floats(F, D) <= kSmallMaxFloats;
}

__global__ void __launch_bounds__(256) scout_norm_kernel(const float* __restrict__ H,
                                                         const float* __restrict__ P, int64_t frames,
                                                         int n_req, int D, float* __restrict__ Hn,
                                                         float* __restrict__ Tn) {
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= frames + n_req) return;
  const float* src = row < frames ? H + row * D : P + (row - frames) * D;
  float* dst = row < frames ? Hn + row * D : Tn + (row - frames) * D;
  float ss = 0.f;
  for (int j = lane; j < D; j += 32) ss = fmaf(src[j], src[j], ss);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
  for (int j = lane; j < D; j += 32) dst[j] = src[j] * inv;
}

// S_r = Hn_r Hn_r^T; block (tile row, tile col, video), 256 threads, 4 x 4
// outputs each.
__global__ void __launch_bounds__(256) scout_sim_kernel(const __grid_constant__ ScoutTable tb,
                                                        const float* __restrict__ Hn,
                                                        float* __restrict__ S) {
  __shared__ float a[kSimChunk][kSimTile + 1], b[kSimChunk][kSimTile + 1];
  const int r = blockIdx.z;
  const int F = tb.F[r], D = tb.D;
  const int i0 = blockIdx.y * kSimTile, j0 = blockIdx.x * kSimTile;
  if (i0 >= F || j0 >= F || small_video(F, D)) return;
  const float* h = Hn + tb.h_off[r] * D;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int d0 = 0; d0 < D; d0 += kSimChunk) {
    for (int e = threadIdx.x; e < kSimChunk * kSimTile; e += 256) {
      const int row = e / kSimChunk, col = e % kSimChunk;   // consecutive threads read one row
      const int d = d0 + col;
      a[col][row] = (i0 + row < F && d < D) ? h[(int64_t)(i0 + row) * D + d] : 0.f;
      b[col][row] = (j0 + row < F && d < D) ? h[(int64_t)(j0 + row) * D + d] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int c = 0; c < kSimChunk; ++c) {
      float x[4], y[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        x[u] = a[c][ty * 4 + u];
        y[u] = b[c][tx * 4 + u];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(x[u], y[v], acc[u][v]);
    }
    __syncthreads();
  }
  float* s = S + tb.s_off[r];
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int i = i0 + ty * 4 + u, j = j0 + tx * 4 + v;
      if (i < F && j < F) s[(int64_t)i * F + j] = acc[u][v];
    }
}

// Order-preserving map of a float onto uint32 (ascending) and back.
__device__ __forceinline__ uint32_t ord_key(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord_value(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

// Block-wide maximum of a 64-bit key; every thread gets the result.
__device__ __forceinline__ unsigned long long block_max(unsigned long long v, unsigned long long* warp_max,
                                                        unsigned long long* result) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  if (lane == 0) warp_max[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = warp_max[lane];                      // 32 warps
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
      v = w > v ? w : v;
    }
    if (lane == 0) *result = v;
  }
  __syncthreads();
  return *result;
}

// Exclusive prefix count of a per-thread flag over the block (thread order);
// *total gets the block's count.
__device__ __forceinline__ int block_exclusive_count(bool flag, int* warp_cnt, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned m = __ballot_sync(0xffffffffu, flag);
  if (lane == 0) warp_cnt[warp] = __popc(m);
  __syncthreads();
  if (warp == 0) {
    const int c = warp_cnt[lane];
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    warp_cnt[lane] = incl - c;
    if (lane == 31) *total = incl;
  }
  __syncthreads();
  const int before = warp_cnt[warp] + __popc(m & ((1u << lane) - 1u));
  __syncthreads();                           // warp_cnt is reused by the next call
  return before;
}

__global__ void __launch_bounds__(kMmrThreads, 1) scout_mmr_kernel(const __grid_constant__ ScoutTable tb,
                                                                   const float* __restrict__ Hn,
                                                                   const float* __restrict__ Tn,
                                                                   const float* __restrict__ S,
                                                                   int32_t* __restrict__ order,
                                                                   int32_t* __restrict__ keyframes,
                                                                   float* __restrict__ gains) {
  __shared__ unsigned long long warp_max[32];
  __shared__ unsigned long long winner;
  __shared__ int warp_cnt[32];
  __shared__ int seg_total;
  const int r = blockIdx.x;
  const int F = tb.F[r], k = tb.k[r], D = tb.D;
  if (small_video(F, D)) return;               // the fused kernel takes it
  const float lam = tb.lam;
  const float* hn = Hn + tb.h_off[r] * D;
  const float* tn = Tn + (int64_t)r * D;
  const float* s = S + tb.s_off[r];
  const int t = threadIdx.x;

  float rel[kFpt], red[kFpt];
  bool sel[kFpt];
#pragma unroll
  for (int j = 0; j < kFpt; ++j) {
    const int f = t + j * kMmrThreads;
    float acc = 0.f;
    if (f < F)
      for (int d = 0; d < D; ++d) acc = fmaf(hn[(int64_t)f * D + d], tn[d], acc);
    rel[j] = acc;
    red[j] = 0.f;                            // empty selected set: no redundancy
    sel[j] = false;
  }
  for (int i = 0; i < k; ++i) {
    unsigned long long best = 0;             // below every real key
#pragma unroll
    for (int j = 0; j < kFpt; ++j) {
      const int f = t + j * kMmrThreads;
      if (f < F && !sel[j]) {
        const float sc = fmaf(-(1.f - lam), red[j], lam * rel[j]);   // same rounding in both paths
        const unsigned long long key = ((unsigned long long)ord_key(sc) << 32) | (0xffffffffu - (uint32_t)f);
        best = key > best ? key : best;
      }
    }
    const unsigned long long w = block_max(best, warp_max, &winner);
    const int fs = (int)(0xffffffffu - (uint32_t)w);
    if (t == 0) {
      order[tb.k_off[r] + i] = fs;
      if (gains) gains[tb.k_off[r] + i] = ord_value((uint32_t)(w >> 32));
    }
    const float* row = s + (int64_t)fs * F;   // S is symmetric: row fs = column fs
#pragma unroll
    for (int j = 0; j < kFpt; ++j) {
      const int f = t + j * kMmrThreads;
      if (f < F) {
        const float x = row[f];
        red[j] = i == 0 ? x : fmaxf(red[j], x);
        if (f == fs) sel[j] = true;
      }
    }
  }
  // ascending frame order: frame f = t + j*1024 goes to (selected frames
  // before it), counted segment by segment
  int base = 0;
#pragma unroll
  for (int j = 0; j < kFpt; ++j) {
    const int before = block_exclusive_count(sel[j], warp_cnt, &seg_total);
    if (sel[j]) keyframes[tb.k_off[r] + base + before] = t + j * kMmrThreads;
    base += seg_total;
    __syncthreads();                         // seg_total is rewritten by the next segment
  }
}

__global__ void __launch_bounds__(kSmallThreads) scout_small_kernel(const __grid_constant__ ScoutTable tb,
                                                                    const float* __restrict__ H,
                                                                    const float* __restrict__ P,
                                                                    int32_t* __restrict__ order,
                                                                    int32_t* __restrict__ keyframes,
                                                                    float* __restrict__ gains) {
  extern __shared__ __align__(16) float sm[];
  __shared__ float inv_norm[kSmallMaxFrames + 1];
  __shared__ int pick[kSmallMaxFrames];
  __shared__ float pick_gain[kSmallMaxFrames];
  const int r = blockIdx.x;
  const int F = tb.F[r], D = tb.D;
  if (!small_video(F, D)) return;              // the three-kernel path takes it
  const int k = tb.k[r], ld = small_ld(F);
  const float lam = tb.lam;
  float* hT = sm;                              // [D][ld] unit rows, d-major
  float* S = hT + (size_t)D * ld;              // [F][F]
  float* tn = S + (size_t)F * F;               // [D] unit prompt
  float* rel = tn + D;                         // [F] relevance
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* h = H + tb.h_off[r] * D;
  // raw rows into shared memory (d-major; the prompt as row F) and each
  // row's inverse norm; dot products of raw rows are scaled by both inverse
  // norms afterwards (one pass over global memory, no scaling pass)
  for (int row = warp; row <= F; row += kSmallThreads / 32) {
    const float* src = row < F ? h + (int64_t)row * D : P + (int64_t)r * D;
    float ss = 0.f;
#pragma unroll 8
    for (int j = lane; j < D; j += 32) {
      const float x = src[j];
      ss = fmaf(x, x, ss);
      if (row < F) hT[(size_t)j * ld + row] = x;
      else tn[j] = x;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) inv_norm[row] = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
  }
  __syncthreads();
  // S = hn hn^T: 4 x 4 tiles of the upper triangle, mirrored.  Four adjacent
  // lanes share a tile, lane part p summing widths p, p+4, ... (four frames
  // per 16-byte load, two products per packed fma); the parts are added as
  // (p0 + p1) + (p2 + p3) by two shuffles.
  const int nt = (F + 3) / 4;
  const int ntri = nt * (nt + 1) / 2;
  for (int item = threadIdx.x; item < 4 * ((ntri + 7) / 8) * 8; item += kSmallThreads) {
    const int t = item >> 2, part = item & 3;
    const bool live = t < ntri;
    int a = 0, rem = live ? t : 0;
    while (rem >= nt - a) {
      rem -= nt - a;
      ++a;
    }
    const int i0 = a * 4, j0 = (a + rem) * 4;
    float2 acc[4][2];
#pragma unroll
    for (int u = 0; u < 4; ++u) acc[u][0] = acc[u][1] = make_float2(0.f, 0.f);
    if (live) {
#pragma unroll 4
      for (int d = part; d < D; d += 4) {
        const float4 x = *reinterpret_cast<const float4*>(hT + (size_t)d * ld + i0);
        const float4 y = *reinterpret_cast<const float4*>(hT + (size_t)d * ld + j0);
        const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc[u][0] = __ffma2_rn(make_float2(xs[u], xs[u]), make_float2(y.x, y.y), acc[u][0]);
          acc[u][1] = __ffma2_rn(make_float2(xs[u], xs[u]), make_float2(y.z, y.w), acc[u][1]);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int v = 0; v < 2; ++v) {
        float2 w = acc[u][v];
        w.x += __shfl_xor_sync(0xffffffffu, w.x, 1);
        w.y += __shfl_xor_sync(0xffffffffu, w.y, 1);
        w.x += __shfl_xor_sync(0xffffffffu, w.x, 2);
        w.y += __shfl_xor_sync(0xffffffffu, w.y, 2);
        acc[u][v] = w;
      }
    if (live && part == 0) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float v4[4] = {acc[u][0].x, acc[u][0].y, acc[u][1].x, acc[u][1].y};
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int i = i0 + u, j = j0 + v;
          if (i < F && j < F) {
            const float c = (v4[v] * inv_norm[i]) * inv_norm[j];
            S[(size_t)i * F + j] = c;
            S[(size_t)j * F + i] = c;
          }
        }
      }
    }
  }
  // relevance: four lanes per frame, parts combined as for S
  for (int item = threadIdx.x; item < 4 * ((F + 7) / 8) * 8; item += kSmallThreads) {
    const int f = item >> 2, part = item & 3;
    float acc = 0.f;
    if (f < F)
      for (int d = part; d < D; d += 4) acc = fmaf(hT[(size_t)d * ld + f], tn[d], acc);
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);
    if (f < F && part == 0) rel[f] = (acc * inv_norm[f]) * inv_norm[F];
  }
  __syncthreads();
  if (warp != 0) return;
  // greedy loop in warp 0: lane holds frames lane, lane + 32, ...
  constexpr int kLaneFrames = kSmallMaxFrames / 32;
  float rl[kLaneFrames], red[kLaneFrames];
  bool sel[kLaneFrames];
#pragma unroll
  for (int j = 0; j < kLaneFrames; ++j) {
    const int f = lane + 32 * j;
    rl[j] = f < F ? rel[f] : 0.f;
    red[j] = 0.f;                                // empty selected set: no redundancy
    sel[j] = f >= F;                             // frames past F are never picked
  }
  const int o0 = tb.k_off[r];
  for (int i = 0; i < k; ++i) {
    // this lane's best frame (highest score, then lowest index), then the
    // warp's: the highest score key, and the lowest frame holding it
    uint32_t kb = 0, fb = 0xffffffffu;
#pragma unroll
    for (int j = 0; j < kLaneFrames; ++j) {
      if (!sel[j]) {
        const uint32_t key = ord_key(fmaf(-(1.f - lam), red[j], lam * rl[j]));
        if (key > kb) {
          kb = key;
          fb = (uint32_t)(lane + 32 * j);
        }
      }
    }
    const uint32_t kmax = __reduce_max_sync(0xffffffffu, kb);
    const int fs = (int)__reduce_min_sync(0xffffffffu, kb == kmax ? fb : 0xffffffffu);
    if (lane == 0) {
      pick[i] = fs;
      pick_gain[i] = ord_value(kmax);
    }
    const float* row = S + (size_t)fs * F;
#pragma unroll
    for (int j = 0; j < kLaneFrames; ++j) {
      const int f = lane + 32 * j;
      if (f < F) {
        red[j] = i == 0 ? row[f] : fmaxf(red[j], row[f]);
        if (f == fs) sel[j] = true;
      }
    }
  }
  __syncwarp();
  for (int i = lane; i < k; i += 32) {
    order[o0 + i] = pick[i];
    if (gains) gains[o0 + i] = pick_gain[i];
  }
  // ascending frame order: frame lane + 32 j after the picks of lower frames
  int base = 0;
#pragma unroll
  for (int j = 0; j < kLaneFrames; ++j) {
    const bool mine = sel[j] && lane + 32 * j < F;
    const unsigned m = __ballot_sync(0xffffffffu, mine);
    if (mine) keyframes[o0 + base + __popc(m & ((1u << lane) - 1u))] = lane + 32 * j;
    base += __popc(m);
  }
}

inline size_t align_up(size_t x) { return (x + kWsAlign - 1) / kWsAlign * kWsAlign; }

struct ScoutLayout {
  size_t o_hn = 0, o_tn = 0, o_s = 0, total = 0;
  int64_t frames = 0, s_elems = 0;
};

// Host checks and the per-video table; returns VC_OK or an error code.
int scout_plan(int32_t n_req, const int32_t* n_frames, int32_t D, uint32_t p_num, uint32_t p_den,
               float lam, ScoutTable* tb, ScoutLayout* lay) {
  if (n_req < 1 || n_req > kScoutMaxReq || !n_frames || D < 1 || D > 8192) return VC_ERR_INVALID_ARG;
  if (p_den == 0 || p_num == 0 || p_num > p_den || !(lam >= 0.f && lam <= 1.f)) return VC_ERR_INVALID_ARG;
  tb->n_req = n_req;
  tb->D = D;
  tb->lam = lam;
  int64_t frames = 0, s_elems = 0;
  int32_t k_off = 0;
  for (int r = 0; r < n_req; ++r) {
    const int32_t F = n_frames[r];
    if (F < 1 || F > kScoutMaxFrames) return VC_ERR_INVALID_ARG;
    // k = ceil(p F), at least 1 (p > 0 and F >= 1 give k >= 1), at most F
    const int64_t k = ((int64_t)p_num * F + p_den - 1) / p_den;
    tb->F[r] = F;
    tb->k[r] = (int32_t)k;
    tb->k_off[r] = k_off;
    tb->h_off[r] = frames;
    tb->s_off[r] = s_elems;
    k_off += (int32_t)k;
    frames += F;
    s_elems += (int64_t)F * F;
  }
  lay->frames = frames;
  lay->s_elems = s_elems;
  lay->o_hn = 0;
  lay->o_tn = align_up(sizeof(float) * frames * D);
  lay->o_s = lay->o_tn + align_up(sizeof(float) * (size_t)n_req * D);
  lay->total = lay->o_s + align_up(sizeof(float) * s_elems);
  return VC_OK;
}

}  // namespace
}  // namespace vc

using namespace vc;

extern "C" size_t viscache_scout_workspace_size(int32_t n_req, const int32_t* n_frames, int32_t D) {
  ScoutTable tb;
  ScoutLayout lay;
  return scout_plan(n_req, n_frames, D, 1, 1, 0.5f, &tb, &lay) == VC_OK ? lay.total : 0;
}

extern "C" int viscache_scout_sizes(int32_t n_req, const int32_t* n_frames, uint32_t p_num,
                                    uint32_t p_den, int32_t* k_out) {
  if (!k_out) return VC_ERR_INVALID_ARG;
  ScoutTable tb;
  ScoutLayout lay;
  const int rc = scout_plan(n_req, n_frames, 1, p_num, p_den, 0.5f, &tb, &lay);
  if (rc != VC_OK) return rc;
  for (int r = 0; r < n_req; ++r) k_out[r] = tb.k[r];
  return VC_OK;
}

extern "C" int viscache_scout_mmr(const float* H, const float* prompt, int32_t n_req,
                                  const int32_t* n_frames, int32_t D, float lambda, uint32_t p_num,
                                  uint32_t p_den, int32_t* order_out, int32_t* keyframes_out,
                                  float* gains_out, int32_t* k_out, void* ws, size_t ws_bytes,
                                  void* stream) {
  ScoutTable tb;
  ScoutLayout lay;
  const int rc = scout_plan(n_req, n_frames, D, p_num, p_den, lambda, &tb, &lay);
  if (rc != VC_OK) return rc;
  if (!H || !prompt || !order_out || !keyframes_out) return VC_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(H) | reinterpret_cast<uintptr_t>(prompt)) & 3u) return VC_ERR_INVALID_ARG;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kWsAlign - 1)) != 0 || ws_bytes < lay.total)
    return VC_ERR_WORKSPACE;
  if (k_out)
    for (int r = 0; r < n_req; ++r) k_out[r] = tb.k[r];
  uint8_t* w = static_cast<uint8_t*>(ws);
  float* Hn = reinterpret_cast<float*>(w + lay.o_hn);
  float* Tn = reinterpret_cast<float*>(w + lay.o_tn);
  float* S = reinterpret_cast<float*>(w + lay.o_s);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // each video goes to the fused kernel or to the three-kernel path by its size
  int fmax_small = 0, fmax_large = 0;
  for (int r = 0; r < n_req; ++r) {
    if (small_video(tb.F[r], D)) fmax_small = tb.F[r] > fmax_small ? tb.F[r] : fmax_small;
    else fmax_large = tb.F[r] > fmax_large ? tb.F[r] : fmax_large;
  }
  if (fmax_small > 0) {
    ProfileScope ps("scout_small", st);
    const size_t smem = sizeof(float) * (size_t)small_floats(fmax_small, D);
    if (cudaFuncSetAttribute(scout_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return VC_ERR_CUDA;
    scout_small_kernel<<<(unsigned)n_req, kSmallThreads, smem, st>>>(tb, H, prompt, order_out, keyframes_out,
                                                                    gains_out);
    if (cudaGetLastError() != cudaSuccess) return VC_ERR_CUDA;
  }
  if (fmax_large == 0) return VC_OK;
  {
    ProfileScope ps("scout_norm", st);
    const int64_t rows = lay.frames + n_req;
    scout_norm_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(H, prompt, lay.frames, n_req, D, Hn, Tn);
    if (cudaGetLastError() != cudaSuccess) return VC_ERR_CUDA;
  }
  {
    ProfileScope ps("scout_sim", st);
    const unsigned tiles = (unsigned)((fmax_large + kSimTile - 1) / kSimTile);
    scout_sim_kernel<<<dim3(tiles, tiles, (unsigned)n_req), 256, 0, st>>>(tb, Hn, S);
    if (cudaGetLastError() != cudaSuccess) return VC_ERR_CUDA;
  }
  {
    ProfileScope ps("scout_mmr", st);
    scout_mmr_kernel<<<(unsigned)n_req, kMmrThreads, 0, st>>>(tb, Hn, Tn, S, order_out, keyframes_out,
                                                              gains_out);
    if (cudaGetLastError() != cudaSuccess) return VC_ERR_CUDA;
  }
  return VC_OK;
}
