// Decode attention over the compressed cache (Sec. 2 "VLLM Decoding", with the
// visual part of layer l's cache replaced by PruneKV's (K_new, V_new), Sec. 3.2):
//     out_j = softmax(q_j K_g^T * scale) V_g,  g = j // G,
// over KV head g's B kept visual rows of the layer followed by its T text rows.
//
// A decode step reads the whole layer cache once for a handful of query rows,
// so the work is bound by those reads (2*G flops per K or V element): CUDA
// cores, every K and V element loaded once per step.
//   decode_partial_kernel  one 128-thread CTA per (request, KV head, split of
//                          kSplit keys), the G query rows in shared memory.
//                          Phase 1: each thread takes whole keys (16-byte row
//                          loads) and forms their G logits against broadcast
//                          query values, keeping its running maxima; a block
//                          max per query follows.  Phase 2: each thread turns
//                          its own keys' logits into exp2 terms and sums them.
//                          Phase 3: threads own two output dimensions of a key
//                          slice and sum p * V over the slice's keys (V rows
//                          read coalesced, a key's G probabilities as 16-byte
//                          broadcasts); slices are added in shared memory.
//                          Writes the unnormalised partial output and (max, sum).
//   decode_combine_kernel  one warp per (request, query head): merges the
//                          splits' states and writes out = O / sum.
// A query with no keys at all (an evicted layer, no text) gets zeros.
#include <cuda_bf16.h>
#include <stdint.h>

#include "kernels.h"
#include "profile.h"
#include "vc_common.cuh"

namespace vc {
namespace {

constexpr int kSplit = 512;                   // keys per partial CTA
constexpr int kDecThreads = 128;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kGm = kDecodeMaxGroup;
constexpr float kLog2eF = 1.4426950408889634f;

__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
__device__ __forceinline__ float2 load2(const float* p) { return *reinterpret_cast<const float2*>(p); }
__device__ __forceinline__ float2 load2(const __nv_bfloat16* p) {
  const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
  return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

__device__ __forceinline__ int find_req(const DecodeTable& tb, int unit) {
  int lo = 0, hi = tb.n_req - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tb.req[mid].unit0 <= unit) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <typename T, int D>
__global__ void __launch_bounds__(kDecThreads) decode_partial_kernel(
    const __grid_constant__ DecodeTable tb, const T* __restrict__ q, const T* __restrict__ Kc,
    const T* __restrict__ Vc, const T* __restrict__ Kt, const T* __restrict__ Vt,
    float* __restrict__ part_o, float2* __restrict__ part_ml) {
  constexpr int TPK = D / 2;                  // phase-3 threads per key, two dimensions each
  constexpr int KS = kDecThreads / TPK;       // phase-3 key slices
  __shared__ __align__(16) float qs[kGm][D];
  __shared__ __align__(16) float ps[kSplit][kGm];        // logits, then exp2 terms
  __shared__ __align__(16) float red[KS - 1][kGm][D];
  __shared__ float wmax[kDecWarps][kGm], wsum[kDecWarps][kGm];
  const int unit = blockIdx.x;
  const int r = find_req(tb, unit);
  const DecodeReq rq = tb.req[r];
  const int u = unit - rq.unit0;
  const int g = u / rq.nsplit, s = u % rq.nsplit;
  const int G = tb.G;
  const int k0 = s * kSplit;
  const int nk = min(kSplit, rq.B + rq.T - k0);
  const int nv = max(0, min(nk, rq.B - k0));  // the split's visual keys come first
  const int64_t vis0 = rq.vis_row0 + (int64_t)g * rq.B + k0;
  const int64_t txt0 = rq.txt_row0 + (int64_t)g * rq.T + (k0 + nv - rq.B);
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  // query rows g*G ... of request r, scaled into log2 units
  const float c2 = tb.scale * kLog2eF;
  for (int e = t; e < kGm * D; e += kDecThreads) {
    const int jj = e / D, d = e % D;
    qs[jj][d] = jj < G ? Elem<T>::to_f(q[((int64_t)r * tb.Hq + g * G + jj) * D + d]) * c2 : 0.f;
  }
  __syncthreads();
  // phase 1: logits of this thread's keys and its running maxima
  float m_t[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) m_t[jj] = -INFINITY;
  for (int kk = t; kk < nk; kk += kDecThreads) {
    const T* krow = kk < nv ? Kc + (vis0 + kk) * D : Kt + (txt0 + (kk - nv)) * D;
    float acc[kGm];
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) acc[jj] = 0.f;
#pragma unroll 2
    for (int d0 = 0; d0 < D; d0 += 8) {
      float kv[8];
      load8(krow + d0, kv);
#pragma unroll
      for (int jj = 0; jj < kGm; ++jj) {
        if (jj < G) {
          const float4 x = *reinterpret_cast<const float4*>(&qs[jj][d0]);
          const float4 y = *reinterpret_cast<const float4*>(&qs[jj][d0 + 4]);
          acc[jj] = fmaf(kv[0], x.x, acc[jj]);
          acc[jj] = fmaf(kv[1], x.y, acc[jj]);
          acc[jj] = fmaf(kv[2], x.z, acc[jj]);
          acc[jj] = fmaf(kv[3], x.w, acc[jj]);
          acc[jj] = fmaf(kv[4], y.x, acc[jj]);
          acc[jj] = fmaf(kv[5], y.y, acc[jj]);
          acc[jj] = fmaf(kv[6], y.z, acc[jj]);
          acc[jj] = fmaf(kv[7], y.w, acc[jj]);
        }
      }
    }
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) m_t[jj] = fmaxf(m_t[jj], acc[jj]);
    *reinterpret_cast<float4*>(&ps[kk][0]) = make_float4(acc[0], acc[1], acc[2], acc[3]);
    *reinterpret_cast<float4*>(&ps[kk][4]) = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m_t[jj] = fmaxf(m_t[jj], __shfl_xor_sync(0xffffffffu, m_t[jj], o));
  }
  if (lane == 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) wmax[warp][jj] = m_t[jj];
  }
  __syncthreads();
  // phase 2: exp2 terms of this thread's keys against the split maxima
  float M[kGm], l_t[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
    M[jj] = wmax[0][jj];
#pragma unroll
    for (int w = 1; w < kDecWarps; ++w) M[jj] = fmaxf(M[jj], wmax[w][jj]);
    l_t[jj] = 0.f;
  }
  for (int kk = t; kk < nk; kk += kDecThreads) {
    float4 a = *reinterpret_cast<const float4*>(&ps[kk][0]);
    float4 b = *reinterpret_cast<const float4*>(&ps[kk][4]);
    float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) {
      x[jj] = jj < G ? exp2f(x[jj] - M[jj]) : 0.f;
      l_t[jj] += x[jj];
    }
    *reinterpret_cast<float4*>(&ps[kk][0]) = make_float4(x[0], x[1], x[2], x[3]);
    *reinterpret_cast<float4*>(&ps[kk][4]) = make_float4(x[4], x[5], x[6], x[7]);
  }
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l_t[jj] += __shfl_xor_sync(0xffffffffu, l_t[jj], o);
  }
  if (lane == 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) wsum[warp][jj] = l_t[jj];
  }
  __syncthreads();
  if (t < G) {
    float m = wmax[0][t], l = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) {
      m = fmaxf(m, wmax[w][t]);
      l += wsum[w][t];
    }
    part_ml[(int64_t)unit * kGm + t] = make_float2(m, l);
  }
  // phase 3: O[jj][dims] = sum_k p[k][jj] V[k][dims] over key slice ks
  const int dp = 2 * (t % TPK), ks = t / TPK;
  float o0[kGm], o1[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) o0[jj] = o1[jj] = 0.f;
#pragma unroll 4
  for (int kk = ks; kk < nk; kk += KS) {
    const T* vrow = kk < nv ? Vc + (vis0 + kk) * D : Vt + (txt0 + (kk - nv)) * D;
    const float2 v = load2(vrow + dp);
    const float4 a = *reinterpret_cast<const float4*>(&ps[kk][0]);
    const float4 b = *reinterpret_cast<const float4*>(&ps[kk][4]);
    const float p[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) {
      o0[jj] = fmaf(p[jj], v.x, o0[jj]);
      o1[jj] = fmaf(p[jj], v.y, o1[jj]);
    }
  }
  if (ks > 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj)
      *reinterpret_cast<float2*>(&red[ks - 1][jj][dp]) = make_float2(o0[jj], o1[jj]);
  }
  __syncthreads();
  if (ks == 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) {
      if (jj < G) {
        float x = o0[jj], y = o1[jj];
#pragma unroll
        for (int i = 0; i < KS - 1; ++i) {
          const float2 z = *reinterpret_cast<const float2*>(&red[i][jj][dp]);
          x += z.x;
          y += z.y;
        }
        *reinterpret_cast<float2*>(&part_o[((int64_t)unit * kGm + jj) * D + dp]) = make_float2(x, y);
      }
    }
  }
}

// One warp per (request, query head): merge the splits of its KV head.
template <typename T, int D>
__global__ void __launch_bounds__(128) decode_combine_kernel(const __grid_constant__ DecodeTable tb,
                                                             const float* __restrict__ part_o,
                                                             const float2* __restrict__ part_ml,
                                                             T* __restrict__ out) {
  const int w = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (w >= tb.n_req * tb.Hq) return;
  const int r = w / tb.Hq, j = w % tb.Hq;
  const DecodeReq rq = tb.req[r];
  const int g = j / tb.G, jj = j % tb.G;
  const int64_t u0 = rq.unit0 + (int64_t)g * rq.nsplit;
  const int ns = rq.B + rq.T > 0 ? rq.nsplit : 0;
  float M = -INFINITY;
  for (int s = 0; s < ns; ++s) M = fmaxf(M, part_ml[(u0 + s) * kDecodeMaxGroup + jj].x);
  float Lsum = 0.f;
  float acc[(D + 31) / 32];
#pragma unroll
  for (int i = 0; i < (D + 31) / 32; ++i) acc[i] = 0.f;
  for (int s = 0; s < ns; ++s) {
    const float2 ml = part_ml[(u0 + s) * kDecodeMaxGroup + jj];
    const float w_s = exp2f(ml.x - M);
    Lsum = fmaf(ml.y, w_s, Lsum);
    const float* o = part_o + ((u0 + s) * kDecodeMaxGroup + jj) * D;
#pragma unroll
    for (int i = 0; i < (D + 31) / 32; ++i)
      if (lane + 32 * i < D) acc[i] = fmaf(o[lane + 32 * i], w_s, acc[i]);
  }
  const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
  T* dst = out + ((int64_t)r * tb.Hq + j) * D;
#pragma unroll
  for (int i = 0; i < (D + 31) / 32; ++i)
    if (lane + 32 * i < D) dst[lane + 32 * i] = Elem<T>::from_f(acc[i] * inv);
}

template <typename T, int D>
cudaError_t launch_decode_t(const DecodeTable& tb, const void* q, const void* Kc, const void* Vc,
                            const void* Kt, const void* Vt, void* out, float* part_o, float2* part_ml,
                            cudaStream_t st) {
  if (tb.units > 0) {
    ProfileScope ps("decode_partial", st);
    decode_partial_kernel<T, D><<<(unsigned)tb.units, kDecThreads, 0, st>>>(
        tb, static_cast<const T*>(q), static_cast<const T*>(Kc), static_cast<const T*>(Vc),
        static_cast<const T*>(Kt), static_cast<const T*>(Vt), part_o, part_ml);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  ProfileScope ps("decode_combine", st);
  const int warps = tb.n_req * tb.Hq;
  decode_combine_kernel<T, D><<<(unsigned)((warps + 3) / 4), 128, 0, st>>>(tb, part_o, part_ml,
                                                                          static_cast<T*>(out));
  return cudaGetLastError();
}

}  // namespace

int decode_split_keys() { return kSplit; }

cudaError_t launch_decode(const DecodeTable& tb, int dtype, int d, const void* q, const void* Kc,
                          const void* Vc, const void* Kt, const void* Vt, void* out, float* part_o,
                          float2* part_ml, cudaStream_t st) {
  if (dtype == VC_BF16) {
    if (d == 128) return launch_decode_t<__nv_bfloat16, 128>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
    return launch_decode_t<__nv_bfloat16, 64>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
  }
  if (d == 128) return launch_decode_t<float, 128>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
  return launch_decode_t<float, 64>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
}

}  // namespace vc
