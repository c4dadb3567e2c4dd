// Token scoring on CUDA cores (fp32 FFMA), Eq. (token_score).
//
// Two passes per (request, layer, KV head):
//   pass 1  lse2[l][j][i] = log2 sum_v exp2(x2_{j,i,v}),  x2 = scale*log2(e) * q_{j,i}.k_v
//   pass 2  s[g][v] += sum_{j in group g} sum_i exp2(x2_{j,i,v} - lse2[l][j][i])
// In the shared ranking mode pass 2 keeps each token's sum over all layers in
// registers (compensated) and writes s = sum / L once; in the layer-specific
// mode it writes one row per layer.  This path serves fp32 inputs and is the
// portable reference path for bf16.
#include "vc_common.cuh"
#include "kernels.h"
#include "profile.h"

namespace vc {
namespace {

constexpr int kThreads = 256;   // 8 warps
constexpr int kRows = 32;       // query rows per tile (4 per warp)
constexpr int kKeys = 64;       // keys per tile (2 per lane)

// Stage rows [r0, r0+count) of a (request, layer, KV-head) row set into smem.
// Row rho of the group maps to query head g*G + rho / W, window row rho % W.
template <typename T, int D>
__device__ __forceinline__ void load_q_tile(float (*qs)[D + 4], const T* Qw, const Req& rq,
                                            const Shape& sh, int l, int g, int r0, int rows) {
  for (int e = threadIdx.x; e < kRows * (D / 4); e += kThreads) {
    const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r0 + r < rows) {
      const int rho = r0 + r;
      const int j = g * sh.G + rho / rq.W, i = rho % rq.W;
      v = load4(Qw + rq.q_off + ((int64_t)(l * sh.Hq + j) * rq.W + i) * D + c4);
    }
    qs[r][c4 + 0] = v.x; qs[r][c4 + 1] = v.y; qs[r][c4 + 2] = v.z; qs[r][c4 + 3] = v.w;
  }
}

template <typename T, int D>
__device__ __forceinline__ void load_k_tile(float (*ks)[D + 1], const T* Kl, int n, int v0) {
  for (int e = threadIdx.x; e < kKeys * (D / 4); e += kThreads) {
    const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (v0 + r < n) v = load4(Kl + (int64_t)(v0 + r) * D + c4);
    ks[r][c4 + 0] = v.x; ks[r][c4 + 1] = v.y; ks[r][c4 + 2] = v.z; ks[r][c4 + 3] = v.w;
  }
}

// acc[a][b] = q_row(4*warp + a) . k_key(lane + 32*b)
template <int D>
__device__ __forceinline__ void tile_dots(float acc[4][2], const float (*qs)[D + 4],
                                          const float (*ks)[D + 1], int warp, int lane) {
#pragma unroll
  for (int a = 0; a < 4; ++a) acc[a][0] = acc[a][1] = 0.f;
#pragma unroll 8
  for (int c = 0; c < D; ++c) {
    const float k0 = ks[lane][c], k1 = ks[lane + 32][c];
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const float q = qs[4 * warp + a][c];
      acc[a][0] = fmaf(q, k0, acc[a][0]);
      acc[a][1] = fmaf(q, k1, acc[a][1]);
    }
  }
}

// Pass 1: grid (units over (request, row tile), L, Hkv).
template <typename T, int D>
__global__ void __launch_bounds__(kThreads) lse_simt_kernel(const T* __restrict__ Qw,
                                                            const T* __restrict__ K, Shape sh,
                                                            Tables tb, float* __restrict__ lse) {
  extern __shared__ float4 smem4[];
  float (*qs)[D + 4] = reinterpret_cast<float (*)[D + 4]>(smem4);
  float (*ks)[D + 1] = reinterpret_cast<float (*)[D + 1]>(reinterpret_cast<float*>(smem4) + kRows * (D + 4));
  const int r = upper_index(tb.unit0_lse, sh.n_req, (int32_t)blockIdx.x);
  const Req rq = tb.req[r];
  const int l = blockIdx.y, g = blockIdx.z;
  const int rows = sh.G * rq.W;
  const int r0 = (blockIdx.x - tb.unit0_lse[r]) * kRows;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const T* Kl = K + rq.kv_off + (int64_t)(l * sh.Hkv + g) * rq.n * D;

  load_q_tile<T, D>(qs, Qw, rq, sh, l, g, r0, rows);
  float m[4], z[4];
#pragma unroll
  for (int a = 0; a < 4; ++a) { m[a] = -INFINITY; z[a] = 0.f; }

  for (int v0 = 0; v0 < rq.n; v0 += kKeys) {
    __syncthreads();
    load_k_tile<T, D>(ks, Kl, rq.n, v0);
    __syncthreads();
    float acc[4][2];
    tile_dots<D>(acc, qs, ks, warp, lane);
    const bool ok0 = v0 + lane < rq.n, ok1 = v0 + lane + 32 < rq.n;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const float x0 = ok0 ? acc[a][0] * sh.scale_log2 : -INFINITY;
      const float x1 = ok1 ? acc[a][1] * sh.scale_log2 : -INFINITY;
      const float mn = fmaxf(m[a], fmaxf(x0, x1));
      if (mn != -INFINITY) {
        z[a] = z[a] * exp2f(m[a] - mn) + exp2f(x0 - mn) + exp2f(x1 - mn);
        m[a] = mn;
      }
    }
  }
  // merge the 32 lanes' partial (max, sum) of each row
#pragma unroll
  for (int a = 0; a < 4; ++a) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, m[a], off);
      const float zo = __shfl_xor_sync(0xffffffffu, z[a], off);
      const float mn = fmaxf(m[a], mo);
      if (mn != -INFINITY) {
        z[a] = z[a] * exp2f(m[a] - mn) + zo * exp2f(mo - mn);
        m[a] = mn;
      }
    }
    const int rho = r0 + 4 * warp + a;
    if (lane == 0 && rho < rows) {
      const int j = g * sh.G + rho / rq.W, i = rho % rq.W;
      lse[rq.lse_off + (int64_t)(l * sh.Hq + j) * rq.W + i] = m[a] + log2f(z[a]);
    }
  }
}

// Pass 2: grid (units over (request, key tile), Hkv).  Loops over all layers.
// lse_nat != nullptr: normalisers come from the caller (natural log, [L][Hq][W]).
template <typename T, int D>
__global__ void __launch_bounds__(kThreads) colsum_simt_kernel(const T* __restrict__ Qw,
                                                               const T* __restrict__ K, Shape sh,
                                                               Tables tb,
                                                               const float* __restrict__ lse,
                                                               const float* __restrict__ lse_nat,
                                                               float* __restrict__ scores) {
  extern __shared__ float4 smem4[];
  float* sm = reinterpret_cast<float*>(smem4);
  float (*qs)[D + 4] = reinterpret_cast<float (*)[D + 4]>(sm);
  float (*ks)[D + 1] = reinterpret_cast<float (*)[D + 1]>(sm + kRows * (D + 4));
  float* ls = sm + kRows * (D + 4) + kKeys * (D + 1);
  float (*red)[kKeys] = reinterpret_cast<float (*)[kKeys]>(ls + kRows);
  const int r = upper_index(tb.unit0_col, sh.n_req, (int32_t)blockIdx.x);
  const Req rq = tb.req[r];
  const int g = blockIdx.y;
  const int v0 = (blockIdx.x - tb.unit0_col[r]) * kKeys;
  const int rows = sh.G * rq.W;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  Kahan tot[2];
  tot[0].init(); tot[1].init();
  for (int l = 0; l < sh.L; ++l) {
    const T* Kl = K + rq.kv_off + (int64_t)(l * sh.Hkv + g) * rq.n * D;
    __syncthreads();
    load_k_tile<T, D>(ks, Kl, rq.n, v0);
    Kahan lay[2];
    lay[0].init(); lay[1].init();
    for (int r0 = 0; r0 < rows; r0 += kRows) {
      __syncthreads();
      load_q_tile<T, D>(qs, Qw, rq, sh, l, g, r0, rows);
      if (threadIdx.x < kRows) {
        const int rho = r0 + threadIdx.x;
        float v = INFINITY;   // padded rows contribute exp2(-inf) = 0
        if (rho < rows) {
          const int j = g * sh.G + rho / rq.W, i = rho % rq.W;
          const int64_t o = rq.lse_off + (int64_t)(l * sh.Hq + j) * rq.W + i;
          v = lse_nat ? lse_nat[o] * kLog2e : lse[o];
        }
        ls[threadIdx.x] = v;
      }
      __syncthreads();
      float acc[4][2];
      tile_dots<D>(acc, qs, ks, warp, lane);
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float lz = ls[4 * warp + a];
        lay[0].add(exp2f(fmaf(acc[a][0], sh.scale_log2, -lz)));
        lay[1].add(exp2f(fmaf(acc[a][1], sh.scale_log2, -lz)));
      }
    }
    if (sh.rank_mode == VC_RANK_PER_LAYER) {
      __syncthreads();
      red[warp][lane] = lay[0].s;
      red[warp][lane + 32] = lay[1].s;
      __syncthreads();
      if (threadIdx.x < kKeys && v0 + threadIdx.x < rq.n) {
        Kahan k; k.init();
        for (int w = 0; w < 8; ++w) k.add(red[w][threadIdx.x]);
        scores[rq.s_off + ((int64_t)l * sh.Hkv + g) * rq.n + v0 + threadIdx.x] = k.s;
      }
    } else {
      tot[0].add(lay[0].s);
      tot[1].add(lay[1].s);
    }
  }
  if (sh.rank_mode != VC_RANK_PER_LAYER) {
    __syncthreads();
    red[warp][lane] = tot[0].s;
    red[warp][lane + 32] = tot[1].s;
    __syncthreads();
    if (threadIdx.x < kKeys && v0 + threadIdx.x < rq.n) {
      Kahan k; k.init();
      for (int w = 0; w < 8; ++w) k.add(red[w][threadIdx.x]);
      scores[rq.s_off + (int64_t)g * rq.n + v0 + threadIdx.x] = k.s / (float)sh.L;
    }
  }
}

template <typename T, int D>
cudaError_t launch_t(const void* Qw, const void* K, const Shape& sh, const Tables& tb,
                     int units_lse, int units_col, float* lse, const float* lse_nat,
                     float* scores, cudaStream_t st) {
  const T* q = static_cast<const T*>(Qw);
  const T* k = static_cast<const T*>(K);
  const size_t smem1 = sizeof(float) * (kRows * (D + 4) + kKeys * (D + 1));
  const size_t smem2 = smem1 + sizeof(float) * (kRows + 8 * kKeys);
  cudaError_t e;
  if (!lse_nat) {
    e = cudaFuncSetAttribute(lse_simt_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return e;
    ProfileScope ps("score_lse_simt", st);
    lse_simt_kernel<T, D><<<dim3(units_lse, sh.L, sh.Hkv), kThreads, smem1, st>>>(q, k, sh, tb, lse);
  }
  e = cudaFuncSetAttribute(colsum_simt_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  if (e != cudaSuccess) return e;
  {
    ProfileScope ps("score_colsum_simt", st);
    colsum_simt_kernel<T, D><<<dim3(units_col, sh.Hkv), kThreads, smem2, st>>>(q, k, sh, tb, lse,
                                                                             lse_nat, scores);
  }
  return cudaGetLastError();
}

}  // namespace

int score_rows_per_tile_simt() { return kRows; }
int score_keys_per_tile_simt() { return kKeys; }

cudaError_t launch_score_simt(int dtype, const void* Qw, const void* K, const Shape& sh,
                              const Tables& tb, int units_lse, int units_col, float* lse,
                              const float* lse_nat, float* scores, cudaStream_t st) {
  if (dtype == VC_F32) {
    if (sh.d == 64) return launch_t<float, 64>(Qw, K, sh, tb, units_lse, units_col, lse, lse_nat, scores, st);
    return launch_t<float, 128>(Qw, K, sh, tb, units_lse, units_col, lse, lse_nat, scores, st);
  }
  if (sh.d == 64)
    return launch_t<__nv_bfloat16, 64>(Qw, K, sh, tb, units_lse, units_col, lse, lse_nat, scores, st);
  return launch_t<__nv_bfloat16, 128>(Qw, K, sh, tb, units_lse, units_col, lse, lse_nat, scores, st);
}

}  // namespace vc
