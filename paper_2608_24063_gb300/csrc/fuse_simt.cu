// Prune keys, fuse values, compact -- Algorithm 1 step 3.
//
// gather_k_kernel: K_out row = K row of the kept token (bit-exact 16-byte
//   vector copies, one thread per 16 bytes, coalesced within a row).
// fuse_v_simt_kernel: per (request, layer, KV head, tile of 32 kept rows)
//   O = softmax_row(V_k V_d^T / tau) V_d with an online (running max / sum)
//   softmax over tiles of 64 dropped rows, then V_out = mu V_k + (1-mu) O,
//   Eq. (redistribution) and Eq. (weight_fusion).  Empty drop set: V_out = V_k.
#include "vc_common.cuh"
#include "kernels.h"
#include "profile.h"

namespace vc {
namespace {

// ---------------------------------------------------------------------------
constexpr int kGatherThreads = 256;

__global__ void __launch_bounds__(kGatherThreads) gather_k_kernel(
    const uint4* __restrict__ K, Shape sh, Tables tb, const int32_t* __restrict__ keep_idx,
    uint4* __restrict__ K_out, int64_t total_rows, int chunks_per_row) {
  const int64_t t = (int64_t)blockIdx.x * kGatherThreads + threadIdx.x;
  const int64_t row = t / chunks_per_row;
  const int c = (int)(t % chunks_per_row);
  if (row >= total_rows) return;
  // (request, layer) block containing this output row
  const int rl = upper_index(tb.row0_out, sh.n_req * sh.L, row);
  const int r = rl / sh.L, l = rl % sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  const int64_t within = row - tb.row0_out[rl];
  const int g = (int)(within / ly.B);
  const int v = keep_idx[row];
  if (v < 0 || v >= rq.n) { set_status(tb.status, VC_ERR_DEVICE_INDEX); return; }
  const int64_t src_row = rq.kv_off / sh.d + ((int64_t)l * sh.Hkv + g) * rq.n + v;
  K_out[row * chunks_per_row + c] = K[src_row * chunks_per_row + c];
}

// ---------------------------------------------------------------------------
constexpr int kFuseThreads = 256;   // 8 warps x 4 kept rows
constexpr int kFuseRows = 32;
constexpr int kFuseKeys = 64;       // dropped rows per tile (2 per lane)

template <typename T, int D>
__global__ void __launch_bounds__(kFuseThreads) fuse_v_simt_kernel(
    const T* __restrict__ V, Shape sh, Tables tb, const int32_t* __restrict__ keep_idx,
    const int32_t* __restrict__ drop_idx, float mu, float inv_tau_log2, T* __restrict__ V_out) {
  extern __shared__ float4 smem4[];
  float* sm = reinterpret_cast<float*>(smem4);
  float (*vk)[D + 4] = reinterpret_cast<float (*)[D + 4]>(sm);
  float (*vd)[D + 1] = reinterpret_cast<float (*)[D + 1]>(sm + kFuseRows * (D + 4));
  float (*ps)[kFuseKeys + 1] =
      reinterpret_cast<float (*)[kFuseKeys + 1]>(sm + kFuseRows * (D + 4) + kFuseKeys * (D + 1));

  // unit -> (request, layer), then (KV head, row tile)
  const int rl = upper_index(tb.unit0_fuse, sh.n_req * sh.L, (int32_t)blockIdx.x);
  const int r = rl / sh.L, l = rl % sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  const int tiles = (ly.B + kFuseRows - 1) / kFuseRows;
  const int u = blockIdx.x - tb.unit0_fuse[rl];
  const int g = u / tiles;
  const int r0 = (u % tiles) * kFuseRows;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const T* Vl = V + rq.kv_off + ((int64_t)l * sh.Hkv + g) * rq.n * D;
  const int32_t* kp = keep_idx + rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B;
  const int32_t* dp = drop_idx + rq.drop_row0 + (int64_t)sh.Hkv * ly.Qd + (int64_t)g * ly.D;
  T* out = V_out + (rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B) * D;
  const int rows = min(kFuseRows, ly.B - r0);

  // kept rows
  for (int e = threadIdx.x; e < kFuseRows * (D / 4); e += kFuseThreads) {
    const int rr = e / (D / 4), c4 = (e % (D / 4)) * 4;
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (rr < rows) {
      const int v = kp[r0 + rr];
      if (v >= 0 && v < rq.n) x = load4(Vl + (int64_t)v * D + c4);
      else set_status(tb.status, VC_ERR_DEVICE_INDEX);
    }
    vk[rr][c4 + 0] = x.x; vk[rr][c4 + 1] = x.y; vk[rr][c4 + 2] = x.z; vk[rr][c4 + 3] = x.w;
  }

  constexpr int CPL = D / 32;   // output columns per lane
  float o[4][CPL];
  float m[4], zs[4];
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    m[a] = -INFINITY; zs[a] = 0.f;
#pragma unroll
    for (int c = 0; c < CPL; ++c) o[a][c] = 0.f;
  }

  for (int j0 = 0; j0 < ly.D; j0 += kFuseKeys) {
    __syncthreads();
    for (int e = threadIdx.x; e < kFuseKeys * (D / 4); e += kFuseThreads) {
      const int rr = e / (D / 4), c4 = (e % (D / 4)) * 4;
      float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
      if (j0 + rr < ly.D) {
        const int v = dp[j0 + rr];
        if (v >= 0 && v < rq.n) x = load4(Vl + (int64_t)v * D + c4);
        else set_status(tb.status, VC_ERR_DEVICE_INDEX);
      }
      vd[rr][c4 + 0] = x.x; vd[rr][c4 + 1] = x.y; vd[rr][c4 + 2] = x.z; vd[rr][c4 + 3] = x.w;
    }
    __syncthreads();
    // logits for 4 kept rows x 2 dropped rows
    float acc[4][2];
#pragma unroll
    for (int a = 0; a < 4; ++a) acc[a][0] = acc[a][1] = 0.f;
#pragma unroll 8
    for (int c = 0; c < D; ++c) {
      const float d0 = vd[lane][c], d1 = vd[lane + 32][c];
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float q = vk[4 * warp + a][c];
        acc[a][0] = fmaf(q, d0, acc[a][0]);
        acc[a][1] = fmaf(q, d1, acc[a][1]);
      }
    }
    const bool ok0 = j0 + lane < ly.D, ok1 = j0 + lane + 32 < ly.D;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const float x0 = ok0 ? acc[a][0] * inv_tau_log2 : -INFINITY;
      const float x1 = ok1 ? acc[a][1] * inv_tau_log2 : -INFINITY;
      float tm = fmaxf(x0, x1);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, off));
      const float mn = fmaxf(m[a], tm);          // finite: at least one valid key per tile
      const float corr = exp2f(m[a] - mn);
      const float p0 = exp2f(x0 - mn), p1 = exp2f(x1 - mn);
      float ts = p0 + p1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) ts += __shfl_xor_sync(0xffffffffu, ts, off);
      zs[a] = zs[a] * corr + ts;
      m[a] = mn;
#pragma unroll
      for (int c = 0; c < CPL; ++c) o[a][c] *= corr;
      ps[4 * warp + a][lane] = p0;
      ps[4 * warp + a][lane + 32] = p1;
    }
    __syncwarp();
    // O[row][col] += sum_k P[row][k] V_d[k][col]  (cols lane + 32 c); rows are warp-private
#pragma unroll 4
    for (int k = 0; k < kFuseKeys; ++k) {
      float dv[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) dv[c] = vd[k][lane + 32 * c];
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float p = ps[4 * warp + a][k];
#pragma unroll
        for (int c = 0; c < CPL; ++c) o[a][c] = fmaf(p, dv[c], o[a][c]);
      }
    }
  }
  __syncthreads();
  // epilogue: V_out = mu V_k + (1 - mu) O / Z   (V_k itself when the drop set is empty)
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int rr = 4 * warp + a;
    if (rr >= rows) continue;
    const float inv = ly.D > 0 ? 1.f / zs[a] : 0.f;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int col = lane + 32 * c;
      const float vkc = vk[rr][col];
      const float y = ly.D > 0 ? fmaf(mu, vkc, (1.f - mu) * (o[a][c] * inv)) : vkc;
      out[(int64_t)(r0 + rr) * D + col] = Elem<T>::from_f(y);
    }
  }
}

template <typename T, int D>
cudaError_t launch_fuse_t(const void* V, const Shape& sh, const Tables& tb,
                          const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                          void* V_out, int units, cudaStream_t st) {
  const size_t smem = sizeof(float) * (kFuseRows * (D + 4) + kFuseKeys * (D + 1) +
                                       kFuseRows * (kFuseKeys + 1));
  cudaError_t e = cudaFuncSetAttribute(fuse_v_simt_kernel<T, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  ProfileScope ps("fuse_v_simt", st);
  fuse_v_simt_kernel<T, D><<<units, kFuseThreads, smem, st>>>(
      static_cast<const T*>(V), sh, tb, keep_idx, drop_idx, mu, kLog2e / tau,
      static_cast<T*>(V_out));
  return cudaGetLastError();
}

}  // namespace

int fuse_rows_per_tile_simt() { return kFuseRows; }

cudaError_t launch_gather_k(int dtype, const void* K, const Shape& sh, const Tables& tb,
                            const int32_t* keep_idx, void* K_out, int64_t total_rows,
                            cudaStream_t st) {
  if (total_rows == 0) return cudaSuccess;
  const int64_t eb = dtype == VC_F32 ? 4 : 2;
  const int chunks = (int)(sh.d * eb / 16);
  const int64_t threads = total_rows * chunks;
  const int64_t blocks = (threads + kGatherThreads - 1) / kGatherThreads;
  ProfileScope ps("gather_k", st);
  gather_k_kernel<<<(unsigned)blocks, kGatherThreads, 0, st>>>(
      static_cast<const uint4*>(K), sh, tb, keep_idx, static_cast<uint4*>(K_out), total_rows,
      chunks);
  return cudaGetLastError();
}

cudaError_t launch_fuse_simt(int dtype, const void* V, const Shape& sh, const Tables& tb,
                             const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                             void* V_out, int units, cudaStream_t st) {
  if (units == 0) return cudaSuccess;
  if (dtype == VC_F32) {
    if (sh.d == 64) return launch_fuse_t<float, 64>(V, sh, tb, keep_idx, drop_idx, mu, tau, V_out, units, st);
    return launch_fuse_t<float, 128>(V, sh, tb, keep_idx, drop_idx, mu, tau, V_out, units, st);
  }
  if (sh.d == 64)
    return launch_fuse_t<__nv_bfloat16, 64>(V, sh, tb, keep_idx, drop_idx, mu, tau, V_out, units, st);
  return launch_fuse_t<__nv_bfloat16, 128>(V, sh, tb, keep_idx, drop_idx, mu, tau, V_out, units, st);
}

}  // namespace vc
