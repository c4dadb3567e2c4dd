// Key pruning and value fusion on the tcgen05 tensor cores, Eq. (redistribution)
// and Eq. (weight_fusion); bf16 inputs, d = 128.
//
// One CTA per (request, layer, KV head, tile of 256 kept rows):
//   K_out = K[keep]                                   (bit-exact row copy)
//   O     = softmax_row(V_k V_d^T / tau) V_d          (online over tiles of 128 dropped rows)
//   V_out = mu V_k + (1 - mu) O
// Kept and dropped value rows are gathered by index with cp.async into
// 128-byte swizzled tiles (the layout TMA would write).  S = V_k V_d^T and
// O += P V_d run on tcgen05.mma with fp32 accumulators in tensor memory; V_d
// is read K-major for the first product and MN-major for the second, P goes
// through shared memory in bf16.  The two halves of the kept tile (two
// consumer warpgroups) share every gathered V_d tile.  The softmax keeps a
// per-row reference maximum and rescales O (in tensor memory) only when a
// tile's maximum exceeds it by more than 2^8.
//
// Warp roles (384 threads, one CTA per SM): warps 0-3 and 4-7 own one kept
// row each (= TMEM lane) for the softmax and the epilogue, warps 8-10 gather
// rows and copy the kept keys, warp 11 allocates tensor memory and one of its
// threads issues the MMAs.  Every wait is bounded (see tc_common.cuh).
#include "kernels.h"
#include "profile.h"
#include "tc_common.cuh"
#include "vc_common.cuh"

namespace vc {
namespace {

using namespace tc;

constexpr int kThreads = 384;
constexpr int kProducers = 96;                   // warps 8-10
constexpr int kMmaWarp = 11;
constexpr uint32_t kTile = 128;
constexpr uint32_t kKB = kTile * 128;            // one K-block: 128 rows x 128 bytes
constexpr int kVdStages = 3;
constexpr int kKChunks = (2 * 128 * 16 + kProducers - 1) / kProducers;   // kept-row chunks per producer
constexpr uint32_t kTmemCols = 512;              // O_0, O_1, S_0, S_1: 128 columns each
constexpr float kRescaleLog2 = 8.f;

struct FSmem {
  uint8_t vk[2][2][kKB];              // [half][K-block] kept rows: A operand of S = V_k V_d^T
  uint8_t vd[kVdStages][2][kKB];      // dropped rows: B operand of both products
  uint8_t p[2][2][kKB];               // [half][K-block] numerators (bf16): A of O += P V_d
  int32_t idx_d[kVdStages][kTile];    // dropped positions of each stage
  uint64_t vk_full;
  uint64_t vd_full[kVdStages], vd_empty[kVdStages];
  uint64_t s_full[2], s_empty[2], p_full[2], p_empty[2];
  uint64_t o_full, mma_done;
  uint32_t tmem_base;
  int abort;
  int gather_go;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  const uint32_t a = smem_u32(p);
  return p + ((1024u - (a & 1023u)) & 1023u);
}

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  int dummy = 0;
  mbar_wait(bar, parity, &dummy);
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  const bool ok = mbar_wait(bar, parity, abort);
  return __all_sync(0xffffffffu, ok);
}

// Byte offset of 16-byte chunk c (0..15) of row r in a swizzled 128-row tile pair.
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)((c >> 3) * kKB + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// Position r of a list pos[0..count): -1 beyond count or outside [0, n)
// (the latter recorded in the status word).
__device__ __forceinline__ int32_t list_pos(const int32_t* pos, int count, int r, int n,
                                            int32_t* status) {
  if (r >= count) return -1;
  const int32_t v = pos[r];
  if (v < 0 || v >= n) {
    set_status(status, VC_ERR_DEVICE_INDEX);
    return -1;
  }
  return v;
}

// Gather the 128 rows listed in idx (shared memory, -1 = zeros) of a [n][128]
// bf16 slab into a swizzled tile pair; 16 consecutive threads copy one row.
__device__ __forceinline__ void gather_tile(uint8_t* dst, const __nv_bfloat16* slab,
                                            const int32_t* idx, int tid) {
  for (int e = tid; e < (int)kTile * 16; e += kProducers) {
    const int r = e >> 4, c = e & 15;
    const int32_t v = idx[r];
    cp_async16(dst + swz(r, c), v >= 0 ? slab + (int64_t)v * 128 + c * 8 : slab, v >= 0 ? 16u : 0u);
  }
}

// K_out rows of the tile: bit-exact 16-byte copies of the kept key rows.
// Producer thread tid owns chunks e = tid + kProducers * i of the 256-row tile,
// whose row positions it holds in kpos[i] (-1 = no row).
__device__ __forceinline__ void copy_keys(__nv_bfloat16* K_out, int64_t orow,
                                          const __nv_bfloat16* Kl, const int32_t (&kpos)[kKChunks],
                                          int tid) {
#pragma unroll
  for (int i = 0; i < kKChunks; ++i) {
    const int e = tid + kProducers * i;
    if (kpos[i] >= 0)
      reinterpret_cast<uint4*>(K_out + (orow + (e >> 4)) * 128)[e & 15] =
          reinterpret_cast<const uint4*>(Kl + (int64_t)kpos[i] * 128)[e & 15];
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// 64 consecutive TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_cols64(uint32_t taddr, float (&x)[4][16]) {
  uint32_t v[4][16];
#pragma unroll
  for (int p = 0; p < 4; ++p) tmem_ld16(taddr + p * 16, v[p]);
  tmem_wait_only();
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    reg_fence(v[p]);
#pragma unroll
    for (int q = 0; q < 16; ++q) x[p][q] = __uint_as_float(v[p][q]);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
fuse_v_tc_kernel(const __nv_bfloat16* __restrict__ K, const __nv_bfloat16* __restrict__ V,
                 Shape sh, Tables tb, const int32_t* __restrict__ keep_idx,
                 const int32_t* __restrict__ drop_idx, float mu, float c2,
                 __nv_bfloat16* __restrict__ K_out, __nv_bfloat16* __restrict__ V_out) {
  extern __shared__ uint8_t smem_raw[];
  FSmem& sm = *reinterpret_cast<FSmem*>(align1024(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int rl = upper_index(tb.unit0_fuse_tc, sh.n_req * sh.L, (int32_t)blockIdx.x);
  const int r = rl / sh.L, l = rl % sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  const int ktiles = (ly.B + 2 * (int)kTile - 1) / (2 * (int)kTile);
  const int u = blockIdx.x - tb.unit0_fuse_tc[rl];
  const int g = u / ktiles;
  const int r0 = (u % ktiles) * 2 * (int)kTile;
  const int rows = min(2 * (int)kTile, ly.B - r0);        // kept rows of this CTA
  const int nhalf = rows > (int)kTile ? 2 : 1;            // halves with kept rows
  const int D = ly.D;
  const int nt = (D + (int)kTile - 1) / (int)kTile;

  const int64_t slab = ((int64_t)l * sh.Hkv + g) * rq.n * 128;
  const __nv_bfloat16* Vl = V + rq.kv_off + slab;
  const __nv_bfloat16* Kl = K + rq.kv_off + slab;
  const int64_t orow = rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + r0;
  const int32_t* kp = keep_idx + orow;
  const int32_t* dp = drop_idx + rq.drop_row0 + (int64_t)sh.Hkv * ly.Qd + (int64_t)g * D;

  if (threadIdx.x == 0) {
    mbar_init(&sm.vk_full, kProducers);
    for (int i = 0; i < kVdStages; ++i) { mbar_init(&sm.vd_full[i], kProducers); mbar_init(&sm.vd_empty[i], 1); }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.s_full[i], 1);
      mbar_init(&sm.s_empty[i], kTile);
      mbar_init(&sm.p_full[i], kTile);
      mbar_init(&sm.p_empty[i], 1);
    }
    mbar_init(&sm.o_full, 1);
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kMmaWarp) {
    if (lane == 0) {
      // ---- MMA issuer.  Per drop tile j: S_h = V_k,h V_d(j)^T for both halves,
      // then O_h += P_h(j-1) V_d(j-1) for both halves.
      const uint32_t id_s = idesc_bf16_f32(kTile, kTile);
      const uint32_t id_o = idesc_bf16_f32_bmn(kTile, kTile);
      bool ok = mbar_wait(&sm.vk_full, 0, abort);
      for (int j = 0; ok && j <= nt; ++j) {
        if (j < nt) {
          const int st = j % kVdStages;
          if (!mbar_wait(&sm.vd_full[st], (j / kVdStages) & 1, abort)) break;
          for (int h = 0; h < nhalf && ok; ++h) {
            if (!mbar_wait(&sm.s_empty[h], (j & 1) ^ 1, abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d = tbase + (uint32_t)(2 + h) * kTile;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              mma_bf16(d, desc_sw128(smem_u32(sm.vk[h][kk >> 2]) + (kk & 3) * 32),
                       desc_sw128(smem_u32(sm.vd[st][kk >> 2]) + (kk & 3) * 32), id_s, kk ? 1u : 0u);
            mma_commit(&sm.s_full[h]);
          }
          if (!ok) break;
        }
        if (j >= 1) {
          const int jp = j - 1, st = jp % kVdStages;
          for (int h = 0; h < nhalf && ok; ++h) {
            if (!mbar_wait(&sm.p_full[h], jp & 1, abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d = tbase + (uint32_t)h * kTile;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              mma_bf16(d, desc_sw128(smem_u32(sm.p[h][kk >> 2]) + (kk & 3) * 32),
                       desc_sw128_mn(smem_u32(sm.vd[st][0]) + kk * 2048, kKB), id_o,
                       (jp > 0 || kk > 0) ? 1u : 0u);
            mma_commit(&sm.p_empty[h]);
          }
          if (ok) mma_commit(&sm.vd_empty[st]);
        }
      }
      mma_commit(&sm.o_full);
      mma_commit(&sm.mma_done);
      drain_wait(&sm.mma_done, 0);
    }
  } else if (warp >= 8) {
    // ---- row gathers (cp.async) and the key copy.  Positions go to shared
    // memory first (the next tile's fetched one tile ahead) so the copies issue
    // back to back; a stage is published once its copies landed.
    const int tid = threadIdx.x - 256;
    int32_t kpos[kKChunks];                      // positions of this thread's kept-row chunks
#pragma unroll
    for (int i = 0; i < kKChunks; ++i) {
      const int e = tid + kProducers * i;
      kpos[i] = e < 2 * (int)kTile * 16 ? list_pos(kp, rows, e >> 4, rq.n, tb.status) : -1;
    }
#pragma unroll
    for (int i = 0; i < kKChunks; ++i) {
      const int e = tid + kProducers * i;
      if (e < 2 * (int)kTile * 16) {
        const int rr = e >> 4, c = e & 15;
        cp_async16(&sm.vk[rr >> 7][0][0] + swz(rr & 127, c), kpos[i] >= 0 ? Vl + (int64_t)kpos[i] * 128 + c * 8 : Vl,
                   kpos[i] >= 0 ? 16u : 0u);
      }
    }
    cp_async_commit();
    cp_async_wait<0>();
    fence_proxy_async();
    mbar_arrive(&sm.vk_full);
    int32_t a0 = -1, a1 = -1;
    if (nt > 0) {
      const int cnt = min((int)kTile, D);
      a0 = list_pos(dp, cnt, tid, rq.n, tb.status);
      a1 = tid + kProducers < (int)kTile ? list_pos(dp, cnt, tid + kProducers, rq.n, tb.status) : -1;
    }
    bool keys_done = false;
    int j = 0;
    for (; j < nt; ++j) {
      const int st = j % kVdStages;
      int32_t* buf = sm.idx_d[st];
      if (tid == 0) sm.gather_go = mbar_wait(&sm.vd_empty[st], ((j / kVdStages) & 1) ^ 1, abort) ? 1 : 0;
      named_sync(1, kProducers);                 // the stage is free and its old positions unread
      if (!sm.gather_go) break;
      buf[tid] = a0;
      if (tid + kProducers < (int)kTile) buf[tid + kProducers] = a1;
      named_sync(1, kProducers);
      if (j + 1 < nt) {
        const int32_t* nxt = dp + (j + 1) * (int)kTile;
        const int cnt = min((int)kTile, D - (j + 1) * (int)kTile);
        a0 = list_pos(nxt, cnt, tid, rq.n, tb.status);
        a1 = tid + kProducers < (int)kTile ? list_pos(nxt, cnt, tid + kProducers, rq.n, tb.status) : -1;
      }
      gather_tile(&sm.vd[st][0][0], Vl, buf, tid);
      cp_async_commit();
      if (j >= 1) {
        cp_async_wait<1>();
        fence_proxy_async();
        mbar_arrive(&sm.vd_full[(j - 1) % kVdStages]);
        if (!keys_done) {                        // while the first products run
          copy_keys(K_out, orow, Kl, kpos, tid);
          keys_done = true;
        }
      }
    }
    cp_async_wait<0>();
    fence_proxy_async();
    if (j >= 1) mbar_arrive(&sm.vd_full[(j - 1) % kVdStages]);
    if (!keys_done) copy_keys(K_out, orow, Kl, kpos, tid);
  } else {
    // ---- softmax over the drop set and epilogue: one thread per kept row
    const int h = warp >> 2;                              // half of the kept tile
    const int row = ((warp & 3) << 5) + lane;             // row within the half = TMEM lane
    const uint32_t lane_off = (uint32_t)((warp & 3) << 5) << 16;
    const uint32_t o_col = tbase + lane_off + (uint32_t)h * kTile;
    const uint32_t s_col = tbase + lane_off + (uint32_t)(2 + h) * kTile;
    const bool active = h < nhalf;
    float m = -INFINITY, lsum = 0.f;
    bool ok = true;
    for (int j = 0; active && j < nt; ++j) {
      if (!warp_wait(&sm.s_full[h], j & 1, abort)) { ok = false; break; }
      tc_fence_after();
      const int valid = min((int)kTile, D - j * (int)kTile);
      // pass A over S: the tile maximum
      float tm = -INFINITY;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        float x[4][16];
        tmem_cols64(s_col + hh * 64, x);
        float pm[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          float a = -INFINITY;
#pragma unroll
          for (int q = 0; q < 16; ++q)
            if (hh * 64 + p * 16 + q < valid) a = fmaxf(a, x[p][q]);
          pm[p] = a;
        }
        tm = fmax3(tm, fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3]));
      }
      tm *= c2;
      // raise the reference maximum when this tile exceeds it by more than 2^8
      const bool raise = tm > m + kRescaleLog2;
      const float m_new = raise ? tm : m;
      const float corr = raise ? ex2(m - m_new) : 1.f;     // 0 on the first tile
      if (__any_sync(0xffffffffu, raise && j > 0)) {
        // O holds the tiles before j: wait for their last product, then rescale in place
        if (!warp_wait(&sm.p_empty[h], (j - 1) & 1, abort)) { ok = false; break; }
        tc_fence_after();
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t v[4][16];
#pragma unroll
          for (int p = 0; p < 4; ++p) tmem_ld16(o_col + hh * 64 + p * 16, v[p]);
          tmem_wait_only();
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            reg_fence(v[p]);
#pragma unroll
            for (int q = 0; q < 16; ++q) v[p][q] = __float_as_uint(__uint_as_float(v[p][q]) * corr);
            tmem_st16(o_col + hh * 64 + p * 16, v[p]);
          }
        }
        tmem_wait_st();
      }
      lsum *= corr;
      m = m_new;
      // the P tile is free once the previous product has read it
      if (!warp_wait(&sm.p_empty[h], (j & 1) ^ 1, abort)) { ok = false; break; }
      // pass B over S: numerators in bf16 into the P tile (swizzled K-major A operand)
      uint8_t* pt = &sm.p[h][0][0];
      float2 ls = make_float2(0.f, 0.f);
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        float x[4][16];
        tmem_cols64(s_col + hh * 64, x);
        if (hh == 1) {
          tc_fence_before();
          mbar_arrive(&sm.s_empty[h]);             // S copied out: the next product may start
        }
#pragma unroll
        for (int p = 0; p < 4; ++p) {
#pragma unroll
          for (int c8 = 0; c8 < 2; ++c8) {
            float e[8];
#pragma unroll
            for (int q = 0; q < 8; q += 2) {
              const int col = hh * 64 + p * 16 + c8 * 8 + q;
              const float2 t = __ffma2_rn(make_float2(x[p][c8 * 8 + q], x[p][c8 * 8 + q + 1]),
                                          make_float2(c2, c2), make_float2(-m, -m));
              e[q] = col < valid ? ex2(t.x) : 0.f;
              e[q + 1] = col + 1 < valid ? ex2(t.y) : 0.f;
              ls = __fadd2_rn(ls, make_float2(e[q], e[q + 1]));
            }
            uint4 w;
            w.x = pack_bf16x2(e[0], e[1]);
            w.y = pack_bf16x2(e[2], e[3]);
            w.z = pack_bf16x2(e[4], e[5]);
            w.w = pack_bf16x2(e[6], e[7]);
            *reinterpret_cast<uint4*>(pt + swz(row, hh * 8 + p * 2 + c8)) = w;
          }
        }
      }
      lsum += ls.x + ls.y;
      fence_proxy_async();
      tc_fence_before();
      mbar_arrive(&sm.p_full[h]);
    }
    // epilogue: V_out = mu V_k + (1 - mu) O / lsum, or V_k when nothing is dropped;
    // the kept rows are read from shared memory once their gather has landed
    const bool have_k = warp_wait(&sm.vk_full, 0, abort);
    const bool have_o = active && have_k && ok && nt > 0 && warp_wait(&sm.o_full, 0, abort);
    if (have_o) tc_fence_after();
    const float w_o = have_o ? (1.f - mu) / lsum : 0.f;
    const float w_k = have_o ? mu : 1.f;
    const int grow = h * (int)kTile + row;                // row within the CTA's kept tile
#pragma unroll 1
    for (int hh = 0; hh < 2; ++hh) {
      float o[4][16];
      if (have_o) {
        tmem_cols64(o_col + hh * 64, o);
      } else {
#pragma unroll
        for (int p = 0; p < 4; ++p)
#pragma unroll
          for (int q = 0; q < 16; ++q) o[p][q] = 0.f;
      }
      if (have_k && grow < rows) {
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) {
          const int c = hh * 8 + c8;
          const uint4 kv = *reinterpret_cast<const uint4*>(&sm.vk[h][0][0] + swz(row, c));
          const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kv);
          uint4 w;
          uint32_t* wp = &w.x;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 kf = __bfloat1622float2(k2[q]);
            const float a = fmaf(w_k, kf.x, w_o * o[c8 >> 1][(c8 & 1) * 8 + 2 * q]);
            const float b = fmaf(w_k, kf.y, w_o * o[c8 >> 1][(c8 & 1) * 8 + 2 * q + 1]);
            wp[q] = pack_bf16x2(a, b);
          }
          *reinterpret_cast<uint4*>(V_out + (orow + grow) * 128 + c * 8) = w;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tbase, kTmemCols);
  }
  if (threadIdx.x == 0 && sm.abort) set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
}

}  // namespace

int fuse_rows_per_tile_tc() { return 2 * (int)kTile; }

cudaError_t launch_fuse_tc(const void* K, const void* V, const Shape& sh, const Tables& tb,
                           const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                           void* K_out, void* V_out, int units, cudaStream_t st) {
  if (units == 0) return cudaSuccess;
  const size_t smem = sizeof(FSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(fuse_v_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  ProfileScope ps("fuse_kv_tc", st);
  fuse_v_tc_kernel<<<units, kThreads, smem, st>>>(
      static_cast<const __nv_bfloat16*>(K), static_cast<const __nv_bfloat16*>(V), sh, tb, keep_idx,
      drop_idx, mu, kLog2e / tau, static_cast<__nv_bfloat16*>(K_out),
      static_cast<__nv_bfloat16*>(V_out));
  return cudaGetLastError();
}

}  // namespace vc
