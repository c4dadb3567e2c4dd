// Key pruning and value fusion for bf16, d = 128; Eq. (redistribution) and
// Eq. (weight_fusion), Algorithm 1 step 3.
//
// gather_kv_kernel (HBM-bound copy): for every (request, layer, KV head) the
//   kept key rows go to K_out (bit-exact), and the survivors' value rows --
//   kept then dropped, each list in ascending position -- are compacted into a
//   dense workspace slab Vs, so the fusion can stream them with TMA.
// fuse_v_tc_kernel: one CTA per (request, layer, KV head, 256 kept rows):
//   O = softmax_row(V_k V_d^T / tau) V_d online over tiles of 128 dropped rows,
//   V_out = mu V_k + (1 - mu) O.
//   V_k and V_d tiles arrive by TMA (128-byte swizzle); S = V_k V_d^T and
//   O += P V_d run on tcgen05.mma with fp32 accumulators in tensor memory (V_d
//   read K-major for the first product, MN-major for the second), P goes
//   through shared memory in bf16.  The softmax keeps a per-row reference
//   maximum and rescales O in tensor memory only when a tile's maximum exceeds
//   it by more than 2^8.
//   Warp roles (320 threads, one CTA per SM): warps 0-3 and 4-7 own one kept
//   row each (= TMEM lane), warp 8 issues TMA and owns the tensor memory, one
//   thread of warp 9 issues the MMAs.  Every wait is bounded (tc_common.cuh).
#include <cudaTypedefs.h>

#include <mutex>

#include "kernels.h"
#include "profile.h"
#include "tc_common.cuh"
#include "vc_common.cuh"

namespace vc {
namespace {

using namespace tc;

// ---------------------------------------------------------------------------
// survivor gather

constexpr int kGatherThreads = 256;   // 16 rows x 16 chunks of 16 bytes
constexpr int kGatherRows = 16;

__global__ void __launch_bounds__(kGatherThreads) gather_kv_kernel(
    const uint4* __restrict__ K, const uint4* __restrict__ V, Shape sh, Tables tb,
    const int32_t* __restrict__ keep_idx, const int32_t* __restrict__ drop_idx,
    uint4* __restrict__ K_out, uint4* __restrict__ Vs) {
  const int rl = upper_index(tb.unit0_gather, sh.n_req * sh.L, (int32_t)blockIdx.x);
  const int r = rl / sh.L, l = rl % sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  const int nsurv = ly.B + ly.D;
  const int blocks = (nsurv + kGatherRows - 1) / kGatherRows;
  const int u = blockIdx.x - tb.unit0_gather[rl];
  const int g = u / blocks;
  const int i = (u % blocks) * kGatherRows + (threadIdx.x >> 4);
  const int c = threadIdx.x & 15;
  if (i >= nsurv) return;
  const int32_t v = i < ly.B ? keep_idx[rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + i]
                             : drop_idx[rq.drop_row0 + (int64_t)sh.Hkv * ly.Qd + (int64_t)g * ly.D + (i - ly.B)];
  if (v < 0 || v >= rq.n) {
    if (c == 0) set_status(tb.status, VC_ERR_DEVICE_INDEX);
    return;
  }
  const int64_t src = (rq.kv_off / 8) + (((int64_t)l * sh.Hkv + g) * rq.n + v) * 16 + c;
  Vs[(rq.vs_row0 + (int64_t)sh.Hkv * (ly.P + ly.Qd) + (int64_t)g * nsurv + i) * 16 + c] = V[src];
  if (i < ly.B) K_out[(rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + i) * 16 + c] = K[src];
}

// ---------------------------------------------------------------------------
// fusion

constexpr int kThreads = 320;
constexpr int kProducerWarp = 8, kMmaWarp = 9;
constexpr uint32_t kTile = 128;
constexpr uint32_t kKB = kTile * 128;            // one K-block: 128 rows x 128 bytes
constexpr uint32_t kTileBytes = 2 * kKB;
constexpr int kVdStages = 3;
constexpr uint32_t kTmemCols = 512;              // O_0, O_1, S_0, S_1: 128 columns each
constexpr float kRescaleLog2 = 8.f;

struct FSmem {
  uint8_t vk[2][2][kKB];              // [half][K-block] kept rows: A operand of S = V_k V_d^T
  uint8_t vd[kVdStages][2][kKB];      // dropped rows: B operand of both products
  uint8_t p[2][2][kKB];               // [half][K-block] numerators (bf16): A of O += P V_d
  uint64_t vk_full;
  uint64_t vd_full[kVdStages], vd_empty[kVdStages];
  uint64_t s_full[2], s_empty[2], p_full[2], p_empty[2];
  uint64_t o_full, mma_done;
  uint32_t tmem_base;
  int abort;
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

// Byte offset of 16-byte chunk c (0..15) of row r in a swizzled 128-row tile pair
// (the 128-byte swizzle TMA writes and the MMA descriptors expect).
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)((c >> 3) * kKB + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__global__ void __launch_bounds__(kThreads, 1)
fuse_v_tc_kernel(const __grid_constant__ CUtensorMap tmVs, Shape sh, Tables tb, float mu, float c2,
                 __nv_bfloat16* __restrict__ V_out) {
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
  // rows of this (layer, KV head) in Vs: B kept, then D dropped
  const int vs0 = (int)(rq.vs_row0 + (int64_t)sh.Hkv * (ly.P + ly.Qd) + (int64_t)g * (ly.B + D));
  const int64_t orow = rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + r0;

  if (threadIdx.x == 0) {
    mbar_init(&sm.vk_full, 1);
    for (int i = 0; i < kVdStages; ++i) { mbar_init(&sm.vd_full[i], 1); mbar_init(&sm.vd_empty[i], 1); }
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
  if (warp == kProducerWarp) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kProducerWarp) {
    if (lane == 0) {
      // ---- TMA producer: the kept rows once, then a ring of dropped-row tiles
      prefetch_tmap(&tmVs);
      mbar_arrive_expect_tx(&sm.vk_full, nhalf * kTileBytes);
      for (int h = 0; h < nhalf; ++h)
        for (int kb = 0; kb < 2; ++kb)
          tma_load_2d(sm.vk[h][kb], &tmVs, kb * 64, vs0 + r0 + h * (int)kTile, &sm.vk_full);
      int issued = 0;
      for (int j = 0; j < nt; ++j) {
        const int st = j % kVdStages;
        if (!mbar_wait(&sm.vd_empty[st], ((j / kVdStages) & 1) ^ 1, abort)) break;
        mbar_arrive_expect_tx(&sm.vd_full[st], kTileBytes);
        const int y = vs0 + ly.B + j * (int)kTile;
        tma_load_2d(sm.vd[st][0], &tmVs, 0, y, &sm.vd_full[st]);
        tma_load_2d(sm.vd[st][1], &tmVs, 64, y, &sm.vd_full[st]);
        ++issued;
      }
      drain_wait(&sm.vk_full, 0);
      for (int i = max(0, issued - kVdStages); i < issued; ++i)
        drain_wait(&sm.vd_full[i % kVdStages], (i / kVdStages) & 1);
    }
  } else if (warp == kMmaWarp) {
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
      uint32_t xs[8][16];                                 // S row of this thread (fp32 bits)
#pragma unroll
      for (int p = 0; p < 8; ++p) tmem_ld16(s_col + p * 16, xs[p]);
      tmem_wait_only();
#pragma unroll
      for (int p = 0; p < 8; ++p) reg_fence(xs[p]);
      tc_fence_before();
      mbar_arrive(&sm.s_empty[h]);                        // S copied out: the next product may start
      const int valid = min((int)kTile, D - j * (int)kTile);
      if (valid < (int)kTile) {                           // last tile: drop columns past D
#pragma unroll
        for (int p = 0; p < 8; ++p)
#pragma unroll
          for (int q = 0; q < 16; ++q)
            if (p * 16 + q >= valid) xs[p][q] = 0xff800000u;   // -inf
      }
      float pm[8];
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        float a = fmaxf(__uint_as_float(xs[p][0]), __uint_as_float(xs[p][1]));
#pragma unroll
        for (int q = 2; q < 16; q += 2) a = fmax3(a, __uint_as_float(xs[p][q]), __uint_as_float(xs[p][q + 1]));
        pm[p] = a;
      }
      const float tm = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])) * c2;
      // raise the reference maximum when this tile exceeds it by more than 2^8
      const bool raise = tm > m + kRescaleLog2;
      const float m_new = raise ? tm : m;
      const float corr = raise ? ex2(m - m_new) : 1.f;     // 0 on the first tile
      // the previous product must be done before P is rewritten (and before O is rescaled)
      if (!warp_wait(&sm.p_empty[h], (j & 1) ^ 1, abort)) { ok = false; break; }
      if (__any_sync(0xffffffffu, raise && j > 0)) {
        tc_fence_after();
#pragma unroll 1
        for (int p = 0; p < 8; ++p) {                    // rare: 16 columns at a time
          uint32_t v[16];
          tmem_ld16(o_col + p * 16, v);
          tmem_wait(v);
#pragma unroll
          for (int q = 0; q < 16; ++q) v[q] = __float_as_uint(__uint_as_float(v[q]) * corr);
          tmem_st16(o_col + p * 16, v);
        }
        tmem_wait_st();
      }
      lsum *= corr;
      m = m_new;
      // numerators in bf16 into the P tile (swizzled K-major A operand)
      uint8_t* pt = &sm.p[h][0][0];
      float2 ls = make_float2(0.f, 0.f);
      const float2 sc = make_float2(c2, c2), nm = make_float2(-m, -m);
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        float e[8];
#pragma unroll
        for (int q = 0; q < 8; q += 2) {
          const float2 t = __ffma2_rn(make_float2(__uint_as_float(xs[c >> 1][(c & 1) * 8 + q]),
                                                  __uint_as_float(xs[c >> 1][(c & 1) * 8 + q + 1])), sc, nm);
          e[q] = ex2(t.x);
          e[q + 1] = ex2(t.y);
          ls = __fadd2_rn(ls, make_float2(e[q], e[q + 1]));
        }
        uint4 w;
        w.x = pack_bf16x2(e[0], e[1]);
        w.y = pack_bf16x2(e[2], e[3]);
        w.z = pack_bf16x2(e[4], e[5]);
        w.w = pack_bf16x2(e[6], e[7]);
        *reinterpret_cast<uint4*>(pt + swz(row, c)) = w;
      }
      lsum += ls.x + ls.y;
      fence_proxy_async();
      tc_fence_before();
      mbar_arrive(&sm.p_full[h]);
    }
    // epilogue: V_out = mu V_k + (1 - mu) O / lsum, or V_k when nothing is dropped
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
        uint32_t v[4][16];
#pragma unroll
        for (int p = 0; p < 4; ++p) tmem_ld16(o_col + hh * 64 + p * 16, v[p]);
        tmem_wait_only();
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          reg_fence(v[p]);
#pragma unroll
          for (int q = 0; q < 16; ++q) o[p][q] = __uint_as_float(v[p][q]);
        }
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
  if (warp == kProducerWarp) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tbase, kTmemCols);
  }
  if (threadIdx.x == 0 && sm.abort) set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

bool make_rows_map(CUtensorMap* m, const void* base, uint64_t rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc || rows == 0 || rows > 0x7fffffffull) return false;
  cuuint64_t dims[2] = {128, rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, kTile};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int fuse_rows_per_tile_tc() { return 2 * (int)kTile; }
int gather_rows_per_block() { return kGatherRows; }

cudaError_t launch_fuse_tc(const void* K, const void* V, const Shape& sh, const Tables& tb,
                           const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                           void* K_out, void* V_out, void* Vs, int64_t vs_rows, int units_gather,
                           int units, cudaStream_t st) {
  if (units_gather == 0) return cudaSuccess;
  {
    ProfileScope ps("gather_kv", st);
    gather_kv_kernel<<<units_gather, kGatherThreads, 0, st>>>(
        static_cast<const uint4*>(K), static_cast<const uint4*>(V), sh, tb, keep_idx, drop_idx,
        static_cast<uint4*>(K_out), static_cast<uint4*>(Vs));
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  CUtensorMap mv;
  if (!make_rows_map(&mv, Vs, (uint64_t)vs_rows)) return cudaErrorInvalidValue;
  const size_t smem = sizeof(FSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(fuse_v_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  ProfileScope ps("fuse_v_tc", st);
  fuse_v_tc_kernel<<<units, kThreads, smem, st>>>(mv, sh, tb, mu, kLog2e / tau,
                                                  static_cast<__nv_bfloat16*>(V_out));
  return cudaGetLastError();
}

}  // namespace vc
