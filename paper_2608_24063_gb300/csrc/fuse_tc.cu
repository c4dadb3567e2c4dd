// Key pruning and value fusion for bf16, d = 128; Eq. (redistribution) and
// Eq. (weight_fusion), Algorithm 1 step 3.
//
// gather_kv_kernel (HBM-bound copy): for every (request, layer, KV head) the
//   kept key rows go to K_out (bit-exact), and the survivors' value rows --
//   kept then dropped, each list in ascending position -- are compacted into a
//   dense workspace slab Vs, so the fusion can stream them with TMA.
// fuse_v_tc_kernel: one CTA pair per (request, layer, KV head, 256 kept rows):
//   O = softmax_row(V_k V_d^T / tau) V_d online over tiles of 128 dropped rows,
//   V_out = mu V_k + (1 - mu) O, on 2-SM tcgen05.mma with fp32 accumulators in
//   tensor memory; the numerators P go from the softmax warps to the second
//   product through tensor memory.  Warp roles (320 threads, two CTAs per SM):
//   warps 0-7 softmax and epilogue, warp 8 TMA and the tensor-memory
//   allocation, one thread of warp 9 (even CTA) the MMAs.  Every wait is
//   bounded (tc_common.cuh).
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

constexpr int kGatherThreads = 256;   // 16 row slots x 16 chunks of 16 bytes
constexpr int kGatherRowsPerThread = 4;
constexpr int kGatherRows = 16 * kGatherRowsPerThread;   // rows per block

// Each thread copies its 16-byte chunk of four rows (i, i+16, i+32, i+48 of
// the block), all index loads and then all row loads in flight before the
// stores, so the dependent loads overlap.
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
  const int i0 = (u % blocks) * kGatherRows + (threadIdx.x >> 4);
  const int c = threadIdx.x & 15;
  const int64_t kbase = rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B;
  const int64_t dbase = rq.drop_row0 + (int64_t)sh.Hkv * ly.Qd + (int64_t)g * ly.D;
  const int64_t sbase = rq.vs_row0 + (int64_t)sh.Hkv * (ly.P + ly.Qd) + (int64_t)g * nsurv;
  const int64_t src0 = (rq.kv_off / 8) + ((int64_t)l * sh.Hkv + g) * rq.n * 16 + c;
  int32_t v[kGatherRowsPerThread];
#pragma unroll
  for (int k = 0; k < kGatherRowsPerThread; ++k) {
    const int i = i0 + 16 * k;
    v[k] = -1;
    if (i < nsurv) {
      const int32_t t = i < ly.B ? keep_idx[kbase + i] : drop_idx[dbase + (i - ly.B)];
      if (t >= 0 && t < rq.n) v[k] = t;
      else if (c == 0) set_status(tb.status, VC_ERR_DEVICE_INDEX);
    }
  }
  uint4 vv[kGatherRowsPerThread], kv[kGatherRowsPerThread];
#pragma unroll
  for (int k = 0; k < kGatherRowsPerThread; ++k) {
    if (v[k] >= 0) {
      const int64_t src = src0 + (int64_t)v[k] * 16;
      vv[k] = V[src];
      if (i0 + 16 * k < ly.B) kv[k] = K[src];
    }
  }
#pragma unroll
  for (int k = 0; k < kGatherRowsPerThread; ++k) {
    const int i = i0 + 16 * k;
    if (v[k] >= 0) {
      Vs[(sbase + i) * 16 + c] = vv[k];
      if (i < ly.B) K_out[(kbase + i) * 16 + c] = kv[k];
    }
  }
}

// ---------------------------------------------------------------------------
// fusion on CTA pairs
//
// A pair owns 256 kept rows of one (request, layer, KV head) (CTA r: rows
// r*128 ... r*128+127, one per TMEM lane) and streams the dropped rows in
// tiles of 64.  Per tile j the even CTA issues
//   S(j) = V_k V_d(j)^T  2-SM MMA, M = 256, N = 64 dropped rows (CTA r stages
//                        dropped rows r*32 ... r*32+31, K-major),
//   O += P(j) V_d(j)     2-SM MMA, M = 256, N = 128 value columns, K = 64 (CTA
//                        r stages columns r*64 ... of all 64 dropped rows,
//                        MN-major), A = P read from tensor memory,
// in the order S(0), S(1), [P(0)] O(0), S(2), [P(1)] O(1), ...: S is double
// buffered, so S(j+1) is computed while the softmax works on tile j.  P(j) is
// written in bf16 over the first half of each softmax warp's own S(j)
// columns; S(j+2) reuses the buffer only after O(j) (issued before it) has
// read P(j).  Two pairs run per TPC, so one pair's prologue and epilogue
// overlap the other's work.
//
// Tensor memory per CTA (256 columns): O in [0, 128), S/P buffer b in
// [128 + 64b, 192 + 64b).  Softmax: warps w and w+4 share the TMEM lanes of
// warp w % 4; warp w takes S columns 0-31 (dropped rows 0-31 of the tile), warp
// w+4 columns 32-63.  They agree on the row's reference maximum through shared
// memory each tile; the maximum is raised (and O rescaled in tensor memory,
// after O(j-1) is done) only when a tile exceeds it by more than 2^8.

constexpr int kThreads = 320;
constexpr int kProducerWarp = 8, kMmaWarp = 9;
constexpr uint32_t kTile = 128;                  // kept rows per CTA
constexpr uint32_t kKB = kTile * 128;            // 128 rows x 128 bytes
constexpr uint32_t kDTile = 64;                  // dropped rows per tile (both CTAs)
constexpr uint32_t kDHalfKB = 32 * 128;          // 32 rows x 128 bytes
constexpr uint32_t kDKB = kDTile * 128;          // 64 rows x 128 bytes
constexpr int kVdStages = 4;
constexpr uint32_t kTmemCols = 256;              // O: [0,128), S/P buffers: [128,192), [192,256)
constexpr uint32_t kSCol = 128;
constexpr float kRescaleLog2 = 8.f;

struct FSmem {
  uint8_t vk[2][kKB];                  // this CTA's 128 kept rows [K-block]: A of S = V_k V_d^T
  uint8_t vdo[kVdStages][kDKB];        // all 64 dropped rows, this CTA's 64 columns: B of O += P V_d
  uint8_t vds[kVdStages][2][kDHalfKB]; // this CTA's 32 dropped rows [stage][K-block]: B of S
  float xmax[2][4][2][32];             // [tile & 1][lane quadrant][column half][lane]: tile maxima
  float lsum[2][4][32];                // [column half][lane quadrant][lane]: partial row sums
  uint64_t vk_own;                     // this CTA's kept rows landed
  uint64_t vk_pair;                    // even CTA: both CTAs' kept rows landed (2 arrivals)
  uint64_t vd_full[kVdStages];         // even CTA: both CTAs' dropped tiles landed
  uint64_t vd_empty[kVdStages];        // both: the MMAs reading the stage are done
  uint64_t s_full[2];                  // both: S(j) is in S/P buffer j % 2
  uint64_t p_full[2];                  // even CTA: all 16 softmax warps wrote P(j), buffer j % 2
  uint64_t o_done;                     // both: O(j) is done (phase j)
  uint64_t mma_done;                   // both: every MMA of the pair is done (one phase)
  uint64_t never;                      // test support: never completes
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

// Byte offset of 16-byte chunk c (0..7) of row r in a 128-byte-swizzled
// K-block (the layout TMA writes and the MMA descriptors expect).
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 2)
fuse_v_tc_kernel(const __grid_constant__ CUtensorMap tmRows128, const __grid_constant__ CUtensorMap tmRows64,
                 const __grid_constant__ CUtensorMap tmRows32, Shape sh, Tables tb, float mu, float c2,
                 __nv_bfloat16* __restrict__ V_out) {
  extern __shared__ uint8_t smem_raw[];
  FSmem& sm = *reinterpret_cast<FSmem*>(align1024(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  // units in reverse order: later layers have fewer kept and more dropped
  // rows, so their units are the longest; starting them first leaves the
  // short units of the first layers to fill the last wave
  const int unit = (int)(gridDim.x >> 1) - 1 - (int)(blockIdx.x >> 1);

  const int rl = upper_index_warp(tb.unit0_fuse_tc, sh.n_req * sh.L, (int32_t)unit);
  const int r = rl / sh.L;
  const Req rq = tb.req[r];
  const Layer ly = tb.layer[rl];
  const int ktiles = (ly.B + 2 * (int)kTile - 1) / (2 * (int)kTile);
  const int u = unit - tb.unit0_fuse_tc[rl];
  const int g = u / ktiles;
  const int r0 = (u % ktiles) * 2 * (int)kTile + (int)rank * (int)kTile;   // this CTA's first kept row
  const int rows = max(0, min((int)kTile, ly.B - r0));                    // kept rows of this CTA
  const int D = ly.D;
  const int nt = (D + (int)kDTile - 1) / (int)kDTile;
  // rows of this (layer, KV head) in Vs: B kept, then D dropped
  const int vs0 = (int)(rq.vs_row0 + (int64_t)sh.Hkv * (ly.P + ly.Qd) + (int64_t)g * (ly.B + D));
  const int64_t orow = rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + r0;

  if (threadIdx.x == 0) {
    mbar_init(&sm.vk_own, 1);
    mbar_init(&sm.vk_pair, 2);
    for (int i = 0; i < kVdStages; ++i) { mbar_init(&sm.vd_full[i], 1); mbar_init(&sm.vd_empty[i], 1); }
    mbar_init(&sm.s_full[0], 1);
    mbar_init(&sm.s_full[1], 1);
    mbar_init(&sm.p_full[0], 16);
    mbar_init(&sm.p_full[1], 16);
    mbar_init(&sm.o_done, 1);
    mbar_init(&sm.mma_done, 1);
    mbar_init(&sm.never, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == kProducerWarp) {
    tmem_alloc_pair(&sm.tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  __syncwarp();
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kProducerWarp && lane == 0) {
    // ---- TMA producer (both CTAs)
    prefetch_tmap(&tmRows128);
    prefetch_tmap(&tmRows64);
    prefetch_tmap(&tmRows32);
    mbar_arrive_expect_tx(&sm.vk_own, 2 * kKB);
    for (int kb = 0; kb < 2; ++kb) tma_load_2d(sm.vk[kb], &tmRows128, kb * 64, vs0 + r0, &sm.vk_own);
    int issued = 0;
    for (int j = 0; j < nt; ++j) {
      if (j == kVdStages) {
        // the ring is full: own kept rows landed -> tell the even CTA, whose
        // MMAs read them (and must run before any stage frees up)
        if (!mbar_wait(&sm.vk_own, 0, abort)) break;
        mbar_arrive_cluster(map_to_rank(smem_u32(&sm.vk_pair), 0));
      }
      const int st = j % kVdStages;
      if (!mbar_wait(&sm.vd_empty[st], ((j / kVdStages) & 1) ^ 1, abort)) break;
      if (rank == 0) mbar_arrive_expect_tx(&sm.vd_full[st], 2 * (2 * kDHalfKB + kDKB));
      const uint32_t full0 = map_to_rank(smem_u32(&sm.vd_full[st]), 0);
      const int y = vs0 + ly.B + j * (int)kDTile;
      tma_load_2d_pair(sm.vds[st][0], &tmRows32, 0, y + (int)rank * 32, full0);
      tma_load_2d_pair(sm.vds[st][1], &tmRows32, 64, y + (int)rank * 32, full0);
      tma_load_2d_pair(sm.vdo[st], &tmRows64, (int)rank * 64, y, full0);
      ++issued;
    }
    if (nt <= kVdStages && mbar_wait(&sm.vk_own, 0, abort))
      mbar_arrive_cluster(map_to_rank(smem_u32(&sm.vk_pair), 0));
    if (rank == 0)
      for (int i = max(0, issued - kVdStages); i < issued; ++i)
        drain_wait(&sm.vd_full[i % kVdStages], (i / kVdStages) & 1);
  } else if (warp == kMmaWarp && lane == 0 && rank == 0 && nt > 0) {
    // ---- MMA issuer (even CTA): S(0), S(1), O(0), S(2), O(1), ...
    const uint32_t id_s = idesc_bf16_f32(2 * kTile, kDTile);
    const uint32_t id_o = idesc_bf16_f32_bmn(2 * kTile, kTile);
    bool ok = mbar_wait(&sm.vk_pair, 0, abort);
    for (int j = 0; ok && j <= nt; ++j) {
      if (j < nt) {
        // S(j) into buffer j % 2 (its previous user O(j-2) was issued before)
        const int st = j % kVdStages;
        if (!mbar_wait(&sm.vd_full[st], (j / kVdStages) & 1, abort)) break;
        tc_fence_after();
        const uint32_t s_tm = tbase + kSCol + (uint32_t)(j & 1) * kDTile;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_pair(s_tm, desc_sw128(smem_u32(sm.vk[kk >> 2]) + (kk & 3) * 32),
                        desc_sw128(smem_u32(sm.vds[st][kk >> 2]) + (kk & 3) * 32), id_s, kk ? 1u : 0u);
        mma_commit_pair(&sm.s_full[j & 1], 3);
      }
      if (j >= 1) {
        // O += P(j-1) V_d(j-1), once the softmax has written P(j-1)
        const int jp = j - 1, st = jp % kVdStages;
        if (!mbar_wait(&sm.p_full[jp & 1], (jp >> 1) & 1, abort)) break;
        tc_fence_after();
        const uint32_t p_tm = tbase + kSCol + (uint32_t)(jp & 1) * kDTile;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_bf16_pair_ta(tbase, p_tm + (uint32_t)((kk >> 1) * 32 + (kk & 1) * 8),
                           desc_sw128_mn(smem_u32(sm.vdo[st]) + kk * 2048, kDKB), id_o,
                           (jp > 0 || kk > 0) ? 1u : 0u);
        mma_commit_pair(&sm.vd_empty[st], 3);
        mma_commit_pair(&sm.o_done, 3);
      }
    }
    // always committed (also after a give-up), so the epilogue's wait ends
    mma_commit_pair(&sm.mma_done, 3);
    drain_wait(&sm.mma_done, 0);
  } else if (warp < 8) {
    if ((sh.test_wait & VC_TEST_WAIT_FUSE) && warp == 0) {
      if (lane == 0 && injected_wait_gives_up(&sm.never)) set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
      __syncwarp();
    }
    // ---- softmax over the drop set and epilogue: one kept row per TMEM lane
    const int q4 = warp & 3;                          // lane quadrant
    const int hf = warp >> 2;                         // column half
    const int row = (q4 << 5) + lane;                 // row within this CTA's 128
    const uint32_t lane_off = (uint32_t)(q4 << 5) << 16;
    const uint32_t o_col = tbase + lane_off + (uint32_t)hf * 64;
    float m = -INFINITY, lsum = 0.f;
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      const int bsel = j & 1;
      if (!warp_wait(&sm.s_full[bsel], (j >> 1) & 1, abort)) { ok = false; break; }
      tc_fence_after();
      // this warp's 32 columns of S(j)
      const uint32_t s_col = tbase + lane_off + kSCol + (uint32_t)bsel * kDTile + (uint32_t)hf * 32;
      float x[2][16];
      {
        uint32_t v[2][16];
#pragma unroll
        for (int p = 0; p < 2; ++p) tmem_ld16(s_col + p * 16, v[p]);
        tmem_wait_only();
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          reg_fence(v[p]);
#pragma unroll
          for (int q = 0; q < 16; ++q) x[p][q] = __uint_as_float(v[p][q]);
        }
      }
      const int valid = min(32, D - j * (int)kDTile - hf * 32);
      if (valid < 32) {                               // last tile: columns past D
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int q = 0; q < 16; ++q)
            if (p * 16 + q >= valid) x[p][q] = -INFINITY;
      }
      float a0 = fmaxf(x[0][0], x[0][1]), a1 = fmaxf(x[1][0], x[1][1]);
#pragma unroll
      for (int q = 2; q < 16; q += 2) {
        a0 = fmax3(a0, x[0][q], x[0][q + 1]);
        a1 = fmax3(a1, x[1][q], x[1][q + 1]);
      }
      // this row's tile maximum over both column halves
      sm.xmax[bsel][q4][hf][lane] = fmaxf(a0, a1);
      named_sync(1 + q4, 64);
      const float tm = fmaxf(sm.xmax[bsel][q4][0][lane], sm.xmax[bsel][q4][1][lane]) * c2;
      const bool raise = tm > m + kRescaleLog2;
      const float m_new = raise ? tm : m;
      const float corr = raise ? ex2(m - m_new) : 1.f;   // 0 on the first tile
      lsum *= corr;
      m = m_new;
      // P = exp2(S * c2 - m) in bf16 over the first 16 of this warp's S columns
      const float2 sc = make_float2(c2, c2), nm = make_float2(-m, -m);
      float2 ls = make_float2(0.f, 0.f);
      {
        uint32_t w[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int c = 2 * q;
          const float2 t = __ffma2_rn(make_float2(x[c >> 4][c & 15], x[c >> 4][(c & 15) + 1]), sc, nm);
          const float2 e = make_float2(ex2(t.x), ex2(t.y));
          ls = __fadd2_rn(ls, e);
          w[q] = pack_bf16x2(e.x, e.y);
        }
        tmem_st16(s_col, w);
      }
      lsum += ls.x + ls.y;
      if (__any_sync(0xffffffffu, raise && j > 0)) {
        // rare: rescale this warp's 64 columns of O in tensor memory once
        // O(j-1) is done (O(j) waits for P(j), so nothing else writes O).  The
        // parity wait is unambiguous: s_full(j) was committed after O(j-2), so
        // o_done is in phase j-1 or j here.
        if (!warp_wait(&sm.o_done, (j - 1) & 1, abort)) { ok = false; break; }
        tc_fence_after();
#pragma unroll 1
        for (int p = 0; p < 4; ++p) {
          uint32_t v[16];
          tmem_ld16(o_col + p * 16, v);
          tmem_wait(v);
#pragma unroll
          for (int q = 0; q < 16; ++q) v[q] = __float_as_uint(__uint_as_float(v[q]) * corr);
          tmem_st16(o_col + p * 16, v);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(map_to_rank(smem_u32(&sm.p_full[bsel]), 0));
    }
    // ---- epilogue: V_out = mu V_k + (1 - mu) O / lsum, or V_k when nothing is dropped
    sm.lsum[hf][q4][lane] = lsum;
    const bool have_k = warp_wait(&sm.vk_own, 0, abort);
    // O is final once every MMA of the pair is done.  (A parity wait on o_done
    // for O(nt-1) would be ambiguous here: s_full(nt-1) only guarantees O(nt-3),
    // and with O(nt-2) still running the barrier sits in a phase of the other
    // parity, which that wait would take as complete.)
    const bool have_o = have_k && ok && nt > 0 && warp_wait(&sm.mma_done, 0, abort);
    __syncwarp();
    named_sync(5, 256);
    const float lt = sm.lsum[0][q4][lane] + sm.lsum[1][q4][lane];   // same order in both halves
    if (have_o) tc_fence_after();
    const float w_o = have_o ? (1.f - mu) / lt : 0.f;
    const float w_k = have_o ? mu : 1.f;
    // stage the 128 x 128 output tile in the (now idle) dropped-row buffers
    // (vdo, 4 x 8 KB contiguous): row r at r * 256 bytes, 16-byte chunk c at
    // slot c ^ (r & 15)
    uint8_t* stage = &sm.vdo[0][0];
#pragma unroll 1
    for (int hh = 0; hh < 2; ++hh) {                  // 32 of this warp's 64 columns at a time
      float o[2][16];
      if (have_o) {
        uint32_t v[2][16];
#pragma unroll
        for (int p = 0; p < 2; ++p) tmem_ld16(o_col + hh * 32 + p * 16, v[p]);
        tmem_wait_only();
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          reg_fence(v[p]);
#pragma unroll
          for (int q = 0; q < 16; ++q) o[p][q] = __uint_as_float(v[p][q]);
        }
      } else {
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int q = 0; q < 16; ++q) o[p][q] = 0.f;
      }
      if (have_k) {
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) {
          const int c8 = hh * 4 + c4;                 // 16-byte chunk within the K-block
          const uint4 kv = *reinterpret_cast<const uint4*>(&sm.vk[hf][0] + swz(row, c8));
          const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kv);
          uint4 w;
          uint32_t* wp = &w.x;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 kf = __bfloat1622float2(k2[q]);
            const float a = fmaf(w_k, kf.x, w_o * o[c4 >> 1][(c4 & 1) * 8 + 2 * q]);
            const float b = fmaf(w_k, kf.y, w_o * o[c4 >> 1][(c4 & 1) * 8 + 2 * q + 1]);
            wp[q] = pack_bf16x2(a, b);
          }
          const int c = hf * 8 + c8;
          *reinterpret_cast<uint4*>(stage + row * 256 + ((c ^ (row & 15)) << 4)) = w;
        }
      }
    }
    named_sync(5, 256);
    // coalesced copy-out: 16 threads per 256-byte row
    const int t = threadIdx.x;                        // 0..255
    if (have_k) {
#pragma unroll 4
      for (int i = 0; i < 8; ++i) {
        const int rr = i * 16 + (t >> 4), c = t & 15;
        if (rr < rows)
          *reinterpret_cast<uint4*>(V_out + (orow + rr) * 128 + c * 8) =
              *reinterpret_cast<const uint4*>(stage + rr * 256 + ((c ^ (rr & 15)) << 4));
      }
    }
  }
  __syncwarp();
  tc_fence_before();
  cluster_sync();                  // no CTA leaves while the pair's MMAs or copies may touch it
  if (warp == kProducerWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tbase, kTmemCols);
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

// [rows][128] bf16 tensor, boxes of box_rows rows x 64 elements, 128-byte swizzle.
bool make_rows_map(CUtensorMap* m, const void* base, uint64_t rows, uint32_t box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc || rows == 0 || rows > 0x7fffffffull) return false;
  cuuint64_t dims[2] = {128, rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, box_rows};
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
  CUtensorMap m128, m64, m32;
  if (!make_rows_map(&m128, Vs, (uint64_t)vs_rows, kTile) || !make_rows_map(&m64, Vs, (uint64_t)vs_rows, 64) ||
      !make_rows_map(&m32, Vs, (uint64_t)vs_rows, 32))
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(FSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(fuse_v_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  ProfileScope ps("fuse_v_tc", st);
  fuse_v_tc_kernel<<<2 * units, kThreads, smem, st>>>(m128, m64, m32, sh, tb, mu, kLog2e / tau,
                                                      static_cast<__nv_bfloat16*>(V_out));
  return cudaGetLastError();
}

}  // namespace vc
