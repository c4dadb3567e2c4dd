// Key pruning and value fusion for bf16, d = 128; Eq. (redistribution) and
// Eq. (weight_fusion), Algorithm 1 step 3.
//
// gather_kv_kernel (HBM-bound copy): for every (request, layer, KV head) the
//   survivors' value rows -- kept then dropped, each list in ascending
//   position -- are compacted into a dense workspace slab Vs, so the fusion
//   can stream them with TMA; the kept key rows go to K_out (bit-exact) here
//   only when K is not in device memory (else the fusion copies them).
// fuse_v_tcp_kernel: persistent CTA pairs, each taking a share of the units
//   (request, layer, KV head, 256 kept rows) in turn:
//   O = softmax_row(V_k V_d^T / tau) V_d online over tiles of 128 dropped rows,
//   V_out = mu V_k + (1 - mu) O, on 2-SM tcgen05.mma with fp32 accumulators in
//   tensor memory; the numerators P go from the softmax warps to the second
//   product through tensor memory.  Warp roles (512 threads, one CTA per SM):
//   warps 0-7 softmax, warp 8 TMA and the tensor-memory allocation, one
//   thread of warp 9 (even CTA) the MMAs, warps 10-13 the epilogue, warps
//   14-15 the kept-key copy.  Every wait is bounded (tc_common.cuh).
#include <cudaTypedefs.h>

#include <algorithm>
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
// stores, so the dependent loads overlap.  keys = 0 leaves K_out to the
// fusion (it copies the kept keys while its products run).
__global__ void __launch_bounds__(kGatherThreads) gather_kv_kernel(
    const uint4* __restrict__ K, const uint4* __restrict__ V, Shape sh, Tables tb,
    const int32_t* __restrict__ keep_idx, const int32_t* __restrict__ drop_idx,
    uint4* __restrict__ K_out, uint4* __restrict__ Vs, int keys) {
  dep_wait();                        // the keep and drop lists
  if (threadIdx.x == 0) dep_launch();
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
      if (keys && i0 + 16 * k < ly.B) kv[k] = K[src];
    }
  }
#pragma unroll
  for (int k = 0; k < kGatherRowsPerThread; ++k) {
    const int i = i0 + 16 * k;
    if (v[k] >= 0) {
      Vs[(sbase + i) * 16 + c] = vv[k];
      if (keys && i < ly.B) K_out[(kbase + i) * 16 + c] = kv[k];
    }
  }
}

// ---------------------------------------------------------------------------
// shared helpers of the fusion




// Byte offset of 16-byte chunk c (0..7) of row r in a 128-byte-swizzled
// K-block (the layout TMA writes and the MMA descriptors expect).
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// ---------------------------------------------------------------------------
// persistent fusion: one CTA pair per TPC for the whole launch
//
// Organised so that nothing waits at a unit boundary.  The launch holds as many pairs as fit at once (one CTA per
// SM: 512 tensor-memory columns and ~214 KB of shared memory each); pair p
// takes the units p, p + P, p + 2P, ... of the list ordered longest first.
// Tensor memory per CTA: O[0] [0,128), O[1] [128,256) -- unit k accumulates
// in O[k % 2] -- and S[0] [256,384), S[1] [384,512) -- dropped tile t (counted
// over all of the pair's units) lands in S[t % 2], P(t) over the first half of
// each softmax warp's 64 columns.  Tiles hold 128 dropped rows (N = 128 for
// S, K = 128 for O: 16 MMAs and 2-3 commits per tile).  The issue order is
// S(t), O(t-1), so S(t) runs while the softmax works on tile t-1.
//
// Warps: 0-7 softmax (two per TMEM lane quadrant, 64 columns each), 8 the
// producer (lane 0 issues the TMA loads: the unit's kept rows into vk[k % 2],
// then its dropped tiles into a 3-stage ring; lane 1 tells the even CTA when
// this CTA's kept rows of each unit have landed), 9 the MMA issuer (even
// CTA), 10-13 the epilogue: once O[k % 2] is final it reads O, the row sums
// and V_k, writes mu V_k + (1 - mu) O / lsum in bf16 through a staging buffer,
// and frees O[k % 2] and vk[k % 2] -- while the MMAs and the softmax of unit
// k + 1 go on; 14-15 copy the CTA's kept keys of every unit into K_out.
//
// Every barrier completes once per unit (or per tile) and no waiter can fall
// two phases behind: the loader refills vk[b] only after the epilogue freed it,
// the MMA issuer overwrites O[b] (first O of a unit) only after the epilogue
// freed it, and the softmax writes a unit's row sums only after the epilogue
// read those of the unit two before.  A unit with no dropped rows still runs
// through every handshake (the issuer commits its O barrier without MMAs), so
// phases stay aligned with unit indices.  All waits are bounded.

namespace pf {

constexpr int kProducerWarp = 8, kMmaWarp = 9, kEpiWarp0 = 10, kEpiWarps = 4;
constexpr int kKeyWarp0 = kEpiWarp0 + kEpiWarps, kKeyWarps = 2;
constexpr int kThreads = 32 * (kKeyWarp0 + kKeyWarps);   // 512
constexpr uint32_t kTile = 128;                  // kept rows per CTA
constexpr uint32_t kKB = kTile * 128;            // 128 rows x 128 bytes
constexpr uint32_t kDTile = 128;                 // dropped rows per tile (both CTAs)
constexpr uint32_t kDHalf = kDTile / 2;          // dropped rows staged per CTA for S
constexpr uint32_t kDHalfKB = kDHalf * 128;      // 64 rows x 128 bytes
constexpr uint32_t kDKB = kDTile * 128;          // 128 rows x 128 bytes
constexpr int kStages = 3;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSCol = 256;
constexpr int kMaxUnits = 512;                   // units per pair (descriptor table)
// The softmax keeps a row's reference maximum m until a tile's maximum
// exceeds it by more than 2^32 (log2 units): until then P = 2^(x - m) stays
// below 2^32, which bf16 P, the fp32 row sums and the fp32 O hold without
// overflow, and only a larger rise rescales O.  Logits of 128-dimensional
// rows spread over tens of log2 units, so a small threshold rescaled O on
// most units' second tile.
constexpr float kRescaleLog2 = 32.f;

struct Unit {              // one unit as this CTA sees it
  int32_t vk_row;          // Vs row of this CTA's first kept row
  int32_t vd_row;          // Vs row of the (layer, KV head)'s first dropped row
  int32_t D;               // dropped rows
  int32_t rows;            // kept rows of this CTA (0..128)
  int64_t orow;            // K_out / V_out row (= keep-list position) of this CTA's first kept row
  int32_t kv_row;          // K row of the (layer, KV head)'s token 0
  int32_t n;               // tokens of the request
};

struct Smem {
  uint8_t vk[2][2][kKB];               // kept rows of unit k in vk[k % 2] [K-block]
  uint8_t vdo[kStages][kDKB];          // dropped tile: all 128 rows, this CTA's 64 columns (B of O)
  uint8_t vds[kStages][2][kDHalfKB];   // dropped tile: this CTA's 64 rows [K-block] (B of S)
  uint8_t stg[kTile * 256];            // epilogue staging, 128 rows x 256 bytes
  Unit unit[kMaxUnits];
  float xmax[2][4][2][32];             // [tile & 1][lane quadrant][column half][lane]
  float lsum[2][4][2][32];             // [unit & 1][lane quadrant][column half][lane]
  uint64_t vk_full[2];                 // own kept rows landed (1 arrival + bytes)
  uint64_t vk_pair[2];                 // even CTA: both CTAs' kept rows landed (2)
  uint64_t vk_empty[2];                // own: the epilogue read vk[b] (4 warps)
  uint64_t vd_full[kStages];           // even CTA: both CTAs' dropped tiles landed
  uint64_t vd_empty[kStages];          // both: the O product reading the stage is done
  uint64_t s_full[2];                  // both: S(t) in S[t % 2]
  uint64_t p_full[2];                  // even CTA: the 16 softmax warps wrote P(t)
  uint64_t o_full[2];                  // both: the unit's O[b] is final
  uint64_t o_empty[2];                 // even CTA: the 8 epilogue warps read O[b]
  uint64_t lsum_full[2];               // own: the 8 softmax warps wrote the unit's row sums
  uint64_t lsum_empty[2];              // own: the 4 epilogue warps read them
  uint64_t mma_done;                   // both: every MMA of the pair is done
  uint64_t never;                      // test support: never completes
  uint64_t peer_done;                  // even CTA: the odd CTA's fill count landed (8 bytes)
  int2 peer_fills;                     // even CTA: dropped tiles the odd CTA issued
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
fuse_v_tcp_kernel(const __grid_constant__ CUtensorMap tmRows128, const __grid_constant__ CUtensorMap tmRows64,
                  Shape sh, Tables tb, int units, int o_lo, int o_cnt, float mu, float c2,
                  __nv_bfloat16* __restrict__ V_out, int kcopy, const int32_t* __restrict__ keep_idx,
                  const uint4* __restrict__ K, uint4* __restrict__ K_out) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(align1024(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int pair = (int)(blockIdx.x >> 1), npairs = (int)(gridDim.x >> 1);
  // this launch covers positions [o_lo, o_lo + o_cnt) of the longest-first unit
  // order (position o is unit units-1-o), dealt to the pairs back and forth:
  // in round i pair p takes position i*P + p (i even) or i*P + P-1-p (i odd),
  // so every pair gets long and short units alike
  const int rounds = o_cnt / npairs, rem = o_cnt % npairs;
  const int nunits = min(kMaxUnits, rounds + ((rounds & 1) ? (pair >= npairs - rem) : (pair < rem)));

  // this pair's unit descriptors
  for (int i = threadIdx.x; i < nunits; i += kThreads) {
    const int pos = i * npairs + ((i & 1) ? npairs - 1 - pair : pair);
    const int unit = units - 1 - (o_lo + pos);
    const int rl = upper_index(tb.unit0_fuse_tc, sh.n_req * sh.L, (int32_t)unit);
    const Req rq = tb.req[rl / sh.L];
    const Layer ly = tb.layer[rl];
    const int ktiles = (ly.B + 2 * (int)kTile - 1) / (2 * (int)kTile);
    const int u = unit - tb.unit0_fuse_tc[rl];
    const int g = u / ktiles;
    const int r0 = (u % ktiles) * 2 * (int)kTile + (int)rank * (int)kTile;
    const int vs0 = (int)(rq.vs_row0 + (int64_t)sh.Hkv * (ly.P + ly.Qd) + (int64_t)g * (ly.B + ly.D));
    Unit d;
    d.vk_row = vs0 + r0;
    d.vd_row = vs0 + ly.B;
    d.D = ly.D;
    d.rows = max(0, min((int)kTile, ly.B - r0));
    d.orow = rq.out_row0 + (int64_t)sh.Hkv * ly.P + (int64_t)g * ly.B + r0;
    d.kv_row = (int)(rq.kv_off / 128 + ((int64_t)(rl % sh.L) * sh.Hkv + g) * rq.n);
    d.n = rq.n;
    sm.unit[i] = d;
  }
  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.vk_full[b], 1);
      mbar_init(&sm.vk_pair[b], 2);
      mbar_init(&sm.vk_empty[b], kEpiWarps);
      mbar_init(&sm.s_full[b], 1);
      mbar_init(&sm.p_full[b], 16);
      mbar_init(&sm.o_full[b], 1);
      mbar_init(&sm.o_empty[b], 2 * kEpiWarps);
      mbar_init(&sm.lsum_full[b], 8);
      mbar_init(&sm.lsum_empty[b], kEpiWarps);
    }
    for (int i = 0; i < kStages; ++i) { mbar_init(&sm.vd_full[i], 1); mbar_init(&sm.vd_empty[i], 1); }
    mbar_init(&sm.mma_done, 1);
    mbar_init(&sm.never, 1);
    mbar_init(&sm.peer_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    if (rank == 0) mbar_arrive_expect_tx(&sm.peer_done, 8);
  }
  if (warp == kProducerWarp) {
    tmem_alloc_pair(&sm.tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  __syncwarp();
  tc_fence_before();
  cluster_sync();                  // descriptors, barriers of both CTAs, TMEM
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kProducerWarp && lane == 0) {
    // ---- TMA loader (both CTAs)
    prefetch_tmap(&tmRows128);
    prefetch_tmap(&tmRows64);
    int t = 0, kl = 0;
    bool ok = true;
    // the survivor slab is the output of the kernel just before this one
    dep_wait();
    dep_launch();
    for (int k = 0; ok && k < nunits; ++k) {
      const Unit d = sm.unit[k];
      const int b = k & 1;
      if (!mbar_wait(&sm.vk_empty[b], ((k >> 1) & 1) ^ 1, abort)) break;
      mbar_arrive_expect_tx(&sm.vk_full[b], 2 * kKB);
      for (int kb = 0; kb < 2; ++kb) tma_load_2d(sm.vk[b][kb], &tmRows128, kb * 64, d.vk_row, &sm.vk_full[b]);
      ++kl;
      const int nt = (d.D + (int)kDTile - 1) / (int)kDTile;
      for (int j = 0; j < nt; ++j) {
        const int st = t % kStages;
        if (!mbar_wait(&sm.vd_empty[st], ((t / kStages) & 1) ^ 1, abort)) { ok = false; break; }
        if (rank == 0) mbar_arrive_expect_tx(&sm.vd_full[st], 2 * (2 * kDHalfKB + kDKB));
        const uint32_t full0 = map_to_rank(smem_u32(&sm.vd_full[st]), 0);
        const int y = d.vd_row + j * (int)kDTile;
        tma_load_2d_pair(sm.vds[st][0], &tmRows64, 0, y + (int)rank * (int)kDHalf, full0);
        tma_load_2d_pair(sm.vds[st][1], &tmRows64, 64, y + (int)rank * (int)kDHalf, full0);
        tma_load_2d_pair(sm.vdo[st], &tmRows128, (int)rank * 64, y, full0);
        ++t;
      }
    }
    // every copy this CTA started has landed before the pair may leave: the
    // kept rows on this CTA's barriers, the dropped tiles (both halves) on the
    // even CTA's, drained there with the odd CTA's count of them
    if (rank == 1) report_fills(&sm.peer_fills, &sm.peer_done, t, 0);
    for (int i = max(0, kl - 2); i < kl; ++i) drain_wait(&sm.vk_full[i & 1], (i >> 1) & 1);
    if (rank == 0) {
      const int2 f = peer_fills(&sm.peer_done, &sm.peer_fills, make_int2(t, 0), abort);
      drain_pair_ring(sm.vd_full, kStages, t, f.x, 2 * kDHalfKB + kDKB);
    }
  } else if (warp == kProducerWarp && lane == 1) {
    // ---- kept-rows relay: this CTA's kept rows of unit k landed -> even CTA
    const uint32_t pair0 = map_to_rank(smem_u32(&sm.vk_pair[0]), 0);
    const uint32_t pair1 = map_to_rank(smem_u32(&sm.vk_pair[1]), 0);
    for (int k = 0; k < nunits; ++k) {
      if (!mbar_wait(&sm.vk_full[k & 1], (k >> 1) & 1, abort)) break;
      mbar_arrive_cluster((k & 1) ? pair1 : pair0);
    }
  } else if (warp == kMmaWarp && lane == 0 && rank == 0) {
    // ---- MMA issuer (even CTA): S(t), then O(t-1)
    const uint32_t id_s = idesc_bf16_f32(2 * kTile, kDTile);
    const uint32_t id_o = idesc_bf16_f32_bmn(2 * kTile, kTile);
    struct Pend { int t, st, k, b; bool first, last; };
    Pend pv{0, 0, 0, 0, false, false};
    bool have = false, ok = true;
    // O(pv.t) += P(pv.t) V_d(pv.t); frees the stage, and finishes O[b] on a unit's last tile
    auto issue_o = [&](const Pend& q) -> bool {
      if (q.first && !mbar_wait(&sm.o_empty[q.b], ((q.k >> 1) & 1) ^ 1, abort)) return false;
      if (!mbar_wait(&sm.p_full[q.t & 1], (q.t >> 1) & 1, abort)) return false;
      tc_fence_after();
      const uint32_t p_tm = tbase + kSCol + (uint32_t)(q.t & 1) * kDTile;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        mma_bf16_pair_ta(tbase + (uint32_t)q.b * kTile, p_tm + (uint32_t)((kk >> 2) * 64 + (kk & 3) * 8),
                         desc_sw128_mn(smem_u32(sm.vdo[q.st]) + kk * 2048, kDKB), id_o,
                         (!q.first || kk > 0) ? 1u : 0u);
      mma_commit_pair(&sm.vd_empty[q.st], 3);
      if (q.last) mma_commit_pair(&sm.o_full[q.b], 3);
      return true;
    };
    int t = 0;
    for (int k = 0; ok && k < nunits; ++k) {
      const Unit d = sm.unit[k];
      const int b = k & 1;
      const int nt = (d.D + (int)kDTile - 1) / (int)kDTile;
      if (!mbar_wait(&sm.vk_pair[b], (k >> 1) & 1, abort)) { ok = false; break; }
      if (nt == 0) {
        // nothing dropped: V_out = V_k; keep the O[b] handshake in step
        if (have) { ok = issue_o(pv); have = false; if (!ok) break; }
        if (!mbar_wait(&sm.o_empty[b], ((k >> 1) & 1) ^ 1, abort)) { ok = false; break; }
        mma_commit_pair(&sm.o_full[b], 3);
        continue;
      }
      for (int j = 0; j < nt; ++j, ++t) {
        const int st = t % kStages;
        if (!mbar_wait(&sm.vd_full[st], (t / kStages) & 1, abort)) { ok = false; break; }
        tc_fence_after();
        const uint32_t s_tm = tbase + kSCol + (uint32_t)(t & 1) * kDTile;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_pair(s_tm, desc_sw128(smem_u32(sm.vk[b][kk >> 2]) + (kk & 3) * 32),
                        desc_sw128(smem_u32(sm.vds[st][kk >> 2]) + (kk & 3) * 32), id_s, kk ? 1u : 0u);
        mma_commit_pair(&sm.s_full[t & 1], 3);
        if (have && !issue_o(pv)) { ok = false; break; }
        pv = Pend{t, st, k, b, j == 0, j == nt - 1};
        have = true;
      }
    }
    if (ok && have) issue_o(pv);
    // always committed (also after a give-up), so every wait on it ends
    mma_commit_pair(&sm.mma_done, 3);
    drain_wait(&sm.mma_done, 0);
  } else if (warp == kMmaWarp && lane == 0) {
    // odd CTA: the pair's MMAs (and their arrivals on this CTA's barriers) are done
    drain_wait(&sm.mma_done, 0);
  } else if (warp < 8) {
    if ((sh.test_wait & VC_TEST_WAIT_FUSE) && warp == 0) {
      if (lane == 0 && injected_wait_gives_up(&sm.never)) {
        set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
        *abort = 1;
      }
      __syncwarp();
    }
    // ---- softmax over the drop set: one kept row per TMEM lane
    const int q4 = warp & 3, hf = warp >> 2;
    const uint32_t lane_off = (uint32_t)(q4 << 5) << 16;
    // After a give-up the warp stays in its loops without waiting, touching
    // tensor memory or arriving, but still meets its partner warp at every
    // named barrier (the partner may not have given up).
    int t = 0;
    bool ok = true;
    for (int k = 0; k < nunits; ++k) {
      const Unit d = sm.unit[k];
      const int b = k & 1;
      const int nt = (d.D + (int)kDTile - 1) / (int)kDTile;
      const uint32_t o_col = tbase + lane_off + (uint32_t)b * kTile + (uint32_t)hf * 64;
      float m = -INFINITY, lsum = 0.f;
      for (int j = 0; j < nt; ++j, ++t) {
        const int bsel = t & 1;
        ok = ok && warp_wait(&sm.s_full[bsel], (t >> 1) & 1, abort);
        if (!ok) {
          named_sync(1 + q4, 64);
          continue;
        }
        tc_fence_after();
        const uint32_t s_col = tbase + lane_off + kSCol + (uint32_t)bsel * kDTile + (uint32_t)hf * 64;
        float x[4][16];
        {
          uint32_t v[4][16];
#pragma unroll
          for (int p = 0; p < 4; ++p) tmem_ld16(s_col + p * 16, v[p]);
          tmem_wait_only();
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            reg_fence(v[p]);
#pragma unroll
            for (int q = 0; q < 16; ++q) x[p][q] = __uint_as_float(v[p][q]);
          }
        }
        const int valid = min(64, d.D - j * (int)kDTile - hf * 64);
        if (valid < 64) {                             // last tile: columns past D
#pragma unroll
          for (int p = 0; p < 4; ++p)
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (p * 16 + q >= valid) x[p][q] = -INFINITY;
        }
        float a[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          a[p] = fmaxf(x[p][0], x[p][1]);
#pragma unroll
          for (int q = 2; q < 16; q += 2) a[p] = fmax3(a[p], x[p][q], x[p][q + 1]);
        }
        sm.xmax[bsel][q4][hf][lane] = fmaxf(fmaxf(a[0], a[1]), fmaxf(a[2], a[3]));
        named_sync(1 + q4, 64);
        const float tm = fmaxf(sm.xmax[bsel][q4][0][lane], sm.xmax[bsel][q4][1][lane]) * c2;
        const bool raise = tm > m + kRescaleLog2;
        const float m_new = raise ? tm : m;
        const float corr = raise ? ex2(m - m_new) : 1.f;   // 0 on a unit's first tile
        lsum *= corr;
        m = m_new;
        const float2 sc = make_float2(c2, c2), nm = make_float2(-m, -m);
        float2 ls0 = make_float2(0.f, 0.f), ls1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t w[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int c = 32 * h + 2 * q;
            const float2 tt = __ffma2_rn(make_float2(x[c >> 4][c & 15], x[c >> 4][(c & 15) + 1]), sc, nm);
            const float2 e = make_float2(ex2(tt.x), ex2(tt.y));
            if (q & 1) ls1 = __fadd2_rn(ls1, e);
            else ls0 = __fadd2_rn(ls0, e);
            w[q] = pack_bf16x2(e.x, e.y);
          }
          tmem_st16(s_col + h * 16, w);
        }
        const float2 ls = __fadd2_rn(ls0, ls1);
        lsum += ls.x + ls.y;
        if (__any_sync(0xffffffffu, raise && j > 0)) {
          // rare: rescale this warp's 64 columns of O[b] once O(t-1) is done (its
          // commit frees stage (t-1) % kStages); O(t) waits for P(t), below
          const int tp = t - 1;
          ok = warp_wait(&sm.vd_empty[tp % kStages], (tp / kStages) & 1, abort);
          if (ok) {
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
        }
        tmem_wait_st();
        if (!ok) continue;
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(map_to_rank(smem_u32(&sm.p_full[bsel]), 0));
      }
      // the unit's row sums, once the epilogue has read those of unit k - 2
      ok = ok && warp_wait(&sm.lsum_empty[b], ((k >> 1) & 1) ^ 1, abort);
      if (!ok) continue;
      sm.lsum[b][q4][hf][lane] = lsum;
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.lsum_full[b]);
    }
  } else if (warp >= kKeyWarp0) {
    // ---- kept keys (kcopy): K_out rows of this CTA's kept rows of every unit,
    // K[token], copied while the pipeline runs.  Nothing waits for them and
    // they wait for nothing: K is an input and the keep list was written two
    // kernels back, so both are complete once this kernel is scheduled (they
    // start while the gather drains); each warp takes every other pair of
    // rows, a half-warp a 256-byte row.
    if (kcopy) {
      const int c = lane & 15;
      const int rsub = 2 * (warp - kKeyWarp0) + (lane >> 4);   // 0..3
      // batch q: rows 4 (16 (q % 2) + i) + rsub of unit q / 2's tile, i < 16;
      // the next batch's tokens load while this batch's rows are in flight
      auto load_tok = [&](int q, int (&tk)[16]) {
        const Unit& d = sm.unit[q >> 1];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int rr = 4 * (16 * (q & 1) + i) + rsub;
          tk[i] = rr < d.rows ? __ldg(keep_idx + d.orow + rr) : -1;
        }
      };
      int tok[16];
      if (nunits > 0) load_tok(0, tok);
#pragma unroll 1
      for (int q = 0; q < 2 * nunits; ++q) {
        const Unit d = sm.unit[q >> 1];
        const int h = q & 1;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int rr = 4 * (16 * h + i) + rsub;
          if (rr < d.rows && (tok[i] < 0 || tok[i] >= d.n)) {
            if (c == 0) set_status(tb.status, VC_ERR_DEVICE_INDEX);
            tok[i] = -1;
          }
        }
        const uint4* Kt = K + (int64_t)d.kv_row * 16 + c;
        uint4 kv[16];
        uint32_t have = 0;
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (tok[i] >= 0) {
            kv[i] = __ldg(Kt + (int64_t)tok[i] * 16);
            have |= 1u << i;
          }
        if (q + 1 < 2 * nunits) load_tok(q + 1, tok);
        uint4* Ko = K_out + d.orow * 16 + c;
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if ((have >> i) & 1u) Ko[(int64_t)(4 * (16 * h + i) + rsub) * 16] = kv[i];
      }
    }
  } else if (warp >= kEpiWarp0) {
    // ---- epilogue: V_out = mu V_k + (1 - mu) O / lsum (V_k when nothing is dropped)
    const int q4 = warp & 3;                          // TMEM lane quadrant of this warp
    const int row = (q4 << 5) + lane;
    const uint32_t lane_off = (uint32_t)(q4 << 5) << 16;
    const uint32_t o_empty0 = map_to_rank(smem_u32(&sm.o_empty[0]), 0);
    const uint32_t o_empty1 = map_to_rank(smem_u32(&sm.o_empty[1]), 0);
    const int te = (warp - kEpiWarp0) * 32 + lane;    // 0..127
    // After a give-up the warp keeps meeting the other epilogue warps at both
    // named barriers of every unit, and no warp copies a unit out once any of
    // them has given up.
    bool ok = true;
    for (int k = 0; k < nunits; ++k) {
      const Unit d = sm.unit[k];
      const int b = k & 1;
      const uint32_t ph = (k >> 1) & 1;
      ok = ok && warp_wait(&sm.vk_full[b], ph, abort) && warp_wait(&sm.lsum_full[b], ph, abort) &&
           warp_wait(&sm.o_full[b], ph, abort);
      if (ok) {
        tc_fence_after();
        const bool have_o = d.D > 0;
        const float lt = sm.lsum[b][q4][0][lane] + sm.lsum[b][q4][1][lane];
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.lsum_empty[b]);
        const float w_o = have_o ? (1.f - mu) / lt : 0.f;
        const float w_k = have_o ? mu : 1.f;
        const uint32_t o_col = tbase + lane_off + (uint32_t)b * kTile;
#pragma unroll 1
        for (int hh = 0; hh < 4; ++hh) {                // 32 output columns at a time
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
          const int kb = hh >> 1;
#pragma unroll
          for (int c4 = 0; c4 < 4; ++c4) {
            const int c8 = (hh & 1) * 4 + c4;             // 16-byte chunk within K-block kb
            const uint4 kv = *reinterpret_cast<const uint4*>(&sm.vk[b][kb][0] + swz(row, c8));
            const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kv);
            uint4 w;
            uint32_t* wp = &w.x;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float2 kf = __bfloat1622float2(k2[q]);
              const float a = fmaf(w_k, kf.x, w_o * o[c4 >> 1][(c4 & 1) * 8 + 2 * q]);
              const float bb = fmaf(w_k, kf.y, w_o * o[c4 >> 1][(c4 & 1) * 8 + 2 * q + 1]);
              wp[q] = pack_bf16x2(a, bb);
            }
            const int c = kb * 8 + c8;
            *reinterpret_cast<uint4*>(&sm.stg[0] + row * 256 + ((c ^ (row & 15)) << 4)) = w;
          }
        }
        // O[b] and vk[b] are read: free them
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive_cluster(b ? o_empty1 : o_empty0);
          mbar_arrive(&sm.vk_empty[b]);
        }
      }
      if (!named_sync_any(5, 32 * kEpiWarps, !ok)) {   // staging complete
#pragma unroll 4
        for (int i = 0; i < 16; ++i) {                // coalesced copy-out, 16 threads per row
          const int rr = i * 8 + (te >> 4), c = te & 15;
          if (rr < d.rows)
            *reinterpret_cast<uint4*>(V_out + (d.orow + rr) * 128 + c * 8) =
                *reinterpret_cast<const uint4*>(&sm.stg[0] + rr * 256 + ((c ^ (rr & 15)) << 4));
        }
      }
      named_sync(5, 32 * kEpiWarps);                 // staging free for the next unit
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

}  // namespace pf

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

int fuse_rows_per_tile_tc() { return 2 * (int)pf::kTile; }
int gather_rows_per_block() { return kGatherRows; }

// CTA pairs of the persistent fusion that fit on the device at once.
int fuse_tcp_pairs() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (cached[dev] > 0) return cached[dev];
  const size_t smem = sizeof(pf::Smem) + 1024;
  if (cudaFuncSetAttribute(pf::fuse_v_tcp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(pf::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, pf::fuse_v_tcp_kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    int sms = 2;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    n = std::max(1, sms / 2);
  }
  cached[dev] = n;
  return n;
}

cudaError_t launch_fuse_tc(const void* K, const void* V, const Shape& sh, const Tables& tb,
                           const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                           void* K_out, void* V_out, void* Vs, int64_t vs_rows, bool kcopy,
                           int units_gather, int units, cudaStream_t st) {
  if (units_gather == 0) return cudaSuccess;
  {
    ProfileScope ps(kcopy ? "gather_v" : "gather_kv", st);
    cudaError_t e = launch_dep(gather_kv_kernel, dim3(units_gather), dim3(kGatherThreads), 0, st,
                               static_cast<const uint4*>(K), static_cast<const uint4*>(V), sh, tb, keep_idx,
                               drop_idx, static_cast<uint4*>(K_out), static_cast<uint4*>(Vs), kcopy ? 0 : 1);
    if (e != cudaSuccess) return e;
  }
  if (units == 0) return cudaSuccess;
  CUtensorMap m128, m64;
  if (!make_rows_map(&m128, Vs, (uint64_t)vs_rows, pf::kTile) ||
      !make_rows_map(&m64, Vs, (uint64_t)vs_rows, pf::kDHalf))
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(pf::Smem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(pf::fuse_v_tcp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const int pairs = std::max(1, fuse_tcp_pairs());
  ProfileScope ps("fuse_v_tc", st);
  // one launch per slice of at most pairs * kMaxUnits units (one for every
  // workload here), each pair holding at most kMaxUnits descriptors
  const int64_t per_launch = (int64_t)pairs * pf::kMaxUnits;
  for (int64_t o = 0; o < units; o += per_launch) {
    const int cnt = (int)std::min<int64_t>(per_launch, units - o);
    const int p = std::min(pairs, cnt);
    e = launch_dep(pf::fuse_v_tcp_kernel, dim3(2 * p), dim3(pf::kThreads), smem, st, m128, m64, sh, tb, units,
                   (int)o, cnt, mu, kLog2e / tau, static_cast<__nv_bfloat16*>(V_out), kcopy ? 1 : 0, keep_idx,
                   static_cast<const uint4*>(K), static_cast<uint4*>(K_out));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace vc
