// Token scoring on the tcgen05 tensor cores, Eq. (token_score); bf16 inputs, d = 128.
//
// Per (request, layer, KV head) the G*W window rows (contiguous in Qw) meet
// the n visual keys (contiguous in K).  Logits come from tcgen05.mma (bf16 x
// bf16 -> fp32 in tensor memory), operands staged by TMA with 128-byte
// swizzling.  The exact softmax column sum needs every row's normaliser
// first, so the score takes two passes over the logits:
//
//   pass 1 (score_lse_tc)    CTA pairs, rows in TMEM lanes: per row, running
//                            max and compensated sum of exp2 over a range of
//                            256-key tiles -> partial (m, z) per key split;
//   merge  (lse_merge)       -lse2 = -(m + log2 z) over the splits (or minus
//                            the caller's natural-log normaliser * log2 e),
//                            written per (layer, KV head) padded with -inf to
//                            whole pass-2 chunks; with a single key split
//                            pass 1 writes these values itself and the merge
//                            is skipped;
//   pass 2 (score_colsum_tc) CTA pairs, keys in TMEM lanes: each thread owns
//                            one key and sums exp2(x*scale*log2e - lse2[row])
//                            over all rows of all layers (compensated),
//                            s = sum / L.  Each 256-row chunk's normalisers
//                            arrive beside its Q rows (one bulk copy per
//                            CTA), padding rows contribute 0.
//
// Warp roles in both passes (320 threads, one CTA per SM): warps 0-3 and 4-7
// are two consumer warpgroups (one TMEM lane per thread), warp 8 issues TMA and
// owns the tensor-memory allocation, one thread of warp 9 issues the MMAs (in
// both passes only the even CTA of each pair issues them, as 2-SM MMAs of
// M = N = 256, 128 cycles each, so the issuing thread's barrier waits and
// commits hide behind the tensor pipe).
// Each consumer thread takes a whole tile (up to 128 accumulators) per step,
// so its exps and sums form many independent chains.  Every wait is bounded: on a
// timeout the CTA stops issuing, waits for its own copies and MMAs, frees its
// tensor memory and records VC_ERR_DEVICE_TIMEOUT.
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

constexpr int kThreads = 320;
constexpr int kProducerWarp = 8, kMmaWarp = 9;
constexpr uint32_t kTile = 128;                 // keys per tile, rows per block / chunk
constexpr uint32_t kKBlockBytes = kTile * 128;  // 128 rows x 64 bf16
constexpr uint32_t kTileBytes = 2 * kKBlockBytes;
constexpr uint32_t kTmemCols = 512;




// sum_j exp2(x_j * s + b_j) over 16 values, with packed fp32x2 FMA and adds
// (pairwise, so the rounding error stays a few ulp).
__device__ __forceinline__ float exp2_sum16(const float (&x)[16], float2 s, const float2 (&b)[8]) {
  float2 e[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const float2 t = __ffma2_rn(make_float2(x[2 * j], x[2 * j + 1]), s, b[j]);
    e[j] = make_float2(ex2(t.x), ex2(t.y));
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) e[j] = __fadd2_rn(e[2 * j], e[2 * j + 1]);
  e[0] = __fadd2_rn(e[0], e[1]);
  e[2] = __fadd2_rn(e[2], e[3]);
  e[0] = __fadd2_rn(e[0], e[2]);
  return e[0].x + e[0].y;
}

// ---------------------------------------------------------------------------
// pass 1 on CTA pairs
//
// A pair covers 256 window rows (128 per CTA, rows in TMEM lanes) and walks
// its key range in tiles of 256 keys: each CTA loads its 128 query rows once
// and, per tile, its own 128 keys (CTA r: keys r*128 ... r*128+127 of the
// tile); one 2-SM MMA chain (M = 256, N = 256, K = 128) leaves every row's 256
// logits in its own CTA's tensor memory.  Tensor memory: 2 slots x 256
// columns; consumer warpgroup wg drains slot wg (tiles i with i % 2 == wg),
// so the MMA fills one slot while the other is read, and the two warpgroups'
// per-row (max, sum) pairs are merged at the end.

constexpr uint32_t kPairKeys = 256;             // keys per pass-1 tile (both CTAs)
constexpr int kStagesPair = 4;                  // K ring of pass 1 (per CTA: 32 KB a stage)

struct P1Smem {
  uint8_t q[2][kKBlockBytes];               // this CTA's 128 query rows [K-block]
  uint8_t k[kStagesPair][2][kKBlockBytes];  // this CTA's 128 keys of the tile [stage][K-block]
  float2 half[4][32];                       // (max, sum) of warpgroup 1, merged at the end
  uint64_t q_full;                          // even CTA: both CTAs' Q rows landed
  uint64_t k_full[kStagesPair];             // even CTA: both CTAs' key halves landed
  uint64_t k_empty[kStagesPair];            // both: the MMAs reading the stage are done
  uint64_t tm_full[2];                      // both: the slot's logits are ready
  uint64_t tm_empty[2];                     // even CTA: the slot's 8 consumer warps copied it out
  uint64_t mma_done;                        // both: every MMA of the pair is done
  uint64_t never;                           // test support: never completes
  uint64_t peer_done;                       // even CTA: the odd CTA's fill count landed (8 bytes)
  int2 peer_fills;                          // even CTA: key tiles the odd CTA issued
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
score_lse_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    Shape sh, Tables tb, int S, float2* __restrict__ part, float* __restrict__ nlse) {
  extern __shared__ uint8_t smem_raw[];
  P1Smem& sm = *reinterpret_cast<P1Smem*>(align1024(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  if (threadIdx.x == 0) {
    mbar_init(&sm.q_full, 1);
    for (int i = 0; i < kStagesPair; ++i) { mbar_init(&sm.k_full[i], 1); mbar_init(&sm.k_empty[i], 1); }
    for (int i = 0; i < 2; ++i) { mbar_init(&sm.tm_full[i], 1); mbar_init(&sm.tm_empty[i], 8); }
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
  cluster_sync();                  // barriers of both CTAs initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;
  // the plan tables come from the kernel just before this one
  dep_wait();
  if (threadIdx.x == 0) dep_launch();
  const int unit = (int)(blockIdx.x >> 1);
  const int r = upper_index(tb.unit0_tc1, sh.n_req, (int32_t)unit);
  const Req rq = tb.req[r];
  int u = unit - tb.unit0_tc1[r];
  const int s = u % S;
  u /= S;
  const int rbp = u % rq.nrb;
  u /= rq.nrb;
  const int g = u % sh.Hkv, l = u / sh.Hkv;
  const int rows = sh.G * rq.W;
  const int ntiles_all = (rq.n + (int)kPairKeys - 1) / (int)kPairKeys;
  const int tps = (ntiles_all + S - 1) / S;
  const int t_begin = s * tps;
  const int ntiles = max(0, min(ntiles_all, t_begin + tps) - t_begin);
  const int qrow = (int)(rq.q_off / 128 + ((int64_t)l * sh.Hq + g * sh.G) * rq.W) + rbp * 256 +
                   (int)rank * (int)kTile;
  const int krow0 = (int)(rq.kv_off / 128 + ((int64_t)l * sh.Hkv + g) * rq.n) + (int)rank * (int)kTile;

  if (warp == kProducerWarp && lane == 0) {
    // ---- TMA producer (both CTAs): own rows and key halves, counted on the even CTA's barriers
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    const uint32_t q_full0 = map_to_rank(smem_u32(&sm.q_full), 0);
    if (rank == 0) mbar_arrive_expect_tx(&sm.q_full, 2 * kTileBytes);
    for (int kb = 0; kb < 2; ++kb) tma_load_2d_pair(sm.q[kb], &tmQ, kb * 64, qrow, q_full0);
    int issued = 0;
    for (int i = 0; i < ntiles; ++i) {
      const int st = i % kStagesPair;
      if (!mbar_wait(&sm.k_empty[st], ((i / kStagesPair) & 1) ^ 1, abort)) break;
      if (rank == 0) mbar_arrive_expect_tx(&sm.k_full[st], 2 * kTileBytes);
      const uint32_t k_full0 = map_to_rank(smem_u32(&sm.k_full[st]), 0);
      const int y = krow0 + (t_begin + i) * (int)kPairKeys;
      tma_load_2d_pair(sm.k[st][0], &tmK, 0, y, k_full0);
      tma_load_2d_pair(sm.k[st][1], &tmK, 64, y, k_full0);
      ++issued;
    }
    // the even CTA waits until every copy of both CTAs has landed (both
    // always issue their Q rows; the key ring with the odd CTA's count)
    if (rank == 1) report_fills(&sm.peer_fills, &sm.peer_done, issued, 0);
    if (rank == 0) {
      drain_wait(&sm.q_full, 0);
      const int2 f = peer_fills(&sm.peer_done, &sm.peer_fills, make_int2(issued, 0), abort);
      drain_pair_ring(sm.k_full, kStagesPair, issued, f.x, kTileBytes);
    }
  } else if (warp == kMmaWarp && lane == 0 && rank == 0) {
    // ---- MMA issuer (even CTA): D[row][key] for 256 rows x 256 keys per tile
    const uint32_t idesc = idesc_bf16_f32(2 * kTile, kPairKeys);
    bool ok = mbar_wait(&sm.q_full, 0, abort);
    for (int i = 0; ok && i < ntiles; ++i) {
      const int st = i % kStagesPair;
      const int slot = i & 1;
      if (!mbar_wait(&sm.k_full[st], (i / kStagesPair) & 1, abort)) break;
      if (!mbar_wait(&sm.tm_empty[slot], ((i >> 1) & 1) ^ 1, abort)) break;
      tc_fence_after();
      const uint32_t d = tbase + (uint32_t)slot * kPairKeys;
#pragma unroll
      for (int kb = 0; kb < 2; ++kb)
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16_pair(d, desc_sw128(smem_u32(sm.q[kb]) + k * 32),
                        desc_sw128(smem_u32(sm.k[st][kb]) + k * 32), idesc, (kb | k) ? 1u : 0u);
      mma_commit_pair(&sm.tm_full[slot], 3);
      mma_commit_pair(&sm.k_empty[st], 3);
    }
    mma_commit_pair(&sm.mma_done, 3);
    drain_wait(&sm.mma_done, 0);
  } else if (warp == kMmaWarp && lane == 0) {
    // odd CTA: the pair's MMAs (and their arrivals on this CTA's barriers) are done
    drain_wait(&sm.mma_done, 0);
  } else if (warp < 8) {
    if ((sh.test_wait & VC_TEST_WAIT_SCORE_LSE) && warp == 0) {
      if (lane == 0 && injected_wait_gives_up(&sm.never)) {
        set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
        *abort = 1;
      }
      __syncwarp();
    }
    // ---- row statistics: one thread per row (= TMEM lane).  Warpgroup wg
    // takes the tiles i with i % 2 == wg (TMEM slot wg), all 256 columns in
    // two halves, so the two warpgroups on a sub-partition run a tile apart
    // and one's waits and TMEM loads overlap the other's exps.
    const int wg = warp >> 2;
    const int lrow = ((warp & 3) << 5) + lane;
    const uint32_t lane_off = (uint32_t)((warp & 3) << 5) << 16;
    const uint32_t tm_empty0 = lane == 0 ? map_to_rank(smem_u32(&sm.tm_empty[wg]), 0) : 0u;
    const float s2 = sh.scale_log2;
    float m = -INFINITY;
    Kahan z;
    z.init();
    // The half's exp2 sum is added to z only after the next half's exp2 terms
    // are issued (its terms have arrived by then); adding it at once would
    // stall the warp until the exp2 unit has worked through its queue.
    float pend = 0.f;
    for (int i = wg; i < ntiles; i += 2) {
      if (!warp_wait(&sm.tm_full[wg], (i >> 1) & 1, abort)) break;
      tc_fence_after();
#pragma unroll 1
      for (int hf = 0; hf < 2; ++hf) {
        const int valid = min((int)kTile, rq.n - (t_begin + i) * (int)kPairKeys - hf * (int)kTile);
        const uint32_t col0 = tbase + lane_off + (uint32_t)wg * kPairKeys + (uint32_t)hf * kTile;
        float x[8][16];
        {
          uint32_t v[8][16];
#pragma unroll
          for (int p = 0; p < 8; ++p) tmem_ld16(col0 + p * 16, v[p]);
          tmem_wait_only();
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            reg_fence(v[p]);
#pragma unroll
            for (int j = 0; j < 16; ++j) x[p][j] = __uint_as_float(v[p][j]);
          }
        }
        if (hf == 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(tm_empty0);   // slot copied out
        }
        if (valid < (int)kTile) {                 // keys >= n (ragged last tile)
#pragma unroll
          for (int p = 0; p < 8; ++p)
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (p * 16 + j >= valid) x[p][j] = -INFINITY;
        }
        float pm[8];
#pragma unroll
        for (int p = 0; p < 8; ++p) {
          float a = fmaxf(x[p][0], x[p][1]);
#pragma unroll
          for (int j = 2; j < 16; j += 2) a = fmax3(a, x[p][j], x[p][j + 1]);
          pm[p] = a;
        }
        const float cm = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7]));
        const float xm = cm * s2;
        if (xm > m) {
          const float c = ex2(m - xm);
          z.s *= c;
          z.c *= c;
          pend *= c;
          m = xm;
        }
        if (m != -INFINITY) {
          float2 nb[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) nb[j] = make_float2(-m, -m);
          float ps[8];
#pragma unroll
          for (int p = 0; p < 8; ++p) ps[p] = exp2_sum16(x[p], make_float2(s2, s2), nb);
          z.add(pend);
          pend = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        }
      }
    }
    z.add(pend);
    // merge the two warpgroups' statistics of each row
    if (wg == 1) sm.half[warp & 3][lane] = make_float2(m, z.s);
    __syncwarp();
    named_sync(1, 256);
    if (wg == 0) {
      const float2 o = sm.half[warp & 3][lane];
      const float mm = fmaxf(m, o.x);
      float zz = 0.f;
      if (mm != -INFINITY) {
        if (m != -INFINITY) zz += z.s * ex2(m - mm);
        if (o.x != -INFINITY) zz += o.y * ex2(o.x - mm);
      }
      const int rho = rbp * 256 + (int)rank * (int)kTile + lrow;
      if (S > 1) {
        if (rho < rows)
          part[(rq.lse_off + ((int64_t)l * sh.Hq + g * sh.G) * rq.W + rho) * S + s] = make_float2(mm, zz);
      } else if (rho < rq.C * rq.cw) {
        // one key split: the merge's result directly, same arithmetic
        float out = -INFINITY;                      // padding rows: exp2(x + -inf) = 0
        if (rho < rows) {
          const float z = mm != -INFINITY ? zz * exp2f(0.f) : 0.f;
          out = -(mm + log2f(z));
        }
        nlse[rq.lsep_off + ((int64_t)l * sh.Hkv + g) * (rq.C * rq.cw) + rho] = out;
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

// ---------------------------------------------------------------------------
// merge: minus lse2 per window row into the chunk-padded layout; grid
// (padded rows / 256, n_req)

__global__ void lse_merge_kernel(Shape sh, Tables tb, int S, const float2* __restrict__ part,
                                 const float* __restrict__ lse_nat, float* __restrict__ nlse) {
  dep_wait();                                 // the partial statistics of pass 1
  if (threadIdx.x == 0) dep_launch();
  const Req rq = tb.req[blockIdx.y];
  const int rows = rq.C * rq.cw;              // padded rows of one (layer, KV head)
  const int64_t per = (int64_t)sh.L * sh.Hkv * rows;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= per) return;
  const int p = (int)(i % rows);
  const int grp = (int)(i / rows);
  const int l = grp / sh.Hkv, g = grp % sh.Hkv;
  float out = -INFINITY;                      // padding rows: exp2(x + -inf) = 0
  if (p < sh.G * rq.W) {
    const int64_t o = rq.lse_off + ((int64_t)l * sh.Hq + g * sh.G) * rq.W + p;
    if (lse_nat) {
      out = -lse_nat[o] * kLog2e;
    } else {
      float m = -INFINITY;
      for (int s = 0; s < S; ++s) m = fmaxf(m, part[o * S + s].x);
      float z = 0.f;
      for (int s = 0; s < S; ++s) {
        const float2 q = part[o * S + s];
        if (q.x != -INFINITY) z += q.y * exp2f(q.x - m);
      }
      out = -(m + log2f(z));
    }
  }
  nlse[rq.lsep_off + i] = out;
}

// ---------------------------------------------------------------------------
// pass 2 on CTA pairs
//
// A pair owns a tile of 256 keys (128 per CTA, keys in TMEM lanes) and walks
// all layers: per layer its K rows (each CTA its own 128 keys, double
// buffered), then the layer's G*W window rows in C chunks of cw <= 256 rows
// (G*W spread evenly, rounded up to 16, so a 448-row set is two chunks of
// 224, not two of 256; CTA r uses rows r*cw/2 ... of the chunk from a
// 128-row box).  One 2-SM MMA chain (M = 256 keys, N = cw rows, K = 128)
// leaves each key's cw logits in its own CTA's tensor memory.  Every CTA
// also loads the chunk's cw row normalisers into its own shared memory (rows
// past the row set carry -inf and add 0).  Warpgroup wg takes the chunks q
// with q % 2 == wg (TMEM slot wg), the cw columns in up to two halves of 128.

constexpr uint32_t kChunkRows = 256;            // window rows per pass-2 chunk (both CTAs)

// One pass-2 consumer step over NP groups of 16 TMEM columns (one key per
// lane, one window row per column) starting at col0: load, optionally free
// the slot (last load of the chunk), then sum exp2(x * s2 + nl[col]) over the
// columns.  NP is a compile-time count so the loads and sums unroll fully.
template <int NP>
__device__ __forceinline__ float colsum_group(uint32_t col0, const float* nl_col, float s2, bool release,
                                              uint32_t tm_empty0, int lane) {
  float x[NP][16];
  {
    uint32_t vv[NP][16];
#pragma unroll
    for (int p = 0; p < NP; ++p) tmem_ld16(col0 + p * 16, vv[p]);
    tmem_wait_only();
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      reg_fence(vv[p]);
#pragma unroll
      for (int j = 0; j < 16; ++j) x[p][j] = __uint_as_float(vv[p][j]);
    }
  }
  if (release) {
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive_cluster(tm_empty0);   // slot copied out
  }
  const float4* nl = reinterpret_cast<const float4*>(nl_col);
  float ps[8];
#pragma unroll
  for (int p = 0; p < 8; ++p) ps[p] = 0.f;
#pragma unroll
  for (int p = 0; p < NP; ++p) {
    float2 nb[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 f = nl[p * 4 + j];
      nb[2 * j] = make_float2(f.x, f.y);
      nb[2 * j + 1] = make_float2(f.z, f.w);
    }
    ps[p] = exp2_sum16(x[p], make_float2(s2, s2), nb);
  }
  return ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
}
constexpr int kQStagesPair = 4;                 // Q ring of pass 2 (per CTA: 32 KB + 1 KB a stage)

struct P2Smem {
  uint8_t k[2][2][kKBlockBytes];              // this CTA's 128 keys of layer l [l & 1][K-block]
  uint8_t q[kQStagesPair][2][kKBlockBytes];   // this CTA's 128 rows of the chunk [stage][K-block]
  float nlse[kQStagesPair][kChunkRows];       // minus lse2 of all 256 rows of the chunk
  float red[2][kTile];                        // [warpgroup][key]
  uint64_t k_full[2];                         // even CTA: both CTAs' keys of the layer landed
  uint64_t k_empty[2];                        // both: the layer's MMAs are done
  uint64_t q_full[kQStagesPair];              // even CTA: both CTAs' rows of the chunk landed
  uint64_t nl_full[kQStagesPair];             // both: this CTA's copy of the normalisers landed
  uint64_t q_empty[kQStagesPair];             // both: MMAs done and this CTA's warpgroup read the normalisers
  uint64_t tm_full[2];                        // both: the slot's logits are ready
  uint64_t tm_empty[2];                       // even CTA: the slot's 8 consumer warps copied it out
  uint64_t mma_done;                          // both: every MMA of the pair is done
  uint64_t never;                             // test support: never completes
  uint64_t peer_done;                         // even CTA: the odd CTA's fill counts landed (8 bytes)
  int2 peer_fills;                            // even CTA: (key, chunk) tiles the odd CTA issued
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
score_colsum_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                       Shape sh, Tables tb, const float* __restrict__ nlse, float* __restrict__ scores) {
  extern __shared__ uint8_t smem_raw[];
  P2Smem& sm = *reinterpret_cast<P2Smem*>(align1024(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int unit = (int)(blockIdx.x >> 1);

  const int r = upper_index(tb.unit0_tc2, sh.n_req, (int32_t)unit);
  const Req rq = tb.req[r];
  const int u = unit - tb.unit0_tc2[r];
  const int g = u / rq.tiles, kt = u % rq.tiles;
  const int C2 = rq.C;                         // chunks per layer
  const int cw = rq.cw;                        // rows per chunk (multiple of 16, <= 256)
  const int L = sh.L;
  const int Ls = rq.Ls;                        // layers scored (all L unless per-layer ranking prunes)

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.k_full[i], 1);
      mbar_init(&sm.k_empty[i], 1);
      mbar_init(&sm.tm_full[i], 1);
      mbar_init(&sm.tm_empty[i], 8);
    }
    for (int i = 0; i < kQStagesPair; ++i) {
      mbar_init(&sm.q_full[i], 1);
      mbar_init(&sm.nl_full[i], 1);
      mbar_init(&sm.q_empty[i], 1 + 4);   // MMA commit + the stage's 4 consumer warps of this CTA
    }
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
  cluster_sync();
  tc_fence_after();
  const uint32_t tbase = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kProducerWarp && lane == 0) {
    // ---- TMA producer (both CTAs): K half of layer l, then the layer's row chunks
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    int k_issued = 0, q_issued = 0;
    bool ok = true, waited = false;
    for (int l = 0; ok && l < Ls; ++l) {
      const int ks = l & 1;
      if (!mbar_wait(&sm.k_empty[ks], ((l >> 1) & 1) ^ 1, abort)) break;
      if (rank == 0) mbar_arrive_expect_tx(&sm.k_full[ks], 2 * kTileBytes);
      const uint32_t k_full0 = map_to_rank(smem_u32(&sm.k_full[ks]), 0);
      const int ky = (int)(rq.kv_off / 128 + ((int64_t)l * sh.Hkv + g) * rq.n) + kt * (int)kPairKeys +
                     (int)rank * (int)kTile;
      tma_load_2d_pair(sm.k[ks][0], &tmK, 0, ky, k_full0);
      tma_load_2d_pair(sm.k[ks][1], &tmK, 64, ky, k_full0);
      ++k_issued;
      const int qy0 = (int)(rq.q_off / 128 + ((int64_t)l * sh.Hq + g * sh.G) * rq.W) + (int)rank * (cw >> 1);
      for (int c = 0; c < C2; ++c) {
        const int q = l * C2 + c, qs = q % kQStagesPair;
        if (!mbar_wait(&sm.q_empty[qs], ((q / kQStagesPair) & 1) ^ 1, abort)) { ok = false; break; }
        if (rank == 0) mbar_arrive_expect_tx(&sm.q_full[qs], 2 * kTileBytes);
        const uint32_t q_full0 = map_to_rank(smem_u32(&sm.q_full[qs]), 0);
        tma_load_2d_pair(sm.q[qs][0], &tmQ, 0, qy0 + c * cw, q_full0);
        tma_load_2d_pair(sm.q[qs][1], &tmQ, 64, qy0 + c * cw, q_full0);
        if (!waited) {
          // the keys and the first rows are inputs and load while the
          // kernel before this one drains; the normalisers are its output
          dep_wait();
          dep_launch();
          waited = true;
        }
        mbar_arrive_expect_tx(&sm.nl_full[qs], (uint32_t)cw * 4);
        bulk_load(sm.nlse[qs], nlse + rq.lsep_off + ((int64_t)(l * sh.Hkv + g) * C2 + c) * cw,
                  (uint32_t)cw * 4, &sm.nl_full[qs]);
        ++q_issued;
      }
    }
    if (!waited) {                 // no chunk (nothing scored, or an abort)
      dep_wait();
      dep_launch();
    }
    // every copy this CTA started has landed before the pair may leave: the
    // normalisers on this CTA's barriers, the tiles on the even CTA's
    if (rank == 1) report_fills(&sm.peer_fills, &sm.peer_done, k_issued, q_issued);
    for (int i = max(0, q_issued - kQStagesPair); i < q_issued; ++i)
      drain_wait(&sm.nl_full[i % kQStagesPair], (i / kQStagesPair) & 1);
    if (rank == 0) {
      const int2 f = peer_fills(&sm.peer_done, &sm.peer_fills, make_int2(k_issued, q_issued), abort);
      drain_pair_ring(sm.k_full, 2, k_issued, f.x, kTileBytes);
      drain_pair_ring(sm.q_full, kQStagesPair, q_issued, f.y, kTileBytes);
    }
  } else if (warp == kMmaWarp && lane == 0 && rank == 0) {
    // ---- MMA issuer (even CTA): D[key][row] = K_tile . Q_chunk^T, 256 x cw
    const uint32_t idesc = idesc_bf16_f32(2 * kTile, (uint32_t)cw);
    bool ok = true;
    for (int l = 0; ok && l < Ls; ++l) {
      const int ks = l & 1;
      if (!mbar_wait(&sm.k_full[ks], (l >> 1) & 1, abort)) break;
      for (int c = 0; c < C2; ++c) {
        const int q = l * C2 + c, qs = q % kQStagesPair, slot = q & 1;
        if (!mbar_wait(&sm.q_full[qs], (q / kQStagesPair) & 1, abort)) { ok = false; break; }
        if (!mbar_wait(&sm.tm_empty[slot], ((q >> 1) & 1) ^ 1, abort)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tbase + (uint32_t)slot * kChunkRows;
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16_pair(d, desc_sw128(smem_u32(sm.k[ks][kb]) + k * 32),
                          desc_sw128(smem_u32(sm.q[qs][kb]) + k * 32), idesc, (kb | k) ? 1u : 0u);
        mma_commit_pair(&sm.tm_full[slot], 3);
        mma_commit_pair(&sm.q_empty[qs], 3);
      }
      if (ok) mma_commit_pair(&sm.k_empty[ks], 3);
    }
    mma_commit_pair(&sm.mma_done, 3);
    drain_wait(&sm.mma_done, 0);
  } else if (warp == kMmaWarp && lane == 0) {
    // odd CTA: the pair's MMAs (and their arrivals on this CTA's barriers) are done
    drain_wait(&sm.mma_done, 0);
  } else if (warp < 8) {
    if ((sh.test_wait & VC_TEST_WAIT_SCORE_COLSUM) && warp == 0) {
      if (lane == 0 && injected_wait_gives_up(&sm.never)) {
        set_status(tb.status, VC_ERR_DEVICE_TIMEOUT);
        *abort = 1;
      }
      __syncwarp();
    }
    // ---- column sums: one thread per key (= TMEM lane)
    const int wg = warp >> 2;
    const int key = ((warp & 3) << 5) + lane;
    const uint32_t lane_off = (uint32_t)((warp & 3) << 5) << 16;
    const uint32_t tm_empty0 = lane == 0 ? map_to_rank(smem_u32(&sm.tm_empty[wg]), 0) : 0u;
    const float s2 = sh.scale_log2;
    const int v = kt * (int)kPairKeys + (int)rank * (int)kTile + key;
    const bool per_layer = sh.rank_mode == VC_RANK_PER_LAYER;
    const int nhalf = (cw + (int)kTile - 1) / (int)kTile;   // 1 or 2 halves of 128 columns
    // The sum of a group of exp2 terms is ready only once the exp2 unit has
    // worked through the warp's queue, which takes long after the last one
    // is issued.  So nothing waits for a sum right after issuing it: the last
    // half-sum of a chunk stays pending until the next chunk's first half is
    // issued, and a layer is added to the total only after the next layer's
    // chunk is issued.  Layer l accumulates into a[l & 1]; the additions keep
    // their order (halves in order into the layer, layers in order into the
    // total).
    Kahan tot, a0, a1;
    tot.init();
    a0.init();
    a1.init();
    float pend = 0.f;                               // last half-sum of the latest chunk
    int pend_l = -1;                                // its layer (-1: none)
    auto add_to_layer = [&](int l, float x) {
      if (l & 1) a1.add(x);
      else a0.add(x);
    };
    auto flush = [&](int l) {                       // the pending half-sum, if it is layer l's
      if (pend_l == l) {
        add_to_layer(l, pend);
        pend_l = -1;
      }
    };
    auto half_sum = [&](int qs, int hf) -> float {
      const int np = min(8, (cw >> 4) - hf * 8);    // 16-column groups of this half
      const uint32_t col0 = tbase + lane_off + (uint32_t)wg * kChunkRows + (uint32_t)hf * kTile;
      const float* nl = sm.nlse[qs] + hf * (int)kTile;
      const bool rel = hf == nhalf - 1;             // the slot is free after this load
      switch (np) {
        case 8: return colsum_group<8>(col0, nl, s2, rel, tm_empty0, lane);
        case 7: return colsum_group<7>(col0, nl, s2, rel, tm_empty0, lane);
        case 6: return colsum_group<6>(col0, nl, s2, rel, tm_empty0, lane);
        case 5: return colsum_group<5>(col0, nl, s2, rel, tm_empty0, lane);
        case 4: return colsum_group<4>(col0, nl, s2, rel, tm_empty0, lane);
        case 3: return colsum_group<3>(col0, nl, s2, rel, tm_empty0, lane);
        case 2: return colsum_group<2>(col0, nl, s2, rel, tm_empty0, lane);
        default: return colsum_group<1>(col0, nl, s2, rel, tm_empty0, lane);
      }
    };
    // one chunk q (layer l) of this warpgroup: wait for its logits and
    // normalisers, issue its exp2 terms, release the normaliser stage
    auto run_chunk = [&](int q, int l) {
      const int qs = q % kQStagesPair;
      const bool go = __all_sync(0xffffffffu, *abort == 0);
      if (go && warp_wait(&sm.tm_full[wg], (q >> 1) & 1, abort) &&
          warp_wait(&sm.nl_full[qs], (q / kQStagesPair) & 1, abort)) {
        tc_fence_after();
        const float h0 = half_sum(qs, 0);
        if (pend_l >= 0) {                          // the previous chunk's last half
          add_to_layer(pend_l, pend);
          pend_l = -1;
        }
        if (nhalf == 2) {
          const float h1 = half_sum(qs, 1);
          add_to_layer(l, h0);
          pend = h1;
        } else {
          pend = h0;
        }
        pend_l = l;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.q_empty[qs]);   // this warp is done with the stage's normalisers
    };
    auto layer_total = [&](int l) -> float {         // layer l's sum, its accumulator reset
      flush(l);
      const float t = (l & 1) ? a1.s : a0.s;
      if (l & 1) a1.init();
      else a0.init();
      return t;
    };
    if (per_layer) {
      for (int l = 0; l < Ls; ++l) {
        for (int c = 0; c < C2; ++c) {
          const int q = l * C2 + c;
          if ((q & 1) == wg) run_chunk(q, l);
        }
        sm.red[wg][key] = layer_total(l);
        __syncwarp();
        named_sync(1, 2 * kTile);
        if (wg == 0 && v < rq.n)
          scores[rq.s_off + ((int64_t)l * sh.Hkv + g) * rq.n + v] = sm.red[0][key] + sm.red[1][key];
        named_sync(1, 2 * kTile);
      }
    } else {
      // (Ls == L here: the shared ranking averages every layer)
      for (int l = 0; l < Ls; ++l) {
        for (int c = 0; c < C2; ++c) {
          const int q = l * C2 + c;
          if ((q & 1) == wg) run_chunk(q, l);
        }
        if (l > 0) tot.add(layer_total(l - 1));
      }
      if (Ls > 0) tot.add(layer_total(Ls - 1));
      sm.red[wg][key] = tot.s;
      __syncwarp();
      named_sync(1, 2 * kTile);
      if (wg == 0 && v < rq.n)
        scores[rq.s_off + (int64_t)g * rq.n + v] = (sm.red[0][key] + sm.red[1][key]) / (float)L;
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

// ---------------------------------------------------------------------------
// host side

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

// [rows][128] bf16 tensor, boxes of 128 rows x 64 elements, 128-byte swizzle.
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

int score_tc_max_splits() { return 4; }

// CTA pairs of the lse pass that fit on the device at once (pairs must sit on
// one TPC, so this can be below half the SM count).
int score_tc_pair_slots() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (cached[dev] > 0) return cached[dev];
  const size_t smem1 = sizeof(P1Smem) + 1024;
  if (cudaFuncSetAttribute(score_lse_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1) !=
      cudaSuccess)
    return 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, score_lse_tc_kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    int sms = 2;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    n = std::max(1, sms / 2);
  }
  cached[dev] = n;
  return n;
}

cudaError_t launch_score_tc(const void* Qw, const void* K, const Shape& sh, const Tables& tb,
                            const TcPlan& tp, float2* part, float* nlse_pad, const float* lse_nat,
                            float* scores, cudaStream_t st) {
  CUtensorMap mq, mk;
  if (!make_rows_map(&mq, Qw, tp.q_rows) || !make_rows_map(&mk, K, tp.k_rows))
    return cudaErrorInvalidValue;
  cudaError_t e;
  if (!lse_nat) {
    const size_t smem1 = sizeof(P1Smem) + 1024;
    e = cudaFuncSetAttribute(score_lse_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return e;
    ProfileScope ps("score_lse_tc", st);
    e = launch_dep(score_lse_tc_kernel, dim3(2 * tp.units1), dim3(kThreads), smem1, st, mq, mk, sh, tb, tp.S,
                   part, nlse_pad);
    if (e != cudaSuccess) return e;
  }
  if (lse_nat || tp.S > 1) {
    ProfileScope ps("lse_merge", st);
    e = launch_dep(lse_merge_kernel, dim3((unsigned)((tp.max_prows + 255) / 256), sh.n_req), dim3(256), 0, st,
                   sh, tb, tp.S, static_cast<const float2*>(part), lse_nat, nlse_pad);
    if (e != cudaSuccess) return e;
  }
  const size_t smem2 = sizeof(P2Smem) + 1024;
  e = cudaFuncSetAttribute(score_colsum_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  if (e != cudaSuccess) return e;
  ProfileScope ps("score_colsum_tc", st);
  return launch_dep(score_colsum_tc_kernel, dim3(2 * tp.units2), dim3(kThreads), smem2, st, mq, mk, sh, tb,
                    static_cast<const float*>(nlse_pad), scores);
}

}  // namespace vc
