// Decode attention over the compressed cache (Sec. 2 "VLLM Decoding", with the
// visual part of layer l's cache replaced by PruneKV's (K_new, V_new), Sec. 3.2):
//     out_j = softmax(q_j K_g^T * scale) V_g,  g = j // G,
// over KV head g's B kept visual rows of the layer followed by its T text rows.
//
// A decode step reads the whole layer cache once for a handful of query rows:
// bound by those reads.  One 256-thread CTA per unit (request, KV head, split
// of the keys); a split's rows are staged in shared memory by 16-byte
// asynchronous copies (the whole split in flight at once), the row's 16-byte
// pieces XOR-permuted so that the reads hit distinct banks.
//   decode_mma_kernel      (bf16 caches, splits of 256 keys) K rows, then V
//                          rows, in one buffer; QK^T and PV as mma.sync
//                          m16n8k16 tiles: keys, then output dimensions, as
//                          M and the G <= 8 query heads as N = 8; the
//                          split's softmax in between.  The CTA that
//                          finishes the last split of a (request, KV head)
//                          merges the pair's split states into the output.
//                          Its Q4 form reads the visual rows from the 4-bit
//                          cache: key codes and parameters loaded into
//                          registers and expanded to bf16 rows in the same
//                          buffer; value codes and parameters copied into
//                          shared memory during QK and expanded after the
//                          softmax.
//   decode_partial_kernel  (fp32 caches, splits of 256 keys) the same steps on
//                          CUDA cores, K then V rows in one buffer: two
//                          threads per key pair form the logits with packed
//                          fp32 FMAs against duplicated query values; threads
//                          own 16-byte pieces of the V rows for a key slice;
//                          decode_combine_kernel (one warp per request and
//                          query head) then merges the splits.
// Split states are the unnormalised partial output and (max, sum) per query.
// A query with no keys at all (an evicted layer, no text) gets zeros.
#include <cuda_bf16.h>
#include <algorithm>
#include <stdint.h>

#include "kernels.h"
#include "profile.h"
#include "tc_common.cuh"
#include "vc_common.cuh"

namespace vc {
namespace {

constexpr int kSplitF = 256;                  // keys per CTA, fp32 caches (CUDA cores)
constexpr int kSplitM = 256;                  // keys per CTA, bf16 caches (tensor cores)
constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kGm = kDecodeMaxGroup;
constexpr float kLog2eF = 1.4426950408889634f;

template <typename T, int D>
struct DecCfg {
  static constexpr int RB = D * (int)sizeof(T);          // bytes of a cache row
  static constexpr int PR = RB / 16;                     // 16-byte pieces of a row
  static constexpr int EPP = 16 / (int)sizeof(T);        // elements of a piece
  static constexpr int RW = 32 / PR;                     // rows a warp reads at once (phase 3)
  static constexpr int KS = kDecWarps * RW;              // phase-3 key slices
  static constexpr size_t BUF = (size_t)kSplitF * RB;     // K rows, then V rows, then partials
  static constexpr size_t QS = (size_t)D * kGm * 8;      // (q, q) pairs [D][kGm]
  static constexpr size_t PS = (size_t)kSplitF * kGm * 8; // (p, p) pairs [kSplitF][kGm]
  static constexpr size_t RED = (size_t)2 * kDecWarps * kGm * 4;
  static constexpr size_t SMEM = BUF + QS + PS + RED;
  static_assert(PR >= 8 && PR <= 32, "row of 8..32 pieces");
  static_assert(kSplitF == kDecThreads, "two threads per key pair (p, p + kSplitF / 2)");
  static_assert((size_t)kDecWarps * kGm * D * 4 <= BUF, "warp partials fit the row buffer");
};

__device__ __forceinline__ int piece_slot(int r, int c) { return c ^ ((r & 3) << 1); }

__device__ __forceinline__ void unpack(const uint4& u, const float*, float (&v)[4]) {
  v[0] = __uint_as_float(u.x); v[1] = __uint_as_float(u.y);
  v[2] = __uint_as_float(u.z); v[3] = __uint_as_float(u.w);
}

__device__ __forceinline__ int find_req(const DecodeTable& tb, int unit) {
  int lo = 0, hi = tb.n_req - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tb.req[mid].unit0 <= unit) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Stage rows [0, nk) of the split (visual rows first, then text rows) into buf.
template <typename T, int D>
__device__ __forceinline__ void stage_rows(uint8_t* buf, const T* vis, const T* txt, int nv, int nk) {
  using C = DecCfg<T, D>;
  for (int i = (int)threadIdx.x; i < nk * C::PR; i += kDecThreads) {
    const int r = i / C::PR, c = i % C::PR;
    const T* src = r < nv ? vis + (int64_t)r * D : txt + (int64_t)(r - nv) * D;
    tc::cp_async16(buf + (size_t)r * C::RB + piece_slot(r, c) * 16, src + c * C::EPP, 16);
  }
  tc::cp_async_commit();
}

template <typename T, int D>
__global__ void __launch_bounds__(kDecThreads, 1) decode_partial_kernel(
    const __grid_constant__ DecodeTable tb, const T* __restrict__ q, const T* __restrict__ Kc,
    const T* __restrict__ Vc, const T* __restrict__ Kt, const T* __restrict__ Vt,
    float* __restrict__ part_o, float2* __restrict__ part_ml) {
  using C = DecCfg<T, D>;
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* buf = dsm;
  float2* qs = reinterpret_cast<float2*>(dsm + C::BUF);               // [D][kGm]
  float2* ps = reinterpret_cast<float2*>(dsm + C::BUF + C::QS);       // [kSplitF][kGm]
  float* wmax = reinterpret_cast<float*>(dsm + C::BUF + C::QS + C::PS);
  float* wsum = wmax + kDecWarps * kGm;
  const int unit = blockIdx.x;
  const int r = find_req(tb, unit);
  const DecodeReq rq = tb.req[r];
  const int u = unit - rq.unit0;
  const int g = u / rq.nsplit, s = u % rq.nsplit;
  const int G = tb.G;
  const int k0 = s * tb.split;                // tb.split == kSplitF on this path
  const int nk = min(tb.split, rq.B + rq.T - k0);
  const int nv = max(0, min(nk, rq.B - k0));  // the split's visual keys come first
  const int64_t vis0 = rq.vis_row0 + (int64_t)g * rq.B + k0;
  const int64_t txt0 = rq.txt_row0 + (int64_t)g * rq.T + (k0 + nv - rq.B);
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  stage_rows<T, D>(buf, Kc + vis0 * D, Kt + txt0 * D, nv, nk);
  // query rows g*G ... of request r in log2 units, each value duplicated
  const float c2 = tb.scale * kLog2eF;
  for (int e = t; e < kGm * D; e += kDecThreads) {
    const int jj = e % kGm, d = e / kGm;
    const float x = jj < G ? Elem<T>::to_f(q[((int64_t)r * tb.Hq + g * G + jj) * D + d]) * c2 : 0.f;
    qs[d * kGm + jj] = make_float2(x, x);
  }
  tc::cp_async_wait<0>();
  __syncthreads();
  // phase 1: logits of keys kA = p and kB = p + kSplitF/2 over this thread's pieces
  const int p = t >> 1, h = t & 1;
  const int kA = p, kB = p + kSplitF / 2;
  float2 acc[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) acc[jj] = make_float2(0.f, 0.f);
#pragma unroll 2
  for (int i = 0; i < C::PR / 2; ++i) {
    const int c = 2 * i + h;
    const uint4 ua = *reinterpret_cast<const uint4*>(buf + (size_t)kA * C::RB + piece_slot(kA, c) * 16);
    const uint4 ub = *reinterpret_cast<const uint4*>(buf + (size_t)kB * C::RB + piece_slot(kB, c) * 16);
    float va[C::EPP], vb[C::EPP];
    unpack(ua, (const T*)nullptr, va);
    unpack(ub, (const T*)nullptr, vb);
#pragma unroll
    for (int e = 0; e < C::EPP; ++e) {
      const float2 kv = make_float2(va[e], vb[e]);
      const float4* qrow = reinterpret_cast<const float4*>(qs + (c * C::EPP + e) * kGm);
#pragma unroll
      for (int j2 = 0; j2 < kGm / 2; ++j2) {
        if (2 * j2 < G) {
          const float4 qq = qrow[j2];
          acc[2 * j2] = __ffma2_rn(kv, make_float2(qq.x, qq.y), acc[2 * j2]);
          if (2 * j2 + 1 < G) acc[2 * j2 + 1] = __ffma2_rn(kv, make_float2(qq.z, qq.w), acc[2 * j2 + 1]);
        }
      }
    }
  }
  // the two halves of the row; thread h keeps key h ? kB : kA
  const int kmine = h ? kB : kA;
  const bool valid = kmine < nk;
  float x[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
    const float ax = acc[jj].x + __shfl_xor_sync(0xffffffffu, acc[jj].x, 1);
    const float ay = acc[jj].y + __shfl_xor_sync(0xffffffffu, acc[jj].y, 1);
    x[jj] = valid ? (h ? ay : ax) : -INFINITY;
  }
  __syncthreads();                              // K rows no longer read: stage V
  stage_rows<T, D>(buf, Vc + vis0 * D, Vt + txt0 * D, nv, nk);
  // phase 2: split max per query, exp2 terms and their sum
  float m[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
    m[jj] = x[jj];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m[jj] = fmaxf(m[jj], __shfl_xor_sync(0xffffffffu, m[jj], o));
  }
  if (lane == 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) wmax[warp * kGm + jj] = m[jj];
  }
  __syncthreads();
  float l[kGm];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj) {
    float M = wmax[jj];
#pragma unroll
    for (int w = 1; w < kDecWarps; ++w) M = fmaxf(M, wmax[w * kGm + jj]);
    const float e = valid && jj < G ? exp2f(x[jj] - M) : 0.f;
    if (kmine < kSplitF) ps[kmine * kGm + jj] = make_float2(e, e);
    l[jj] = e;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l[jj] += __shfl_xor_sync(0xffffffffu, l[jj], o);
  }
  if (lane == 0) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) wsum[warp * kGm + jj] = l[jj];
  }
  tc::cp_async_wait<0>();
  __syncthreads();
  if (t < G) {
    float M = wmax[t], L = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) {
      M = fmaxf(M, wmax[w * kGm + t]);
      L += wsum[w * kGm + t];
    }
    part_ml[(int64_t)unit * kGm + t] = make_float2(M, L);
  }
  // phase 3: O[jj][piece c] over key slice ks
  const int c = lane % C::PR, ks = warp * C::RW + lane / C::PR;
  float2 o[kGm][C::EPP / 2];
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj)
#pragma unroll
    for (int e = 0; e < C::EPP / 2; ++e) o[jj][e] = make_float2(0.f, 0.f);
#pragma unroll 2
  for (int kk = ks; kk < nk; kk += C::KS) {
    const uint4 uv = *reinterpret_cast<const uint4*>(buf + (size_t)kk * C::RB + piece_slot(kk, c) * 16);
    float v[C::EPP];
    unpack(uv, (const T*)nullptr, v);
    const float4* prow = reinterpret_cast<const float4*>(ps + kk * kGm);
#pragma unroll
    for (int j2 = 0; j2 < kGm / 2; ++j2) {
      if (2 * j2 < G) {
        const float4 pp = prow[j2];
#pragma unroll
        for (int e = 0; e < C::EPP / 2; ++e) {
          const float2 ve = make_float2(v[2 * e], v[2 * e + 1]);
          o[2 * j2][e] = __ffma2_rn(ve, make_float2(pp.x, pp.y), o[2 * j2][e]);
          if (2 * j2 + 1 < G) o[2 * j2 + 1][e] = __ffma2_rn(ve, make_float2(pp.z, pp.w), o[2 * j2 + 1][e]);
        }
      }
    }
  }
  // rows of a warp, then warps, are added
#pragma unroll
  for (int jj = 0; jj < kGm; ++jj)
#pragma unroll
    for (int e = 0; e < C::EPP / 2; ++e)
#pragma unroll
      for (int sh = C::PR; sh < 32; sh <<= 1) {
        o[jj][e].x += __shfl_xor_sync(0xffffffffu, o[jj][e].x, sh);
        o[jj][e].y += __shfl_xor_sync(0xffffffffu, o[jj][e].y, sh);
      }
  __syncthreads();                              // V rows no longer read: warp partials
  float* wpart = reinterpret_cast<float*>(buf);  // [kDecWarps][kGm][D]
  if (lane < C::PR) {
#pragma unroll
    for (int jj = 0; jj < kGm; ++jj) {
      if (jj < G) {
        float4* dst = reinterpret_cast<float4*>(wpart + ((size_t)warp * kGm + jj) * D + c * C::EPP);
#pragma unroll
        for (int e = 0; e < C::EPP / 4; ++e)
          dst[e] = make_float4(o[jj][2 * e].x, o[jj][2 * e].y, o[jj][2 * e + 1].x, o[jj][2 * e + 1].y);
      }
    }
  }
  __syncthreads();
  for (int i = t; i < G * D; i += kDecThreads) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) sum += wpart[(size_t)w * kGm * D + i];
    part_o[(int64_t)unit * kGm * D + i] = sum;
  }
}

// ---------------------------------------------------------------------------
// bf16 caches: the two contractions of a split on the tensor cores
// (mma.sync m16n8k16, fp32 accumulation) -- keys (QK) or output dimensions
// (PV) as M, the G <= 8 query heads of the KV head as N = 8.  The query rows
// and the probabilities enter as bf16 high + low parts (two MMAs each), so
// the products keep ~16 mantissa bits; K and V are exact in bf16.  Rows are
// staged with the 16-byte pieces of row r XOR-permuted by (r & 7), which
// makes every ldmatrix phase (8 rows, one piece column) conflict-free.

constexpr int kPsLd = kSplitM + 8;             // probability row stride (bf16), 16-byte skew

template <int D>
struct MmaCfg {
  static constexpr int RB = D * 2;
  static constexpr int PR = RB / 16;
  static constexpr int KSTEPS = D / 16;                   // QK k-steps
  static constexpr int DT = D / 16;                       // PV output tiles
  static constexpr int WPT = kDecWarps / DT;              // warps per output tile
  static constexpr int TPW = kSplitM / 16 / kDecWarps;  // QK key tiles per warp
  static constexpr size_t BUF = (size_t)kSplitM * RB;            // one split's K, then V, rows
  static constexpr size_t QBUF = (size_t)kGm * (RB + 16);         // query rows, 16-byte skew
  static constexpr size_t PS = (size_t)2 * kGm * kPsLd * 2;       // P high, P low [kGm][kPsLd]
  static constexpr size_t QF = (size_t)2 * KSTEPS * 2 * 32 * 4;   // Q^T fragments, high and low
  static constexpr size_t RED = (size_t)(2 * kDecWarps * kGm + 2 * kGm + 4) * 4;
  static constexpr size_t SMEM = BUF + PS + RED;
  static_assert(TPW * 16 * kDecWarps == kSplitM, "whole QK key tiles per warp");
  static_assert(QBUF + QF <= PS, "query rows and fragments fit the probability region");
  static_assert(DT * WPT == kDecWarps, "output tiles divide the warps");
  static_assert((size_t)WPT * kGm * D * 4 <= BUF, "warp partials fit a row buffer");
  static_assert((size_t)kGm * 32 * 4 <= BUF, "merge weights fit a row buffer");
};

__device__ __forceinline__ int mma_slot(int r, int c) { return c ^ (r & 7); }

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]) : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Unit u of the table: its request, KV head, split and row ranges.
struct UnitRows {
  int r, g, nk, nv, pair, nsplit;
  int64_t vis0, txt0, u_first;   // first visual / text row, first unit of the (request, KV head)
  int64_t kg;                    // 4-bit cache: the split's first key group
};
__device__ __forceinline__ UnitRows unit_rows(const DecodeTable& tb, int unit) {
  UnitRows x;
  x.r = find_req(tb, unit);
  const DecodeReq& rq = tb.req[x.r];
  const int u = unit - rq.unit0;
  x.g = u / rq.nsplit;
  const int s = u % rq.nsplit;
  const int k0 = s * tb.split;
  x.nk = max(0, min(tb.split, rq.B + rq.T - k0));
  x.nv = max(0, min(x.nk, rq.B - k0));
  x.vis0 = rq.vis_row0 + (int64_t)x.g * rq.B + k0;
  x.txt0 = rq.txt_row0 + (int64_t)x.g * rq.T + (k0 + x.nv - rq.B);
  x.pair = x.r * tb.Hkv + x.g;
  x.nsplit = rq.nsplit;
  x.u_first = rq.unit0 + (int64_t)x.g * rq.nsplit;
  x.kg = rq.kg0 + (int64_t)x.g * rq.nkg + k0 / 32;
  return x;
}

// Stage rows [first, last) of a split's rows [0, nk) (visual, then text) and
// zeros up to the next 16-row boundary, so that the last MMA tile reads
// finite values.  Thread t
// copies piece column t % PR of rows t / PR + k * (threads / PR); that row
// step is a multiple of 8, so the column's XOR slot is the same for all of the
// thread's rows.  `zsrc` is any valid device address: the zero-filling copies
// read no bytes.
template <int D>
__device__ __forceinline__ void stage_split(uint32_t buf_s, const __nv_bfloat16* vis,
                                            const __nv_bfloat16* txt, int nv, int nk,
                                            const __nv_bfloat16* zsrc, int first = 0,
                                            int last = kSplitM) {
  using C = MmaCfg<D>;
  constexpr int RSTEP = kDecThreads / C::PR;
  static_assert(RSTEP % 8 == 0, "row step keeps the XOR slot");
  const int c = (int)threadIdx.x % C::PR, r0 = (int)threadIdx.x / C::PR;
  const int rows = min(last, min(kSplitM, (nk + 15) & ~15));
  const uint32_t dst0 = buf_s + r0 * C::RB + mma_slot(r0, c) * 16;
  int r = r0;                                   // first row >= `first` in this thread's column
  if (first > r0) r += (first - r0 + RSTEP - 1) / RSTEP * RSTEP;
  for (; r < rows; r += RSTEP) {
    const __nv_bfloat16* src = r < nv ? vis + (int64_t)r * D + c * 8
                             : r < nk ? txt + (int64_t)(r - nv) * D + c * 8 : zsrc;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst0 + (r - r0) * C::RB),
                 "l"(src), "r"(r < nk ? 16u : 0u) : "memory");
  }
}

// The G query rows of a unit (rows of the q buffer padded by 16 bytes).
template <int D>
__device__ __forceinline__ void stage_q(uint32_t qbuf_s, const __nv_bfloat16* qrows, int G) {
  using C = MmaCfg<D>;
  for (int i = (int)threadIdx.x; i < G * C::PR; i += kDecThreads) {
    const int jj = i / C::PR, c = i % C::PR;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(qbuf_s + jj * (C::RB + 16) + c * 16),
                 "l"(qrows + (int64_t)jj * D + c * 8) : "memory");
  }
}

// 4-bit visual rows [0, nv) of a split expanded into bf16 rows of the
// (XOR-permuted) row buffer: x = fma(code, scale, min) rounded to bf16, the
// rows viscache_kv4_dequantize writes.  Thread t owns the 8-channel piece
// c = t % PR of the PR consecutive rows (t / PR) * PR ...; those rows lie in
// one 32-row key group, so a key thread loads its 8 channels' parameters
// once.  Codes: D/2 bytes a row (4 bytes per piece); KEYS: parameters per
// (key group, channel) from `par` (the split's first group); values: per
// (row, 32-channel group) from `par` (the split's first row).
template <int D, bool KEYS>
__device__ __forceinline__ void expand_q4(uint8_t* buf, const uint8_t* codes, const float* par, int nv) {
  using C = MmaCfg<D>;
  constexpr int RPT = kSplitM * C::PR / kDecThreads;   // rows per thread (= PR)
  static_assert(32 % RPT == 0, "a thread's rows lie in one key group");
  const int c = (int)threadIdx.x % C::PR, r0 = (int)threadIdx.x / C::PR * RPT;
  if (r0 >= nv) return;
  uint32_t w[RPT];
#pragma unroll
  for (int i = 0; i < RPT; ++i)
    w[i] = r0 + i < nv ? *reinterpret_cast<const uint32_t*>(codes + (size_t)(r0 + i) * (D / 2) + 4 * c) : 0u;
  if (KEYS) {
    float4 pk[4];                                 // (scale, min) of channels 8c + 2j, 8c + 2j + 1
    const float4* pp = reinterpret_cast<const float4*>(par + ((size_t)(r0 >> 5) * D + 8 * c) * 2);
#pragma unroll
    for (int j = 0; j < 4; ++j) pk[j] = pp[j];
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      if (r0 + i >= nv) break;
      float x[8];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        x[2 * j] = fmaf((float)((w[i] >> (8 * j)) & 15u), pk[j].x, pk[j].y);
        x[2 * j + 1] = fmaf((float)((w[i] >> (8 * j + 4)) & 15u), pk[j].z, pk[j].w);
      }
      const int r = r0 + i;
      *reinterpret_cast<uint4*>(buf + (size_t)r * C::RB + mma_slot(r, c) * 16) =
          make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
    }
  } else {
    float2 pv[RPT];
#pragma unroll
    for (int i = 0; i < RPT; ++i)
      pv[i] = r0 + i < nv ? reinterpret_cast<const float2*>(par)[(size_t)(r0 + i) * (D / 32) + (c >> 2)]
                          : make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      if (r0 + i >= nv) break;
      float x[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) x[j] = fmaf((float)((w[i] >> (4 * j)) & 15u), pv[i].x, pv[i].y);
      const int r = r0 + i;
      *reinterpret_cast<uint4*>(buf + (size_t)r * C::RB + mma_slot(r, c) * 16) =
          make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
    }
  }
}

// 4-bit value rows staged in shared memory: the split's codes at byte 0
// (D/2 bytes a row) and their parameters after kSplitM rows of codes (one
// (scale, min) pair per row and 32-channel group).  Rows [0, kQ4StageRows)
// of the row buffer hold them, so the staging is used when the split's text
// rows (which load into rows nv ...) start at or after that row.
template <int D>
struct Q4Stage {
  static constexpr int CODES = kSplitM * (D / 2);
  static constexpr int BYTES = CODES + kSplitM * (D / 32) * 8;
  static constexpr int ROWS = (BYTES + 2 * D - 1) / (2 * D);      // bf16 rows the staging covers
  static_assert(BYTES <= (kSplitM / 2) * 2 * D, "the staging fits the first half of the row buffer");
};

// Copy the split's value codes and parameters into the staging area (16-byte
// asynchronous copies; all addresses are 16-byte aligned).
template <int D>
__device__ __forceinline__ void stage_q4_values(uint32_t buf_s, const uint8_t* codes, const float* par, int nv) {
  using S = Q4Stage<D>;
  const uint8_t* pp = reinterpret_cast<const uint8_t*>(par);
  const int nc = nv * (D / 2) / 16, np = nv * (D / 32) * 8 / 16;
  for (int i = (int)threadIdx.x; i < nc + np; i += kDecThreads) {
    const bool is_code = i < nc;
    const uint32_t dst = buf_s + (is_code ? 16u * i : (uint32_t)S::CODES + 16u * (i - nc));
    const uint8_t* src = is_code ? codes + 16 * i : pp + 16 * (i - nc);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
  }
}

// Value rows [0, nv) expanded from the staging area in two steps, so that no
// thread overwrites codes another has not read: every thread first reads its
// rows' codes and parameters (read_q4_values), then, after a barrier, writes
// its bf16 rows (write_q4_values).  Thread t owns the 8-channel piece
// t % PR of rows (t / PR) * RPT ..., as in expand_q4.
template <int D>
struct Q4Values {
  static constexpr int RPT = kSplitM * (D / 8) / kDecThreads;   // as expand_q4: PR = D / 8 pieces a row
  uint32_t w[RPT];
  float2 p[RPT];
};
template <int D>
__device__ __forceinline__ void read_q4_values(const uint8_t* buf, int nv, Q4Values<D>& v) {
  using C = MmaCfg<D>;
  constexpr int RPT = Q4Values<D>::RPT;
  const int c = (int)threadIdx.x % C::PR, r0 = (int)threadIdx.x / C::PR * RPT;
  const float2* par = reinterpret_cast<const float2*>(buf + Q4Stage<D>::CODES);
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const bool in = r0 + i < nv;
    v.w[i] = in ? *reinterpret_cast<const uint32_t*>(buf + (size_t)(r0 + i) * (D / 2) + 4 * c) : 0u;
    v.p[i] = in ? par[(size_t)(r0 + i) * (D / 32) + (c >> 2)] : make_float2(0.f, 0.f);
  }
}
template <int D>
__device__ __forceinline__ void write_q4_values(uint8_t* buf, int nv, const Q4Values<D>& v) {
  using C = MmaCfg<D>;
  constexpr int RPT = Q4Values<D>::RPT;
  const int c = (int)threadIdx.x % C::PR, r0 = (int)threadIdx.x / C::PR * RPT;
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    if (r0 + i >= nv) break;
    float x[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) x[j] = fmaf((float)((v.w[i] >> (4 * j)) & 15u), v.p[i].x, v.p[i].y);
    const int r = r0 + i;
    *reinterpret_cast<uint4*>(buf + (size_t)r * C::RB + mma_slot(r, c) * 16) =
        make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
  }
}

// Decode kernel for bf16 caches: one CTA per unit (request, KV head, split
// of kSplitM keys), three CTAs per SM.  The split's K rows (with the query
// rows) load first; its V rows load into the same buffer during the softmax.
// The CTA that completes the last split of a (request, KV head) merges that
// pair's split states into `out`: an arrival count per pair; no CTA ever
// waits for another.
template <int D, bool Q4>
__global__ void __launch_bounds__(kDecThreads, 3) decode_mma_kernel(
    const __grid_constant__ DecodeTable tb, const __nv_bfloat16* __restrict__ q,
    const __nv_bfloat16* __restrict__ Kc, const __nv_bfloat16* __restrict__ Vc,
    const __nv_bfloat16* __restrict__ Kt, const __nv_bfloat16* __restrict__ Vt,
    const uint8_t* __restrict__ Kq, const uint8_t* __restrict__ Vq, const float* __restrict__ Kqp,
    const float* __restrict__ Vqp, float* __restrict__ part_o, float2* __restrict__ part_ml,
    int32_t* __restrict__ arrivals, __nv_bfloat16* __restrict__ out) {
  using C = MmaCfg<D>;
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* buf = dsm;                           // K rows, V rows, warp partials, merge weights
  __nv_bfloat16* p_hi = reinterpret_cast<__nv_bfloat16*>(dsm + C::BUF);   // [kGm][kPsLd]
  __nv_bfloat16* p_lo = p_hi + kGm * kPsLd;
  // before P is written the probability region holds the query rows and fragments
  uint8_t* qbuf = dsm + C::BUF;                                          // [kGm][RB + 16]
  uint32_t* qf = reinterpret_cast<uint32_t*>(dsm + C::BUF + C::QBUF);     // [hi|lo][ks][hf][lane]
  float* wmax = reinterpret_cast<float*>(dsm + C::BUF + C::PS);
  float* wsum = wmax + kDecWarps * kGm;
  float* cm = wsum + kDecWarps * kGm;           // merge: max, 1/sum per query
  int* last = reinterpret_cast<int*>(cm + 2 * kGm);
  const uint32_t buf_s = tc::smem_u32(buf), qbuf_s = tc::smem_u32(qbuf);
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int gid = lane >> 2, tig = lane & 3;
  const int G = tb.G;
  const int unit = blockIdx.x;
  const UnitRows cur = unit_rows(tb, unit);
  const int nk = cur.nk;
  // bf16 rows move in halves of kHalf rows, so that loads overlap the MMAs:
  // K rows [0, kHalf) with the query rows, then K rows [kHalf, 2 kHalf); QK of
  // the first half (tile w) runs while the second arrives; V rows [0, kHalf)
  // load into the freed half during QK of the second half (tile w + 8), V rows
  // [kHalf, 2 kHalf) during the softmax; PV takes the halves in turn.
  constexpr int kHalf = kSplitM / 2;
  static_assert(C::TPW == 2 && kHalf == 16 * kDecWarps, "QK tile h of every warp lies in half h");
  // 4-bit: the value codes and parameters move into the first half of the row
  // buffer while QK works on the second half (their load overlaps QK and the
  // softmax), unless the split's text rows would land in the staging area
  const bool q4_stage = Q4 && cur.nv >= Q4Stage<D>::ROWS;
  if (Q4) {
    stage_split<D>(buf_s, Kc, Kt + cur.txt0 * D, cur.nv, nk, q, cur.nv);
    stage_q<D>(qbuf_s, q + ((int64_t)cur.r * tb.Hq + cur.g * G) * D, G);
    tc::cp_async_commit();
    expand_q4<D, true>(buf, Kq + cur.vis0 * (D / 2), Kqp + cur.kg * D * 2, cur.nv);
    tc::cp_async_wait<0>();
  } else {
    stage_split<D>(buf_s, Kc + cur.vis0 * D, Kt + cur.txt0 * D, cur.nv, nk, q, 0, kHalf);
    stage_q<D>(qbuf_s, q + ((int64_t)cur.r * tb.Hq + cur.g * G) * D, G);
    tc::cp_async_commit();
    stage_split<D>(buf_s, Kc + cur.vis0 * D, Kt + cur.txt0 * D, cur.nv, nk, q, kHalf);
    tc::cp_async_commit();
    tc::cp_async_wait<1>();                     // K rows [0, kHalf) and the query rows
  }
  __syncthreads();
  // B fragments of Q^T (k = dimension, n = query) in log2 units, high + low,
  // built once for the CTA: item (ks, hf, lane) of KSTEPS x 2 x 32
  constexpr int ITEMS = C::KSTEPS * 2 * 32;
  {
    const float c2 = tb.scale * kLog2eF;
    for (int it = t; it < ITEMS; it += kDecThreads) {
      const int ln = it & 31, hf = (it >> 5) & 1, ks = it >> 6;
      const int qn = ln >> 2, qt = ln & 3;
      float x0 = 0.f, x1 = 0.f;
      if (qn < G) {
        const uint32_t w = *reinterpret_cast<const uint32_t*>(
            qbuf + qn * (C::RB + 16) + (16 * ks + 2 * qt + 8 * hf) * 2);
        x0 = __uint_as_float(w << 16) * c2;
        x1 = __uint_as_float(w & 0xffff0000u) * c2;
      }
      const float h0 = __bfloat162float(__float2bfloat16_rn(x0));
      const float h1 = __bfloat162float(__float2bfloat16_rn(x1));
      qf[it] = pack_bf16(h0, h1);
      qf[ITEMS + it] = pack_bf16(x0 - h0, x1 - h1);
    }
  }
  __syncthreads();
  // QK: warp w takes key tiles w, w + 8, ... (16 keys each)
  float sacc[C::TPW][4];
  bool live[C::TPW];
#pragma unroll
  for (int h = 0; h < C::TPW; ++h) {
    if (q4_stage && h == 1) {
      __syncthreads();                          // K rows [0, kHalf) read: stage the value codes there
      stage_q4_values<D>(buf_s, Vq + cur.vis0 * (D / 2), Vqp + cur.vis0 * (D / 32) * 2, cur.nv);
      tc::cp_async_commit();
    }
    if (!Q4 && h == 1) {
      __syncthreads();                          // K rows [0, kHalf) read: V rows there
      stage_split<D>(buf_s, Vc + cur.vis0 * D, Vt + cur.txt0 * D, cur.nv, nk, q, 0, kHalf);
      tc::cp_async_commit();
      tc::cp_async_wait<1>();                   // K rows [kHalf, 2 kHalf)
      __syncthreads();
    }
    const int mt = warp + h * kDecWarps;
    live[h] = 16 * mt < nk;
#pragma unroll
    for (int i = 0; i < 4; ++i) sacc[h][i] = 0.f;
    if (live[h]) {
      const int row = 16 * mt + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
      for (int ks = 0; ks < C::KSTEPS; ++ks) {
        uint32_t a[4];
        ldsm_x4(buf_s + row * C::RB + mma_slot(row, 2 * ks + (lane >> 4)) * 16, a);
        mma_bf16(sacc[h], a, qf[(2 * ks) * 32 + lane], qf[(2 * ks + 1) * 32 + lane]);
        mma_bf16(sacc[h], a, qf[ITEMS + (2 * ks) * 32 + lane], qf[ITEMS + (2 * ks + 1) * 32 + lane]);
      }
    }
  }
  __syncthreads();                              // K rows, query rows, fragments read: stage V
  if (Q4) {
    stage_split<D>(buf_s, Vc, Vt + cur.txt0 * D, cur.nv, nk, q, cur.nv);
    tc::cp_async_commit();
    if (!q4_stage) expand_q4<D, false>(buf, Vq + cur.vis0 * (D / 2), Vqp + cur.vis0 * (D / 32) * 2, cur.nv);
  } else {
    stage_split<D>(buf_s, Vc + cur.vis0 * D, Vt + cur.txt0 * D, cur.nv, nk, q, kHalf);
    tc::cp_async_commit();
  }
  // softmax over the split: lane holds keys (16 mt + gid, + 8) x queries (2 tig, + 1)
  float x[C::TPW][4];
  float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
  for (int h = 0; h < C::TPW; ++h)
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int key = 16 * (warp + h * kDecWarps) + gid + (i >> 1) * 8;
      x[h][i] = live[h] && key < nk ? sacc[h][i] : -INFINITY;
      if (i & 1) m1 = fmaxf(m1, x[h][i]); else m0 = fmaxf(m0, x[h][i]);
    }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, o));
    m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
  }
  if (gid == 0) {
    wmax[warp * kGm + 2 * tig] = m0;
    wmax[warp * kGm + 2 * tig + 1] = m1;
  }
  __syncthreads();
  float M0 = wmax[2 * tig], M1 = wmax[2 * tig + 1];
#pragma unroll
  for (int w = 1; w < kDecWarps; ++w) {
    M0 = fmaxf(M0, wmax[w * kGm + 2 * tig]);
    M1 = fmaxf(M1, wmax[w * kGm + 2 * tig + 1]);
  }
  float l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int h = 0; h < C::TPW; ++h) {
    if (!live[h]) continue;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int qi = 2 * tig + (i & 1);
      const int key = 16 * (warp + h * kDecWarps) + gid + (i >> 1) * 8;
      const float e = qi < G && key < nk ? exp2f(x[h][i] - ((i & 1) ? M1 : M0)) : 0.f;
      if (i & 1) l1 += e; else l0 += e;
      const __nv_bfloat16 eh = __float2bfloat16_rn(e);
      p_hi[qi * kPsLd + key] = eh;
      p_lo[qi * kPsLd + key] = __float2bfloat16_rn(e - __bfloat162float(eh));
    }
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  if (gid == 0) {
    wsum[warp * kGm + 2 * tig] = l0;
    wsum[warp * kGm + 2 * tig + 1] = l1;
  }
  if (Q4) tc::cp_async_wait<0>();               // V rows (and the staged codes)
  else tc::cp_async_wait<1>();                  // V rows [0, kHalf)
  __syncthreads();
  if (q4_stage) {
    Q4Values<D> qv;
    read_q4_values<D>(buf, cur.nv, qv);
    __syncthreads();                            // every thread has its codes: overwrite them
    write_q4_values<D>(buf, cur.nv, qv);
    __syncthreads();
  }
  if (t < G) {
    float M = wmax[t], L = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) {
      M = fmaxf(M, wmax[w * kGm + t]);
      L += wsum[w * kGm + t];
    }
    part_ml[(int64_t)unit * kGm + t] = make_float2(M, L);
  }
  // PV: warp w takes output dimensions 16 (w % DT) ... and key steps w / DT, + WPT, ...
  const int dt = warp % C::DT, kw = warp / C::DT;
  float oacc[4] = {0.f, 0.f, 0.f, 0.f};
  const int steps = (nk + 15) >> 4;
  const int mi = lane >> 3;
  auto pv_step = [&](int j) {
    const int row = 16 * j + (lane & 7) + (mi >> 1) * 8;
    uint32_t a[4];
    ldsm_x4_t(buf_s + row * C::RB + mma_slot(row, 2 * dt + (mi & 1)) * 16, a);
    const int kb = 16 * j + 2 * tig;
    const uint32_t bh0 = *reinterpret_cast<const uint32_t*>(p_hi + gid * kPsLd + kb);
    const uint32_t bh1 = *reinterpret_cast<const uint32_t*>(p_hi + gid * kPsLd + kb + 8);
    const uint32_t bl0 = *reinterpret_cast<const uint32_t*>(p_lo + gid * kPsLd + kb);
    const uint32_t bl1 = *reinterpret_cast<const uint32_t*>(p_lo + gid * kPsLd + kb + 8);
    mma_bf16(oacc, a, bh0, bh1);
    mma_bf16(oacc, a, bl0, bl1);
  };
  constexpr int kHalfSteps = kHalf / 16;
  for (int j = kw; j < min(steps, kHalfSteps); j += C::WPT) pv_step(j);
  if (!Q4) {
    tc::cp_async_wait<0>();                     // V rows [kHalf, 2 kHalf)
    __syncthreads();
  }
  for (int j = kHalfSteps + kw % C::WPT; j < steps; j += C::WPT) pv_step(j);
  // oacc: O[query 2 tig (+1)][dimension 16 dt + gid (+8)]
  float* po = part_o + (int64_t)unit * kGm * D;
  const int q0 = 2 * tig;
  if (C::WPT == 1) {
    float* dst = po + 16 * dt + gid;
    if (q0 < G) {
      dst[q0 * D] = oacc[0];
      dst[q0 * D + 8] = oacc[2];
    }
    if (q0 + 1 < G) {
      dst[(q0 + 1) * D] = oacc[1];
      dst[(q0 + 1) * D + 8] = oacc[3];
    }
  } else {
    __syncthreads();                            // V rows read: warp partials in the row buffer
    float* wpart = reinterpret_cast<float*>(buf);   // [WPT][kGm][D]
    float* dst = wpart + (size_t)kw * kGm * D + 16 * dt + gid;
    dst[q0 * D] = oacc[0];
    dst[q0 * D + 8] = oacc[2];
    dst[(q0 + 1) * D] = oacc[1];
    dst[(q0 + 1) * D + 8] = oacc[3];
    __syncthreads();
    for (int i = t; i < G * D; i += kDecThreads) {
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < C::WPT; ++w) sum += wpart[(size_t)w * kGm * D + i];
      po[i] = sum;
    }
  }
  // arrival of this split (release: the CTA's writes, then the count); the
  // last one merges the pair's splits
  __syncthreads();
  if (t == 0) {
    __threadfence();
    const int prev = atomicAdd(&arrivals[cur.pair], 1);
    *last = prev == cur.nsplit - 1;
  }
  __syncthreads();
  if (!*last) return;
  __threadfence();
  const int ns = cur.nsplit;
  const float2* ml = part_ml + cur.u_first * kGm;
  constexpr int TPQ = D / 4;
  const int jq = t / TPQ, dq = 4 * (t % TPQ);   // thread: query jq, dimensions dq .. dq + 3
  float* wts = reinterpret_cast<float*>(buf);   // [kGm][32] split weights
  const float4* po4 = reinterpret_cast<const float4*>(part_o + cur.u_first * kGm * D + jq * D + dq);
  const size_t po4_step = (size_t)kGm * D / 4;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (ns <= 32) {
    // one load of the split states: lane s of warp jj holds split s of query jj
    if (warp < G) {
      const float2 v = lane < ns ? __ldcg(&ml[lane * kGm + warp]) : make_float2(-INFINITY, 0.f);
      float M = v.x;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      const float w = lane < ns && M > -INFINITY ? exp2f(v.x - M) : 0.f;
      float L = v.y * w;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
      wts[warp * 32 + lane] = w;
      if (lane == 0) cm[2 * warp + 1] = L > 0.f ? 1.f / L : 0.f;
    }
    __syncthreads();
    if (jq < G) {
#pragma unroll 16
      for (int i = 0; i < ns; ++i) {
        const float w = wts[jq * 32 + i];
        const float4 v = __ldcg(po4 + i * po4_step);
        acc.x = fmaf(v.x, w, acc.x);
        acc.y = fmaf(v.y, w, acc.y);
        acc.z = fmaf(v.z, w, acc.z);
        acc.w = fmaf(v.w, w, acc.w);
      }
    }
  } else {
    if (warp < G) {
      float M = -INFINITY;
      for (int s = lane; s < ns; s += 32) M = fmaxf(M, __ldcg(&ml[s * kGm + warp]).x);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      float L = 0.f;
      if (M > -INFINITY)
        for (int s = lane; s < ns; s += 32) {
          const float2 v = __ldcg(&ml[s * kGm + warp]);
          L = fmaf(v.y, exp2f(v.x - M), L);
        }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
      if (lane == 0) {
        cm[2 * warp] = M;
        cm[2 * warp + 1] = L > 0.f ? 1.f / L : 0.f;
      }
    }
    // 32 weights at a time
    for (int s0 = 0; s0 < ns; s0 += 32) {
      __syncthreads();
      if (warp < G) {
        const int s = s0 + lane;
        const float M = cm[2 * warp];
        wts[warp * 32 + lane] = s < ns && M > -INFINITY ? exp2f(__ldcg(&ml[s * kGm + warp]).x - M) : 0.f;
      }
      __syncthreads();
      if (jq < G) {
        const int cnt = min(32, ns - s0);
#pragma unroll 16
        for (int i = 0; i < cnt; ++i) {
          const float w = wts[jq * 32 + i];
          const float4 v = __ldcg(po4 + (size_t)(s0 + i) * po4_step);
          acc.x = fmaf(v.x, w, acc.x);
          acc.y = fmaf(v.y, w, acc.y);
          acc.z = fmaf(v.z, w, acc.z);
          acc.w = fmaf(v.w, w, acc.w);
        }
      }
    }
  }
  if (jq < G) {
    const float inv = cm[2 * jq + 1];
    __nv_bfloat16* dst = out + ((int64_t)cur.r * tb.Hq + cur.g * G + jq) * D + dq;
    *reinterpret_cast<uint2*>(dst) = make_uint2(pack_bf16(acc.x * inv, acc.y * inv),
                                                pack_bf16(acc.z * inv, acc.w * inv));
  }
}

// One warp per (request, query head): merge the splits of its KV head.  Lane
// s holds split s's state (s = lane, lane + 32, ...); the weighted partial
// outputs are then summed with several splits' loads in flight.
template <typename T, int D>
__global__ void __launch_bounds__(128) decode_combine_kernel(const __grid_constant__ DecodeTable tb,
                                                             const float* __restrict__ part_o,
                                                             const float2* __restrict__ part_ml,
                                                             T* __restrict__ out) {
  constexpr int EPL = D / 32;                   // output elements per lane
  const int w = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (w >= tb.n_req * tb.Hq) return;
  const int r = w / tb.Hq, j = w % tb.Hq;
  const DecodeReq rq = tb.req[r];
  const int g = j / tb.G, jj = j % tb.G;
  const int64_t u0 = rq.unit0 + (int64_t)g * rq.nsplit;
  const int ns = rq.B + rq.T > 0 ? rq.nsplit : 0;
  float M = -INFINITY;
  for (int s = lane; s < ns; s += 32) M = fmaxf(M, part_ml[(u0 + s) * kGm + jj].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float Lsum = 0.f;
  float acc[EPL];
#pragma unroll
  for (int i = 0; i < EPL; ++i) acc[i] = 0.f;
  for (int s0 = 0; s0 < ns; s0 += 32) {
    const int sl = s0 + lane;
    float wl = 0.f;
    if (sl < ns) {
      const float2 ml = part_ml[(u0 + sl) * kGm + jj];
      wl = exp2f(ml.x - M);
      Lsum = fmaf(ml.y, wl, Lsum);
    }
    const int cnt = min(32, ns - s0);
#pragma unroll 4
    for (int i = 0; i < cnt; ++i) {
      const float ws = __shfl_sync(0xffffffffu, wl, i);
      const float* o = part_o + ((u0 + s0 + i) * kGm + jj) * D + lane * EPL;
      if constexpr (EPL == 4) {
        const float4 v = *reinterpret_cast<const float4*>(o);
        acc[0] = fmaf(v.x, ws, acc[0]);
        acc[1] = fmaf(v.y, ws, acc[1]);
        acc[2] = fmaf(v.z, ws, acc[2]);
        acc[3] = fmaf(v.w, ws, acc[3]);
      } else {
        const float2 v = *reinterpret_cast<const float2*>(o);
        acc[0] = fmaf(v.x, ws, acc[0]);
        acc[1] = fmaf(v.y, ws, acc[1]);
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) Lsum += __shfl_xor_sync(0xffffffffu, Lsum, o);
  const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
  T* dst = out + ((int64_t)r * tb.Hq + j) * D + lane * EPL;
#pragma unroll
  for (int i = 0; i < EPL; ++i) dst[i] = Elem<T>::from_f(acc[i] * inv);
}

template <typename T, int D>
cudaError_t launch_decode_t(const DecodeTable& tb, const void* q, const void* Kc, const void* Vc,
                            const void* Kt, const void* Vt, void* out, float* part_o, float2* part_ml,
                            cudaStream_t st) {
  if (tb.units > 0) {
    constexpr size_t smem = DecCfg<T, D>::SMEM;
    static bool attr = false;
    if (!attr) {
      cudaError_t e = cudaFuncSetAttribute(decode_partial_kernel<T, D>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      // the whole unified L1 as shared memory: two CTAs per SM for bf16 rows
      e = cudaFuncSetAttribute(decode_partial_kernel<T, D>,
                               cudaFuncAttributePreferredSharedMemoryCarveout, 100);
      if (e != cudaSuccess) return e;
      attr = true;
    }
    ProfileScope ps("decode_partial", st);
    decode_partial_kernel<T, D><<<(unsigned)tb.units, kDecThreads, smem, st>>>(
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

template <int D, bool Q4>
cudaError_t launch_decode_mma(const DecodeTable& tb, const void* q, const void* Kc, const void* Vc,
                              const void* Kt, const void* Vt, const uint8_t* Kq, const uint8_t* Vq,
                              const float* Kqp, const float* Vqp, void* out, float* part_o,
                              float2* part_ml, int32_t* arrivals, cudaStream_t st) {
  using B16 = __nv_bfloat16;
  if (tb.units < 1) return cudaSuccess;
  constexpr size_t smem = MmaCfg<D>::SMEM;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(decode_mma_kernel<D, Q4>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    // the whole unified L1 as shared memory: three CTAs per SM
    e = cudaFuncSetAttribute(decode_mma_kernel<D, Q4>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaError_t e = cudaMemsetAsync(arrivals, 0, sizeof(int32_t) * tb.n_req * tb.Hkv, st);
  if (e != cudaSuccess) return e;
  ProfileScope ps(Q4 ? "decode_attn_kv4" : "decode_attn", st);
  decode_mma_kernel<D, Q4><<<(unsigned)tb.units, kDecThreads, smem, st>>>(
      tb, static_cast<const B16*>(q), static_cast<const B16*>(Kc), static_cast<const B16*>(Vc),
      static_cast<const B16*>(Kt), static_cast<const B16*>(Vt), Kq, Vq, Kqp, Vqp, part_o, part_ml,
      arrivals, static_cast<B16*>(out));
  return cudaGetLastError();
}

}  // namespace

int decode_split_keys(int dtype) { return dtype == VC_BF16 ? kSplitM : kSplitF; }

cudaError_t launch_decode(const DecodeTable& tb, int dtype, int d, const void* q, const void* Kc,
                          const void* Vc, const void* Kt, const void* Vt, void* out, float* part_o,
                          float2* part_ml, int32_t* arrivals, cudaStream_t st) {
  if (dtype == VC_BF16) {
    if (d == 128)
      return launch_decode_mma<128, false>(tb, q, Kc, Vc, Kt, Vt, nullptr, nullptr, nullptr, nullptr, out,
                                           part_o, part_ml, arrivals, st);
    return launch_decode_mma<64, false>(tb, q, Kc, Vc, Kt, Vt, nullptr, nullptr, nullptr, nullptr, out,
                                        part_o, part_ml, arrivals, st);
  }
  if (d == 128) return launch_decode_t<float, 128>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
  return launch_decode_t<float, 64>(tb, q, Kc, Vc, Kt, Vt, out, part_o, part_ml, st);
}

cudaError_t launch_decode_kv4(const DecodeTable& tb, int d, const void* q, const uint8_t* Kq,
                              const uint8_t* Vq, const float* Kqp, const float* Vqp, const void* Kt,
                              const void* Vt, void* out, float* part_o, float2* part_ml,
                              int32_t* arrivals, cudaStream_t st) {
  if (d == 128)
    return launch_decode_mma<128, true>(tb, q, nullptr, nullptr, Kt, Vt, Kq, Vq, Kqp, Vqp, out, part_o,
                                        part_ml, arrivals, st);
  return launch_decode_mma<64, true>(tb, q, nullptr, nullptr, Kt, Vt, Kq, Vq, Kqp, Vqp, out, part_o,
                                     part_ml, arrivals, st);
}

}  // namespace vc
