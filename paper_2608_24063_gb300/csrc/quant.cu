// 4-bit quantisation of the compacted cache (the Appendix "Quantization"
// combination: the compressed visual KV under a 4-bit KV cache quantiser) and
// its inverse.  Asymmetric round-to-nearest with a per-group scale and
// minimum:
//     scale = (max - min) / 15,  code = clamp(rint((x - min) / scale), 0, 15),
//     x_hat = code * scale + min  (one fused multiply-add),
// keys per channel over groups of 32 consecutive rows of one (request, layer,
// KV head) segment (the last group of a segment may be shorter), values per
// row over groups of 32 channels.  Codes are packed two per byte, the even
// channel in the low nibble; parameters are fp32 (scale, min) pairs.  The
// code is decided in fp32 with IEEE subtraction and division and rint.
//
// One warp per key group (up to 32 rows of one segment): for the keys lane t
// owns d/32 adjacent channels (vector loads of a row's piece, the codes
// stored as one 8- or 16-bit word, statistics per channel over the group's
// rows); for the values a lane owns one (row, 32-channel group) pair at a
// time (16-byte loads, its own statistics, 16 bytes of codes).  The work is a
// streaming pass (read 2 x 2 bytes, write 2 x ~0.75 bytes per element pair).
#include <cuda_bf16.h>
#include <stdint.h>

#include <type_traits>

#include "kernels.h"
#include "profile.h"
#include "vc_common.cuh"

namespace vc {
namespace {

constexpr int kGroup = 32;
constexpr int kQuantWarps = 4;                // key groups (one per warp) per CTA

__device__ __forceinline__ int find_entry(const QuantTable& tb, int unit) {
  int lo = 0, hi = tb.n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tb.e[mid].unit0 <= unit) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// rint((x - lo) / scale) with an IEEE quotient, clamped to [0, 15]; inv is
// the correctly rounded 1 / scale.  t = (x - lo) * inv is within 1.5 ulp of
// the exact quotient (the IEEE quotient within 0.5 ulp), so for |t| <= 16
// both lie within 4e-6 of it: unless t is within 1e-5 of a half-integer
// they round to the same integer, and only then is the division done.
__device__ __forceinline__ uint32_t code_of(float x, float lo, float scale, float inv) {
  if (!(scale > 0.f)) return 0u;
  const float a = __fsub_rn(x, lo);
  float t = __fmul_rn(a, inv);
  if (fabsf(t - floorf(t) - 0.5f) < 1e-5f || !(fabsf(t) <= 16.f)) t = __fdiv_rn(a, scale);
  return (uint32_t)fminf(fmaxf(rintf(t), 0.f), 15.f);
}

// Two codes with packed fp32 pairs, the same decision as code_of: t is
// rounded to nearest-even by adding 1.5 * 2^23 (exact for 0 <= t < 2^22, the
// integer then sits in the low bits of the sum); a code whose t lies within
// 1e-5 of a half-integer (|t - rint(t)| > 0.5 - 1e-5), outside [0, 16] or is
// NaN, or whose scale is not positive, is decided by code_of instead.
constexpr float kRound = 12582912.f;                 // 1.5 * 2^23
constexpr uint32_t kRoundBits = 0x4B400000u;
__device__ __forceinline__ void codes2(float2 x, float2 lo, float2 scale, float2 inv, uint32_t& q0,
                                       uint32_t& q1) {
  const float2 a = __fadd2_rn(x, make_float2(-lo.x, -lo.y));
  const float2 t = __fmul2_rn(a, inv);
  const float2 r = __fadd2_rn(t, make_float2(kRound, kRound));
  const float2 n = __fadd2_rn(r, make_float2(-kRound, -kRound));
  const float2 e = __fadd2_rn(t, make_float2(-n.x, -n.y));
  const bool f0 = scale.x > 0.f && t.x >= 0.f && t.x <= 16.f && fabsf(e.x) <= 0.5f - 1e-5f;
  const bool f1 = scale.y > 0.f && t.y >= 0.f && t.y <= 16.f && fabsf(e.y) <= 0.5f - 1e-5f;
  q0 = f0 ? min(__float_as_uint(r.x) - kRoundBits, 15u) : code_of(x.x, lo.x, scale.x, inv.x);
  q1 = f1 ? min(__float_as_uint(r.y) - kRoundBits, 15u) : code_of(x.y, lo.y, scale.y, inv.y);
}

// Elementwise minimum and maximum of bf16 pairs (exact: no rounding).
__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t u) {
  return *reinterpret_cast<const __nv_bfloat162*>(&u);
}

struct GroupRows {
  int64_t row;   // first row of the key group
  int nrows;     // rows in the group (1..32)
  int64_t kg;    // global index of the key group (its parameter row)
};
__device__ __forceinline__ GroupRows group_rows(const QuantTable& tb, int unit) {
  const QuantEntry e = tb.e[find_entry(tb, unit)];
  const int local = unit - e.unit0;
  const int nb = (e.B + kGroup - 1) / kGroup;
  const int g = local / nb, b = local % nb;
  GroupRows x;
  x.row = e.row0 + (int64_t)g * e.B + (int64_t)b * kGroup;
  x.nrows = min(kGroup, e.B - b * kGroup);
  x.kg = tb.unit_base + unit;
  return x;
}

// CPT adjacent channels of one row as floats (CPT = 2 or 4; 4 or 8 bf16 bytes,
// 8 or 16 fp32 bytes).
template <typename T, int CPT>
__device__ __forceinline__ void load_cpt(const T* p, float (&v)[CPT]);
template <>
__device__ __forceinline__ void load_cpt<__nv_bfloat16, 4>(const __nv_bfloat16* p, float (&v)[4]) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xffff0000u);
  v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_cpt<__nv_bfloat16, 2>(const __nv_bfloat16* p, float (&v)[2]) {
  const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
  v[0] = __uint_as_float(u << 16); v[1] = __uint_as_float(u & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_cpt<float, 4>(const float* p, float (&v)[4]) {
  const float4 u = *reinterpret_cast<const float4*>(p);
  v[0] = u.x; v[1] = u.y; v[2] = u.z; v[3] = u.w;
}
template <>
__device__ __forceinline__ void load_cpt<float, 2>(const float* p, float (&v)[2]) {
  const float2 u = *reinterpret_cast<const float2*>(p);
  v[0] = u.x; v[1] = u.y;
}

// CPT adjacent outputs of one row in one vector store (rounded to the type).
template <typename T, int CPT>
__device__ __forceinline__ void store_cpt(T* p, const float (&v)[CPT]);
template <>
__device__ __forceinline__ void store_cpt<__nv_bfloat16, 4>(__nv_bfloat16* p, const float (&v)[4]) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
  *reinterpret_cast<uint2*>(p) = make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
}
template <>
__device__ __forceinline__ void store_cpt<__nv_bfloat16, 2>(__nv_bfloat16* p, const float (&v)[2]) {
  *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(v[0], v[1]);
}
template <>
__device__ __forceinline__ void store_cpt<float, 4>(float* p, const float (&v)[4]) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
template <>
__device__ __forceinline__ void store_cpt<float, 2>(float* p, const float (&v)[2]) {
  *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
}

// CPT codes (even channel in the low nibble) as CPT / 2 bytes.
template <int CPT>
__device__ __forceinline__ void store_codes(uint8_t* dst, const uint32_t (&q)[CPT]) {
  if constexpr (CPT == 4)
    *reinterpret_cast<uint16_t*>(dst) = (uint16_t)(q[0] | (q[1] << 4) | (q[2] << 8) | (q[3] << 12));
  else
    *dst = (uint8_t)(q[0] | (q[1] << 4));
}

// One warp per key group: lane t owns channels CPT t .. CPT t + CPT - 1 of the
// group's rows for the keys (a pass over the rows for the per-channel minimum
// and maximum, then a second pass, the rows cache-resident, for the codes);
// for the values each lane takes whole (row, 32-channel group) pairs.
template <typename T, int D>
__global__ void __launch_bounds__(kQuantWarps * 32) quant_kernel(
    const __grid_constant__ QuantTable tb, int units, const T* __restrict__ K, const T* __restrict__ V,
    uint8_t* __restrict__ Kc, uint8_t* __restrict__ Vc, float2* __restrict__ Kp, float2* __restrict__ Vp) {
  constexpr int CPT = D / 32;
  const int unit = blockIdx.x * kQuantWarps + (threadIdx.x >> 5);
  if (unit >= units) return;
  const int lane = threadIdx.x & 31, c0 = lane * CPT;
  const GroupRows gr = group_rows(tb, unit);
  const T* kp = K + gr.row * D + c0;
  constexpr bool kBf16 = std::is_same<T, __nv_bfloat16>::value;
  float mn[CPT], mx[CPT];
  if constexpr (kBf16) {
    // per-channel minimum and maximum on bf16 pairs
    __nv_bfloat162 lo2[CPT / 2], hi2[CPT / 2];
#pragma unroll
    for (int j = 0; j < CPT / 2; ++j) {
      lo2[j] = __floats2bfloat162_rn(INFINITY, INFINITY);
      hi2[j] = __floats2bfloat162_rn(-INFINITY, -INFINITY);
    }
#pragma unroll 8
    for (int i = 0; i < gr.nrows; ++i) {
      uint32_t w[CPT / 2];
      if constexpr (CPT == 4) {
        const uint2 u = *reinterpret_cast<const uint2*>(kp + i * D);
        w[0] = u.x;
        w[CPT / 2 - 1] = u.y;
      } else {
        w[0] = *reinterpret_cast<const uint32_t*>(kp + i * D);
      }
#pragma unroll
      for (int j = 0; j < CPT / 2; ++j) {
        lo2[j] = __hmin2(lo2[j], as_bf162(w[j]));
        hi2[j] = __hmax2(hi2[j], as_bf162(w[j]));
      }
    }
#pragma unroll
    for (int j = 0; j < CPT / 2; ++j) {
      const float2 l = __bfloat1622float2(lo2[j]), h = __bfloat1622float2(hi2[j]);
      mn[2 * j] = l.x;
      mn[2 * j + 1] = l.y;
      mx[2 * j] = h.x;
      mx[2 * j + 1] = h.y;
    }
  } else {
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
      mn[j] = INFINITY;
      mx[j] = -INFINITY;
    }
#pragma unroll 8
    for (int i = 0; i < gr.nrows; ++i) {
      float v[CPT];
      load_cpt<T, CPT>(kp + i * D, v);
#pragma unroll
      for (int j = 0; j < CPT; ++j) {
        mn[j] = fminf(mn[j], v[j]);
        mx[j] = fmaxf(mx[j], v[j]);
      }
    }
  }
  float ks[CPT], ki[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) {
    ks[j] = __fdiv_rn(__fsub_rn(mx[j], mn[j]), 15.f);
    ki[j] = ks[j] > 0.f ? __frcp_rn(ks[j]) : 0.f;
    Kp[gr.kg * D + c0 + j] = make_float2(ks[j], mn[j]);
  }
  uint8_t* kc = Kc + gr.row * (D / 2) + c0 / 2;
#pragma unroll 8
  for (int i = 0; i < gr.nrows; ++i) {
    float v[CPT];
    load_cpt<T, CPT>(kp + i * D, v);
    uint32_t q[CPT];
#pragma unroll
    for (int j = 0; j < CPT; j += 2)
      codes2(make_float2(v[j], v[j + 1]), make_float2(mn[j], mn[j + 1]), make_float2(ks[j], ks[j + 1]),
             make_float2(ki[j], ki[j + 1]), q[j], q[j + 1]);
    store_codes<CPT>(kc + i * (D / 2), q);
  }
  // values: lane (row i, 32-channel group gv) takes the group whole (NG groups
  // a row, 32 / NG rows a pass): 16-byte loads, its own minimum and maximum,
  // 16 bytes of codes
  constexpr int NG = D / kGroup, RPP = 32 / NG;
  const int gv = lane % NG;
  for (int i = lane / NG; i < gr.nrows; i += RPP) {
    float v[kGroup];
    const T* src = V + (gr.row + i) * D + gv * kGroup;
    float lo, hi;
    if constexpr (kBf16) {
      // the group's 32 values as 16 bf16 pairs: minimum and maximum on pairs
      uint32_t w[kGroup / 2];
#pragma unroll
      for (int k = 0; k < kGroup / 2; k += 4) {
        const uint4 u = *reinterpret_cast<const uint4*>(src + 2 * k);
        w[k] = u.x; w[k + 1] = u.y; w[k + 2] = u.z; w[k + 3] = u.w;
      }
      __nv_bfloat162 l2 = as_bf162(w[0]), h2 = as_bf162(w[0]);
#pragma unroll
      for (int k = 1; k < kGroup / 2; ++k) {
        l2 = __hmin2(l2, as_bf162(w[k]));
        h2 = __hmax2(h2, as_bf162(w[k]));
      }
      const float2 lf = __bfloat1622float2(l2), hf = __bfloat1622float2(h2);
      lo = fminf(lf.x, lf.y);
      hi = fmaxf(hf.x, hf.y);
#pragma unroll
      for (int k = 0; k < kGroup / 2; ++k) {
        v[2 * k] = __uint_as_float(w[k] << 16);
        v[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
      }
    } else {
#pragma unroll
      for (int k = 0; k < kGroup; k += CPT) {
        float u[CPT];
        load_cpt<T, CPT>(src + k, u);
#pragma unroll
        for (int j = 0; j < CPT; ++j) v[k + j] = u[j];
      }
      lo = v[0];
      hi = v[0];
#pragma unroll
      for (int k = 1; k < kGroup; ++k) {
        lo = fminf(lo, v[k]);
        hi = fmaxf(hi, v[k]);
      }
    }
    const float vs = __fdiv_rn(__fsub_rn(hi, lo), 15.f);
    const float vi = vs > 0.f ? __frcp_rn(vs) : 0.f;
    Vp[(gr.row + i) * NG + gv] = make_float2(vs, lo);
    uint32_t w[4];
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      w[b] = 0u;
#pragma unroll
      for (int k = 0; k < 8; k += 2) {
        uint32_t q0, q1;
        codes2(make_float2(v[8 * b + k], v[8 * b + k + 1]), make_float2(lo, lo), make_float2(vs, vs),
               make_float2(vi, vi), q0, q1);
        w[b] |= (q0 << (4 * k)) | (q1 << (4 * k + 4));
      }
    }
    *reinterpret_cast<uint4*>(Vc + (gr.row + i) * (D / 2) + gv * (kGroup / 2)) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(kQuantWarps * 32) dequant_kernel(
    const __grid_constant__ QuantTable tb, int units, const uint8_t* __restrict__ Kc,
    const uint8_t* __restrict__ Vc, const float2* __restrict__ Kp, const float2* __restrict__ Vp,
    T* __restrict__ Kh, T* __restrict__ Vh) {
  constexpr int CPT = D / 32, TPG = kGroup / CPT;
  const int unit = blockIdx.x * kQuantWarps + (threadIdx.x >> 5);
  if (unit >= units) return;
  const int lane = threadIdx.x & 31, c0 = lane * CPT;
  const GroupRows gr = group_rows(tb, unit);
  float2 kpar[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) kpar[j] = Kp[gr.kg * D + c0 + j];
#pragma unroll 4
  for (int i = 0; i < gr.nrows; ++i) {
    const int64_t r = gr.row + i;
    uint32_t kb, vb;
    if constexpr (CPT == 4) {
      kb = *reinterpret_cast<const uint16_t*>(Kc + r * (D / 2) + c0 / 2);
      vb = *reinterpret_cast<const uint16_t*>(Vc + r * (D / 2) + c0 / 2);
    } else {
      kb = Kc[r * (D / 2) + c0 / 2];
      vb = Vc[r * (D / 2) + c0 / 2];
    }
    const float2 vpar = Vp[r * (D / kGroup) + lane / TPG];
    float kx[CPT], vx[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
      kx[j] = fmaf((float)((kb >> (4 * j)) & 15u), kpar[j].x, kpar[j].y);
      vx[j] = fmaf((float)((vb >> (4 * j)) & 15u), vpar.x, vpar.y);
    }
    store_cpt<T, CPT>(Kh + r * D + c0, kx);
    store_cpt<T, CPT>(Vh + r * D + c0, vx);
  }
}

template <typename T, int D>
cudaError_t launch_t(const QuantTable& tb, int units, bool quantize, const void* K, const void* V,
                     uint8_t* Kc, uint8_t* Vc, float* Kp, float* Vp, void* Kh, void* Vh,
                     cudaStream_t st) {
  const unsigned grid = (unsigned)((units + kQuantWarps - 1) / kQuantWarps);
  if (quantize) {
    ProfileScope ps("kv4_quantize", st);
    quant_kernel<T, D><<<grid, kQuantWarps * 32, 0, st>>>(tb, units, static_cast<const T*>(K),
                                                          static_cast<const T*>(V), Kc, Vc,
                                                          reinterpret_cast<float2*>(Kp),
                                                          reinterpret_cast<float2*>(Vp));
  } else {
    ProfileScope ps("kv4_dequantize", st);
    dequant_kernel<T, D><<<grid, kQuantWarps * 32, 0, st>>>(
        tb, units, Kc, Vc, reinterpret_cast<const float2*>(Kp), reinterpret_cast<const float2*>(Vp),
        static_cast<T*>(Kh), static_cast<T*>(Vh));
  }
  return cudaGetLastError();
}

}  // namespace

int kv4_group_rows() { return kGroup; }

cudaError_t launch_kv4(const QuantTable& tb, int units, int dtype, int d, bool quantize,
                       const void* K, const void* V, uint8_t* Kc, uint8_t* Vc, float* Kp, float* Vp,
                       void* Kh, void* Vh, cudaStream_t st) {
  if (units < 1) return cudaSuccess;
  if (dtype == VC_BF16) {
    if (d == 128) return launch_t<__nv_bfloat16, 128>(tb, units, quantize, K, V, Kc, Vc, Kp, Vp, Kh, Vh, st);
    return launch_t<__nv_bfloat16, 64>(tb, units, quantize, K, V, Kc, Vc, Kp, Vp, Kh, Vh, st);
  }
  if (d == 128) return launch_t<float, 128>(tb, units, quantize, K, V, Kc, Vc, Kp, Vp, Kh, Vh, st);
  return launch_t<float, 64>(tb, units, quantize, K, V, Kc, Vc, Kp, Vp, Kh, Vh, st);
}

}  // namespace vc
