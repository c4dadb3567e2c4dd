// Shared definitions of libviscache: device-side plan tables, status word,
// element loads and small numeric helpers.  No PruneKV arithmetic lives here.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "viscache.h"

namespace vc {

// ---------------------------------------------------------------------------
// Device plan tables (built on the host, copied into the caller workspace).

struct Req {                 // one request of a batch
  int64_t kv_off;            // element offset of its K/V block [L][Hkv][n][d]
  int64_t q_off;             // element offset of its Qw block [L][Hq][W][d]
  int64_t lse_off;           // float offset of its row log-sum-exp block [L][Hq][W]
  int64_t s_off;             // float offset of its scores [Hkv][n] or [L][Hkv][n]
  int64_t out_row0;          // first output row (K_out/V_out/idx_out)
  int64_t drop_row0;         // first drop-list row
  int64_t lsep_off;          // float offset of its chunk-padded row normalisers [L][Hkv][C*cw]
  int64_t vs_row0;           // first row of its compacted survivors' values (tensor-core fusion)
  int32_t n, W, Nq, h;
  int32_t C;                 // column-sum chunks of one (layer, KV head) row set, ceil(G*W/256)
  int32_t cw;                // rows per chunk: G*W spread over C chunks, rounded up to 16
  int32_t nrb;               // 256-row blocks of that row set, ceil(G*W/256)
  int32_t tiles;             // 256-key tiles, ceil(n/256)
  int32_t chunk0;            // first 1024-key sort chunk of its first ranking problem
  int32_t Ls;                // layers whose scores are needed: L, or in the fused pass with
                             // per-layer ranking the leading layers with B_l > 0
};

struct Layer {               // one (request, layer)
  int32_t B;                 // budget B_l
  int32_t P;                 // sum_{j<l} B_j
  int32_t D;                 // drop count Nq - B_l (0 when B_l == 0)
  int32_t Qd;                // sum_{j<l} D_j
};

struct Shape {
  int32_t L, Hq, Hkv, d, G;
  int32_t n_req;
  int32_t rank_mode;
  float scale_log2;          // logit scale * log2(e)
  int32_t test_wait;         // VC_TEST_WAIT_* bits (test support, normally 0)
};

struct Tables {              // device pointers into the workspace
  const Req* req;            // [n_req]
  const Layer* layer;        // [n_req * L]
  const int32_t* unit0_lse;  // [n_req + 1] row-tile units of the lse pass
  const int32_t* unit0_col;  // [n_req + 1] key-tile units of the column-sum pass
  const int32_t* unit0_fuse; // [n_req * L + 1] kept-row-tile units x Hkv of the fusion
  const int64_t* row0_out;   // [n_req * L + 1] first output row of each (request, layer)
  const int32_t* unit0_tc1;  // [n_req + 1] CTAs of the tensor-core lse pass
  const int32_t* unit0_tc2;  // [n_req + 1] CTAs of the tensor-core column-sum pass
  const int32_t* unit0_fuse_tc;  // [n_req * L + 1] 256-row kept tiles x Hkv (tensor-core fusion)
  const int32_t* unit0_gather;   // [n_req * L + 1] 16-row survivor blocks x Hkv (row gather)
  int32_t* status;           // device status word
};

// ---------------------------------------------------------------------------
// Status word: first error wins.

__device__ __forceinline__ void set_status(int32_t* status, int32_t code) {
  atomicCAS(status, VC_OK, code);
}

// Largest i in [0, count) with prefix[i] <= key (prefix non-decreasing, prefix[0] = 0).
template <typename Int>
__device__ __forceinline__ int upper_index(const Int* prefix, int count, Int key) {
  int lo = 0, hi = count - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (prefix[mid] <= key) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// The same index found by a whole warp at once: it is the number of entries
// <= key, minus one (prefix is non-decreasing and prefix[0] = 0 <= key), so
// each lane counts a strided share and the warp sums the counts.  All loads
// are independent, so the lookup costs one memory latency instead of one per
// bisection step.  Every lane of the warp must call it; all get the result.
template <typename Int>
__device__ __forceinline__ int upper_index_warp(const Int* prefix, int count, Int key) {
  int c = 0;
  for (int i = (int)(threadIdx.x & 31); i < count; i += 32) c += prefix[i] <= key ? 1 : 0;
  return __reduce_add_sync(0xffffffffu, c) - 1;
}

// ---------------------------------------------------------------------------
// Element access.

template <typename T> struct Elem;
template <> struct Elem<float> {
  static __device__ __forceinline__ float load(const float* p) { return *p; }
  static __device__ __forceinline__ float to_f(float x) { return x; }
  static __device__ __forceinline__ float from_f(float x) { return x; }
};
template <> struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
  static __device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
  static __device__ __forceinline__ __nv_bfloat16 from_f(float x) { return __float2bfloat16_rn(x); }
};

// Load 4 consecutive elements as floats (16-byte aligned for float, 8 for bf16).
__device__ __forceinline__ float4 load4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ float4 load4(const __nv_bfloat16* p) {
  uint2 u = *reinterpret_cast<const uint2*>(p);
  float4 f;
  f.x = __uint_as_float(u.x << 16);
  f.y = __uint_as_float(u.x & 0xffff0000u);
  f.z = __uint_as_float(u.y << 16);
  f.w = __uint_as_float(u.y & 0xffff0000u);
  return f;
}

// Compensated (Kahan) accumulation: keeps long fp32 sums of positive terms
// accurate to a few ulp independent of the number of terms.
struct Kahan {
  float s, c;
  __device__ __forceinline__ void init() { s = 0.f; c = 0.f; }
  __device__ __forceinline__ void add(float x) {
    float y = x - c;
    float t = s + y;
    c = (t - s) - y;
    s = t;
  }
};

constexpr float kLog2e = 1.4426950408889634f;

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  The kernels after the first of a call are
// launched with launch_dep (kernels.h), so each may be scheduled while the
// kernel before it on the stream drains, and set up its shared and tensor
// memory and read the inputs meanwhile.  dep_wait() returns once the previous
// kernel of the stream has completed and its writes are visible; dep_launch()
// lets the next kernel be scheduled.  Each such kernel keeps two rules:
//  * a thread of every CTA returns from dep_wait() before the CTA reads what
//    the previous kernel wrote, or writes memory that kernel reads or writes;
//  * a CTA calls dep_launch() only in a thread that has returned from
//    dep_wait().
// So when a kernel is scheduled, every kernel before the previous one has
// completed: what those wrote (the plan tables, the ranks behind the keep
// lists) may be read before dep_wait().  Without the launch attribute both
// instructions return at once.
__device__ __forceinline__ void dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

}  // namespace vc
