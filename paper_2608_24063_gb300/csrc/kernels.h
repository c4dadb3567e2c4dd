// Launchers of the libviscache kernels (internal; the C ABI is include/viscache.h).
#pragma once

#include <cuda_runtime.h>

#include <atomic>

#include "vc_common.cuh"

namespace vc {

// 1 (default): launch_dep lets a kernel start while the one before it drains;
// 0 (viscache_set_dependent_launch, or built with VC_SERIAL_LAUNCH): every
// kernel waits for the previous one to complete, as an ordinary launch.
extern std::atomic<int> g_dependent_launch;

// Launches kernel on st so that it may be scheduled before the previous kernel
// on the stream has completed (programmatic stream serialisation); the kernel
// orders itself with dep_wait / dep_launch (vc_common.cuh).
template <typename... P, typename... A>
cudaError_t launch_dep(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       A&&... args) {
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = g_dependent_launch.load(std::memory_order_relaxed) ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<A&&>(args)...);
}

// Plan-table image passed by value (kernel parameters may hold up to 32 KB).
struct TableImage {
  alignas(16) uint8_t bytes[24 * 1024];
};
cudaError_t launch_upload(const TableImage& im, uint32_t bytes, uint8_t* dst, int32_t* status,
                          cudaStream_t st);

int score_rows_per_tile_simt();
int score_keys_per_tile_simt();
int fuse_rows_per_tile_simt();

// Eq. (token_score) on CUDA cores: lse pass (skipped when lse_nat != nullptr) + column sums.
cudaError_t launch_score_simt(int dtype, const void* Qw, const void* K, const Shape& sh,
                              const Tables& tb, int units_lse, int units_col, float* lse,
                              const float* lse_nat, float* scores, cudaStream_t st);

// Eq. (token_score) on tcgen05 tensor cores (bf16, d = 128): lse pass (skipped when
// lse_nat != nullptr), merge of key splits, column sums.
struct TcPlan {
  int units1;        // CTA pairs of the lse pass (sum over requests of L*Hkv*nrb*S)
  int units2;        // CTA pairs of the column-sum pass (sum of Hkv*tiles)
  int S;             // key splits of the lse pass
  int64_t q_rows;    // rows of the packed Qw tensor
  int64_t k_rows;    // rows of the packed K tensor
  int64_t max_rows;  // max over requests of L*Hq*W
  int64_t max_prows; // max over requests of L*Hkv*C*cw (chunk-padded rows)
};
int score_tc_max_splits();
int score_tc_pair_slots();
cudaError_t launch_score_tc(const void* Qw, const void* K, const Shape& sh, const Tables& tb,
                            const TcPlan& tp, float2* part, float* nlse_pad, const float* lse_nat,
                            float* scores, cudaStream_t st);

// bf16, d = 128: the survivors' values compacted into Vs (gather), then
// V_out = mu V_k + (1-mu) softmax(V_k V_d^T / tau) V_d on tcgen05.  K_out =
// K[keep] is copied by the fusion's own key warps (kcopy: K in device memory)
// or else by the gather.
int fuse_rows_per_tile_tc();
int gather_rows_per_block();
cudaError_t launch_fuse_tc(const void* K, const void* V, const Shape& sh, const Tables& tb,
                           const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                           void* K_out, void* V_out, void* Vs, int64_t vs_rows, bool kcopy,
                           int units_gather, int units, cudaStream_t st);

// Ranking (sorted 1024-key chunks, `chunks`: kSortChunk keys per chunk,
// Req::chunk0 locates a request's chunks) and ascending keep/drop compaction.
constexpr int kSortChunk = 1024;
cudaError_t launch_select(const Shape& sh, const Tables& tb, int n_problems, int max_chunks,
                          const float* scores, int32_t* rank, uint64_t* chunks, int32_t* keep_idx,
                          int32_t* drop_idx, cudaStream_t st);

// K_out = K[keep] (bit-exact), total_rows = Hkv * sum over requests and layers of B_l.
cudaError_t launch_gather_k(int dtype, const void* K, const Shape& sh, const Tables& tb,
                            const int32_t* keep_idx, void* K_out, int64_t total_rows,
                            cudaStream_t st);

// V_out = mu V_k + (1-mu) softmax(V_k V_d^T / tau) V_d on CUDA cores.
cudaError_t launch_fuse_simt(int dtype, const void* V, const Shape& sh, const Tables& tb,
                             const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                             void* V_out, int units, cudaStream_t st);

// Decode attention over the compressed cache of one layer (Sec. 2, after
// Sec. 3.2): per (request, KV head) the layer's B kept visual rows (dense
// varlen layout of prunekv_compress) then T text rows, split into chunks of
// decode_split_keys() keys; partial softmax states are merged per query head.
constexpr int kDecodeMaxReq = 256;
constexpr int kDecodeMaxGroup = 8;            // query heads per KV head
struct DecodeReq {
  int64_t vis_row0;        // first visual row of KV head 0 (rows g*B ... of head g)
  int64_t txt_row0;        // first text row of KV head 0 (rows g*T ... of head g)
  int32_t B, T;            // visual and text rows per KV head
  int32_t unit0;           // first (KV head, split) unit of the request
  int32_t nsplit;          // splits per KV head, max(1, ceil((B+T) / split keys))
  int64_t kg0;             // 4-bit cache: first key group of KV head 0 in this layer
  int32_t nkg;             // 4-bit cache: key groups per KV head, ceil(B / 32)
  int32_t pad;
};
struct DecodeTable {
  int32_t n_req, Hq, Hkv, G;
  float scale;
  int32_t split;           // keys per split (at most decode_split_keys(dtype))
  int32_t units;           // sum over requests of Hkv * nsplit
  DecodeReq req[kDecodeMaxReq];
};
int decode_split_keys(int dtype);   // the largest split a kernel takes
// Decode over the 4-bit form of the visual rows (viscache_kv4_quantize's
// codes and parameters; bf16 query, text rows and output).
cudaError_t launch_decode_kv4(const DecodeTable& tb, int d, const void* q, const uint8_t* Kq,
                              const uint8_t* Vq, const float* Kqp, const float* Vqp, const void* Kt,
                              const void* Vt, void* out, float* part_o, float2* part_ml,
                              int32_t* arrivals, cudaStream_t st);
cudaError_t launch_decode(const DecodeTable& tb, int dtype, int d, const void* q, const void* Kc,
                          const void* Vc, const void* Kt, const void* Vt, void* out, float* part_o,
                          float2* part_ml, int32_t* arrivals, cudaStream_t st);

// 4-bit quantisation of the compacted cache: per (request, layer) with B > 0,
// Hkv segments of B rows starting at row0 (KV head g at row0 + g * B); a
// unit is one group of up to kv4_group_rows() rows of one segment.
struct QuantEntry {
  int64_t row0;            // first row of the (request, layer)
  int32_t B;               // rows per KV head
  int32_t unit0;           // first unit of the entry within the launch
};
constexpr int kQuantMaxEntries = 1792;
struct QuantTable {
  int32_t n;               // entries
  int32_t pad;
  int64_t unit_base;       // global index of the launch's first key group
  QuantEntry e[kQuantMaxEntries];
};
int kv4_group_rows();
cudaError_t launch_kv4(const QuantTable& tb, int units, int dtype, int d, bool quantize,
                       const void* K, const void* V, uint8_t* Kc, uint8_t* Vc, float* Kp, float* Vp,
                       void* Kh, void* Vh, cudaStream_t st);

}  // namespace vc
