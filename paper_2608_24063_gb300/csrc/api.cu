// C ABI of libviscache (declared in include/viscache.h): argument checks,
// workspace layout, device plan tables and kernel launches.  Every step of
// the pass runs in this library's kernels; nothing here computes on the host
// except the integer budget plan and the table offsets.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <vector>

#include "kernels.h"
#include "vc_common.cuh"

namespace vc {

// Programmatic dependent launches between the kernels of a call (launch_dep);
// 0 launches every kernel fully serialised.
#ifdef VC_SERIAL_LAUNCH
std::atomic<int> g_dependent_launch{0};
#else
std::atomic<int> g_dependent_launch{1};
#endif

namespace {

constexpr size_t kAlign = 256;

// Kernel path: VC_PATH_AUTO uses the tcgen05 score kernels for bf16, d = 128.
std::atomic<int> g_path{VC_PATH_AUTO};
// Test support: kernels whose next launches add one wait that must give up.
std::atomic<int> g_test_wait{0};

inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Sequential carving of the caller workspace into 256-byte aligned regions.
struct Arena {
  size_t off = 0;
  size_t take(size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes);
    return o;
  }
};

struct RequestPlan {
  int32_t n = 0, W = 0, Nq = 0, h = 0;
  std::vector<int32_t> B;
};

// Host image of the device tables plus the workspace offsets of every region.
struct Layout {
  // inputs
  int n_req = 0, L = 0, Hq = 0, Hkv = 0, d = 0, rank_mode = VC_RANK_SHARED;
  bool need_lse = false, need_scores = false, need_sort = false, need_drop = false, need_vs = false;
  bool prune_layers = false;   // score and rank only the layers the budgets keep (fused pass)
  // tensor-core score plan
  int S = 1;
  int64_t q_rows = 0, k_rows = 0, max_rows = 0, prows = 0, max_prows = 0;
  std::vector<int32_t> u_tc1, u_tc2, base_tc1, u_fuse_tc, u_gather;
  int units_fuse_tc = 0, units_gather = 0;
  int64_t vs_rows = 0;
  int max_n = 0;
  int64_t total_chunks = 0;
  int max_chunks = 0;
  // derived sizes
  int64_t lse_elems = 0, score_elems = 0, out_rows = 0, drop_rows = 0;
  int units_lse = 0, units_col = 0, units_fuse = 0;
  // workspace offsets
  size_t o_status = 0, o_req = 0, o_layer = 0, o_u_lse = 0, o_u_col = 0, o_u_fuse = 0,
         o_row0 = 0, o_u_tc1 = 0, o_u_tc2 = 0, o_u_fuse_tc = 0, o_u_gather = 0, o_vs = 0, table_begin = 0, table_end = 0, o_lse = 0,
         o_part = 0, o_lsep = 0, o_scores = 0, o_chunks = 0, o_rank = 0, o_drop = 0, total = 0;
  // host images
  std::vector<Req> req;
  std::vector<Layer> layer;
  std::vector<int32_t> u_lse, u_col, u_fuse;
  std::vector<int64_t> row0;

  void build(const std::vector<RequestPlan>& plans) {
    n_req = (int)plans.size();
    const int G = Hq > 0 && Hkv > 0 ? Hq / Hkv : 1;
    req.assign(n_req, Req{});
    layer.assign((size_t)n_req * L, Layer{});
    u_lse.assign(n_req + 1, 0);
    u_col.assign(n_req + 1, 0);
    u_fuse.assign((size_t)n_req * L + 1, 0);
    row0.assign((size_t)n_req * L + 1, 0);
    u_tc1.assign(n_req + 1, 0);
    u_fuse_tc.assign((size_t)n_req * L + 1, 0);
    u_gather.assign((size_t)n_req * L + 1, 0);
    vs_rows = 0;
    max_n = 0;
    total_chunks = 0;
    max_chunks = 0;
    u_tc2.assign(n_req + 1, 0);
    base_tc1.assign(n_req, 0);
    q_rows = k_rows = max_rows = prows = max_prows = 0;
    int64_t cu_n = 0, cu_w = 0;
    const int per_req_problems = rank_mode == VC_RANK_PER_LAYER ? L * Hkv : Hkv;
    const int rows_tile = score_rows_per_tile_simt(), keys_tile = score_keys_per_tile_simt();
    const int fuse_tile = fuse_rows_per_tile_simt();
    const int fuse_tile_tc = fuse_rows_per_tile_tc();
    const int gather_rows = gather_rows_per_block();
    for (int r = 0; r < n_req; ++r) {
      const RequestPlan& p = plans[r];
      Req& q = req[r];
      q.kv_off = (int64_t)L * Hkv * d * cu_n;
      q.q_off = (int64_t)L * Hq * d * cu_w;
      q.lse_off = (int64_t)L * Hq * cu_w;
      q.s_off = (int64_t)per_req_problems * cu_n;
      q.out_row0 = out_rows;
      q.drop_row0 = drop_rows;
      q.n = p.n; q.W = p.W; q.Nq = p.Nq; q.h = p.h;
      q.C = (G * p.W + 255) / 256;
      q.cw = 16 * ((G * p.W + 16 * q.C - 1) / (16 * q.C));
      q.lsep_off = prows;
      q.vs_row0 = vs_rows;
      max_n = std::max(max_n, p.n);
      {
        const int chunks = (p.n + kSortChunk - 1) / kSortChunk;
        q.chunk0 = (int32_t)total_chunks;
        total_chunks += (int64_t)per_req_problems * chunks;
        max_chunks = std::max(max_chunks, chunks);
      }
      prows += (int64_t)L * Hkv * q.C * q.cw;
      max_prows = std::max<int64_t>(max_prows, (int64_t)L * Hkv * q.C * q.cw);
      q.nrb = (G * p.W + 255) / 256;
      q.tiles = (p.n + 255) / 256;
      // per-layer ranking needs no scores of evicted layers (B_l = 0: a suffix,
      // budgets are non-increasing); the shared ranking averages all layers
      q.Ls = L;
      if (prune_layers && rank_mode == VC_RANK_PER_LAYER && !p.B.empty()) {
        q.Ls = 0;
        for (int l = 0; l < L; ++l)
          if (p.B[l] > 0) q.Ls = l + 1;
      }
      base_tc1[r] = q.Ls * Hkv * q.nrb;
      u_tc2[r + 1] = u_tc2[r] + (q.Ls > 0 ? Hkv * q.tiles : 0);
      q_rows += (int64_t)L * Hq * p.W;
      k_rows += (int64_t)L * Hkv * p.n;
      max_rows = std::max<int64_t>(max_rows, (int64_t)L * Hq * p.W);
      u_lse[r + 1] = u_lse[r] + (G * p.W + rows_tile - 1) / rows_tile;
      u_col[r + 1] = u_col[r] + (p.n + keys_tile - 1) / keys_tile;
      int32_t P = 0, Qd = 0;
      for (int l = 0; l < L; ++l) {
        const size_t rl = (size_t)r * L + l;
        const int32_t b = p.B.empty() ? 0 : p.B[l];
        Layer& ly = layer[rl];
        ly.B = b; ly.P = P; ly.D = b > 0 ? p.Nq - b : 0; ly.Qd = Qd;
        row0[rl] = out_rows + (int64_t)Hkv * P;
        u_fuse[rl + 1] = u_fuse[rl] + Hkv * ((b + fuse_tile - 1) / fuse_tile);
        u_fuse_tc[rl + 1] = u_fuse_tc[rl] + Hkv * ((b + fuse_tile_tc - 1) / fuse_tile_tc);
        u_gather[rl + 1] = u_gather[rl] + Hkv * ((b + ly.D + gather_rows - 1) / gather_rows);
        vs_rows += (int64_t)Hkv * (b + ly.D);
        P += b;
        Qd += ly.D;
      }
      out_rows += (int64_t)Hkv * P;
      drop_rows += (int64_t)Hkv * Qd;
      cu_n += p.n;
      cu_w += p.W;
    }
    row0[(size_t)n_req * L] = out_rows;
    lse_elems = (int64_t)L * Hq * cu_w;
    score_elems = (int64_t)per_req_problems * cu_n;
    units_lse = u_lse[n_req];
    units_col = u_col[n_req];
    units_fuse = u_fuse[(size_t)n_req * L];
    units_fuse_tc = u_fuse_tc[(size_t)n_req * L];
    units_gather = u_gather[(size_t)n_req * L];
    set_splits(1);

    Arena a;
    o_status = a.take(kAlign);
    table_begin = a.off;
    o_req = a.take(sizeof(Req) * n_req);
    o_layer = a.take(sizeof(Layer) * layer.size());
    o_u_lse = a.take(sizeof(int32_t) * u_lse.size());
    o_u_col = a.take(sizeof(int32_t) * u_col.size());
    o_u_fuse = a.take(sizeof(int32_t) * u_fuse.size());
    o_row0 = a.take(sizeof(int64_t) * row0.size());
    o_u_tc1 = a.take(sizeof(int32_t) * u_tc1.size());
    o_u_tc2 = a.take(sizeof(int32_t) * u_tc2.size());
    o_u_fuse_tc = a.take(sizeof(int32_t) * u_fuse_tc.size());
    o_u_gather = a.take(sizeof(int32_t) * u_gather.size());
    table_end = a.off;
    if (need_lse) {
      // CUDA-core path: lse rows; tensor-core path: split partials (same region)
      // and the chunk-padded normalisers
      o_lse = o_part = a.take(sizeof(float2) * lse_elems * score_tc_max_splits());
      o_lsep = a.take(sizeof(float) * prows);
    }
    if (need_scores) o_scores = a.take(sizeof(float) * score_elems);
    if (need_sort) {
      o_chunks = a.take(sizeof(uint64_t) * kSortChunk * std::max<int64_t>(total_chunks, 1));
      if (need_scores) o_rank = a.take(sizeof(int32_t) * score_elems);
    }
    if (need_drop) o_drop = a.take(sizeof(int32_t) * drop_rows);
    if (need_vs) o_vs = a.take((size_t)256 * std::max<int64_t>(vs_rows, 1));
    total = a.off;
  }

  // Key splits of the tensor-core lse pass: pick S in [1, max] that fills the
  // last wave of CTA pairs best (`slots` pairs resident at once); ties go to
  // the smaller S.
  void set_splits(int s) {
    S = s;
    for (int r = 0; r < n_req; ++r) u_tc1[r + 1] = u_tc1[r] + base_tc1[r] * S;
  }
  void choose_splits(int slots) {
    int best = 1;
    double best_eff = -1.0;
    for (int s = 1; s <= score_tc_max_splits(); ++s) {
      int64_t units = 0;
      for (int r = 0; r < n_req; ++r) units += (int64_t)base_tc1[r] * s;
      const int64_t waves = (units + slots - 1) / slots;
      const double eff = (double)units / (double)(waves * slots);
      if (eff > best_eff + 1e-9) { best_eff = eff; best = s; }
    }
    set_splits(best);
  }

  TcPlan tc_plan() const {
    TcPlan t;
    t.units1 = u_tc1[n_req];
    t.units2 = u_tc2[n_req];
    t.S = S;
    t.q_rows = q_rows;
    t.k_rows = k_rows;
    t.max_rows = max_rows;
    t.max_prows = max_prows;
    return t;
  }

  // Copy the table image into the workspace and clear the status word.  Small
  // images (every single request and typical batches) travel as a kernel
  // parameter, so the upload is an ordinary launch on the stream (no host
  // blocking, capturable in a CUDA graph); larger ones use one memcpy, and
  // then an upload of no bytes clears the status word, so that the kernels
  // after it always follow a kernel (their dependent launches order
  // themselves on the kernel before them).
  cudaError_t upload(uint8_t* ws, cudaStream_t st) const {
    const size_t bytes = table_end - table_begin;
    int32_t* status = reinterpret_cast<int32_t*>(ws + o_status);
    if (bytes <= sizeof(TableImage::bytes)) {
      TableImage im;
      memset(&im, 0, sizeof(im));
      fill(im.bytes);
      return launch_upload(im, (uint32_t)bytes, ws + table_begin, status, st);
    }
    std::vector<uint8_t> img(bytes, 0);
    fill(img.data());
    cudaError_t e = cudaMemcpyAsync(ws + table_begin, img.data(), bytes, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return e;
    static const TableImage none = {};
    return launch_upload(none, 0u, ws + table_begin, status, st);
  }

  void fill(uint8_t* img) const {
    auto put = [&](size_t off, const void* src, size_t n) {
      if (n) memcpy(img + (off - table_begin), src, n);
    };
    put(o_req, req.data(), sizeof(Req) * req.size());
    put(o_layer, layer.data(), sizeof(Layer) * layer.size());
    put(o_u_lse, u_lse.data(), sizeof(int32_t) * u_lse.size());
    put(o_u_col, u_col.data(), sizeof(int32_t) * u_col.size());
    put(o_u_fuse, u_fuse.data(), sizeof(int32_t) * u_fuse.size());
    put(o_row0, row0.data(), sizeof(int64_t) * row0.size());
    put(o_u_tc1, u_tc1.data(), sizeof(int32_t) * u_tc1.size());
    put(o_u_tc2, u_tc2.data(), sizeof(int32_t) * u_tc2.size());
    put(o_u_fuse_tc, u_fuse_tc.data(), sizeof(int32_t) * u_fuse_tc.size());
    put(o_u_gather, u_gather.data(), sizeof(int32_t) * u_gather.size());
  }

  Tables tables(uint8_t* ws) const {
    Tables t;
    t.req = reinterpret_cast<const Req*>(ws + o_req);
    t.layer = reinterpret_cast<const Layer*>(ws + o_layer);
    t.unit0_lse = reinterpret_cast<const int32_t*>(ws + o_u_lse);
    t.unit0_col = reinterpret_cast<const int32_t*>(ws + o_u_col);
    t.unit0_fuse = reinterpret_cast<const int32_t*>(ws + o_u_fuse);
    t.row0_out = reinterpret_cast<const int64_t*>(ws + o_row0);
    t.unit0_tc1 = reinterpret_cast<const int32_t*>(ws + o_u_tc1);
    t.unit0_tc2 = reinterpret_cast<const int32_t*>(ws + o_u_tc2);
    t.unit0_fuse_tc = reinterpret_cast<const int32_t*>(ws + o_u_fuse_tc);
    t.unit0_gather = reinterpret_cast<const int32_t*>(ws + o_u_gather);
    t.status = reinterpret_cast<int32_t*>(ws + o_status);
    return t;
  }

  Shape shape(float scale) const {
    Shape s;
    s.L = L; s.Hq = Hq; s.Hkv = Hkv; s.d = d; s.G = (Hq > 0 && Hkv > 0) ? Hq / Hkv : 1;
    s.n_req = n_req;
    s.rank_mode = rank_mode;
    s.scale_log2 = scale * kLog2e;
    s.test_wait = g_test_wait.load();
    return s;
  }
};

// Eq. (token_score) through the tensor-core kernels (bf16, d = 128) or the CUDA-core ones.
cudaError_t launch_score(int dtype, const void* Qw, const void* K, Layout& lay, float scale,
                         uint8_t* w, const float* row_lse, float* scores, cudaStream_t st) {
  const bool tc = g_path.load() == VC_PATH_AUTO && dtype == VC_BF16 && lay.d == 128;
  if (tc) lay.choose_splits(score_tc_pair_slots());
  cudaError_t e = lay.upload(w, st);
  if (e != cudaSuccess) return e;
  const Shape sh = lay.shape(scale);
  const Tables tb = lay.tables(w);
  float* lse = reinterpret_cast<float*>(w + lay.o_lse);
  if (tc)
    return launch_score_tc(Qw, K, sh, tb, lay.tc_plan(), reinterpret_cast<float2*>(w + lay.o_part),
                           reinterpret_cast<float*>(w + lay.o_lsep), row_lse, scores, st);
  return launch_score_simt(dtype, Qw, K, sh, tb, lay.units_lse, lay.units_col, lse, row_lse,
                           scores, st);
}

// True when p is ordinary device memory (the fusion's key warps read K only
// then; host or managed memory is left to the gather kernel).
bool on_device(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice;
}

// Prune keys and fuse values, Eq. (redistribution, weight_fusion): one tensor-core
// kernel for bf16, d = 128 (it also copies the kept keys), else the key gather and
// the CUDA-core fusion.
cudaError_t launch_fuse(int dtype, const void* K, const void* V, const Layout& lay,
                        const Shape& sh, const Tables& tb, const int32_t* keep, const int32_t* drop,
                        float mu, float tau, void* K_out, void* V_out, uint8_t* w, cudaStream_t st) {
  if (g_path.load() == VC_PATH_AUTO && dtype == VC_BF16 && lay.d == 128 && lay.need_vs)
    return launch_fuse_tc(K, V, sh, tb, keep, drop, mu, tau, K_out, V_out, w + lay.o_vs,
                          lay.vs_rows, on_device(K), lay.units_gather, lay.units_fuse_tc, st);
  cudaError_t e = launch_gather_k(dtype, K, sh, tb, keep, K_out, lay.out_rows, st);
  if (e != cudaSuccess) return e;
  return launch_fuse_simt(dtype, V, sh, tb, keep, drop, mu, tau, V_out, lay.units_fuse, st);
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool valid_model(int dtype, int L, int Hq, int Hkv, int d) {
  if (dtype != VC_BF16 && dtype != VC_F32) return false;
  if (L < 1 || L > 256 || Hkv < 1 || Hq < Hkv || Hq % Hkv != 0) return false;
  return d == 64 || d == 128;
}

int check_ws(const void* ws, size_t ws_bytes, size_t need) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return VC_ERR_WORKSPACE;
  return ws_bytes < need ? VC_ERR_WORKSPACE : VC_OK;
}

inline int cuda_status(cudaError_t e) { return e == cudaSuccess ? VC_OK : VC_ERR_CUDA; }

// Budgets B (host) must satisfy 0 <= B_l <= Nq <= n.
bool valid_budgets(const int32_t* B, int L, int Nq, int n) {
  if (!B || Nq < 0 || Nq > n) return false;
  for (int l = 0; l < L; ++l)
    if (B[l] < 0 || B[l] > Nq) return false;
  return true;
}

Layout score_layout(int L, int Hq, int Hkv, int d, int n, int W, int rank_mode) {
  Layout lay;
  lay.L = L; lay.Hq = Hq; lay.Hkv = Hkv; lay.d = d; lay.rank_mode = rank_mode;
  lay.need_lse = true;
  RequestPlan p;
  p.n = n; p.W = W;
  lay.build({p});
  return lay;
}

Layout select_layout(int L, int Hkv, int n, const int32_t* B, int Nq, int rank_mode) {
  Layout lay;
  lay.L = L; lay.Hq = Hkv; lay.Hkv = Hkv; lay.d = 64; lay.rank_mode = rank_mode;
  lay.need_sort = true;
  RequestPlan p;
  p.n = n; p.W = 1; p.Nq = Nq;
  if (B) p.B.assign(B, B + L);
  lay.build({p});
  return lay;
}

Layout fuse_layout(int L, int Hkv, int d, int n, const int32_t* B, int Nq) {
  Layout lay;
  lay.L = L; lay.Hq = Hkv; lay.Hkv = Hkv; lay.d = d;
  lay.need_vs = d == 128;
  RequestPlan p;
  p.n = n; p.W = 1; p.Nq = Nq;
  if (B) p.B.assign(B, B + L);
  lay.build({p});
  return lay;
}

int plan_batch(const vc_batch* b, const vc_params* p, std::vector<RequestPlan>* plans) {
  if (!b || !p || b->n_req < 1 || !b->n_vis || !b->W || !b->rr_num || !b->rr_den)
    return VC_ERR_INVALID_ARG;
  if (!valid_model(p->dtype, p->L, p->Hq, p->Hkv, p->d)) return VC_ERR_INVALID_ARG;
  if (p->rank_mode != VC_RANK_SHARED && p->rank_mode != VC_RANK_PER_LAYER) return VC_ERR_INVALID_ARG;
  if (!(p->mu >= 0.f && p->mu <= 1.f) || !(p->tau > 0.f) || !(p->scale >= 0.f))
    return VC_ERR_INVALID_ARG;
  if (p->schedule < VC_SCHED_PARABOLA || p->schedule > VC_SCHED_GEOMETRIC) return VC_ERR_INVALID_ARG;
  if (p->drop_mode != VC_DROP_SURVIVORS && p->drop_mode != VC_DROP_ALL) return VC_ERR_INVALID_ARG;
  // The plans depend only on these numbers; a caller that repeats a batch (a
  // decode step calls once per layer) gets the previous plans back.
  thread_local std::vector<int64_t> last_key;
  thread_local std::vector<RequestPlan> last_plans;
  std::vector<int64_t> key = {b->n_req, p->L, p->h, p->m_num, p->m_den, p->schedule, p->drop_mode};
  key.reserve(key.size() + 4 * (size_t)b->n_req);
  for (int r = 0; r < b->n_req; ++r) {
    key.push_back(b->n_vis[r]);
    key.push_back(b->W[r]);
    key.push_back(b->rr_num[r]);
    key.push_back(b->rr_den[r]);
  }
  if (key == last_key) {
    *plans = last_plans;
    return VC_OK;
  }
  plans->assign(b->n_req, RequestPlan{});
  for (int r = 0; r < b->n_req; ++r) {
    RequestPlan& q = (*plans)[r];
    q.n = b->n_vis[r];
    q.W = b->W[r];
    if (q.n < 1 || q.n > 65536 || q.W < 1) return VC_ERR_INVALID_ARG;
    q.B.assign(p->L, 0);
    const int rc = viscache_plan_budgets_ex(p->L, q.n, b->rr_num[r], b->rr_den[r], p->h, p->m_num,
                                            p->m_den, p->schedule, p->drop_mode, q.B.data(), &q.Nq,
                                            &q.h);
    if (rc != VC_OK) return rc;
  }
  last_key.swap(key);
  last_plans = *plans;
  return VC_OK;
}

Layout compress_layout(const vc_params* p, const std::vector<RequestPlan>& plans) {
  Layout lay;
  lay.L = p->L; lay.Hq = p->Hq; lay.Hkv = p->Hkv; lay.d = p->d; lay.rank_mode = p->rank_mode;
  lay.need_lse = lay.need_scores = lay.need_sort = lay.need_drop = true;
  lay.need_vs = p->dtype == VC_BF16 && p->d == 128;
  lay.prune_layers = true;
  lay.build(plans);
  return lay;
}

// Decode table of one layer: request r's visual rows start at
// R_r + Hkv * P_l (R_r = rows of the earlier requests, P_l = sum of the
// earlier layers' budgets); its text rows at Hkv * (sum of earlier T).
// Returns VC_ERR_INVALID_ARG when the batch does not fit the table.
int decode_table(const vc_params* p, const std::vector<RequestPlan>& plans, int layer,
                 const int32_t* n_text, DecodeTable* tb) {
  const int n_req = (int)plans.size();
  if (n_req > kDecodeMaxReq || p->Hq / p->Hkv > kDecodeMaxGroup) return VC_ERR_INVALID_ARG;
  tb->n_req = n_req; tb->Hq = p->Hq; tb->Hkv = p->Hkv; tb->G = p->Hq / p->Hkv;
  tb->scale = p->scale == 0.f ? 1.0f / sqrtf((float)p->d) : p->scale;
  for (int r = 0; r < n_req; ++r) {
    const int32_t T = n_text ? n_text[r] : 0;
    if (T < 0 || T > (1 << 24)) return VC_ERR_INVALID_ARG;
  }
  const int split = decode_split_keys(p->dtype);
  tb->split = split;
  int64_t rows = 0, text = 0, units = 0, kgroups = 0;
  const int gr = kv4_group_rows();
  for (int r = 0; r < n_req; ++r) {
    const RequestPlan& pl = plans[r];
    const int32_t T = n_text ? n_text[r] : 0;
    int64_t P = 0, all = 0, KG = 0, allg = 0;
    for (int l = 0; l < p->L; ++l) {
      const int64_t g = (pl.B[l] + gr - 1) / gr;
      if (l < layer) {
        P += pl.B[l];
        KG += g;
      }
      all += pl.B[l];
      allg += g;
    }
    DecodeReq& q = tb->req[r];
    // key groups of the 4-bit form are stacked in row order: request, layer, KV head
    q.kg0 = kgroups + (int64_t)p->Hkv * KG;
    q.nkg = (int32_t)((pl.B[layer] + gr - 1) / gr);
    q.pad = 0;
    kgroups += (int64_t)p->Hkv * allg;
    q.vis_row0 = rows + (int64_t)p->Hkv * P;
    q.txt_row0 = text;
    q.B = pl.B[layer];
    q.T = T;
    q.unit0 = (int32_t)units;
    // a pair without keys still gets one (empty) split, whose merge writes zeros
    q.nsplit = (int32_t)std::max<int64_t>(1, (q.B + (int64_t)T + split - 1) / split);
    units += (int64_t)p->Hkv * q.nsplit;
    if (units > (int64_t)1 << 30) return VC_ERR_INVALID_ARG;
    rows += (int64_t)p->Hkv * all;
    text += (int64_t)p->Hkv * T;
  }
  tb->units = (int32_t)units;
  return VC_OK;
}

struct DecodeWs {
  size_t o_arr = 0, o_ml = 0, o_o = 0, total = 0;
};
DecodeWs decode_ws(int64_t units, int d, int pairs) {
  Arena a;
  DecodeWs w;
  w.o_arr = a.take(sizeof(int32_t) * std::max(pairs, 1));
  w.o_ml = a.take(sizeof(float2) * kDecodeMaxGroup * std::max<int64_t>(units, 1));
  w.o_o = a.take(sizeof(float) * kDecodeMaxGroup * d * std::max<int64_t>(units, 1));
  w.total = a.off;
  return w;
}

// The compacted cache's (request, layer) entries with B > 0, in row order,
// cut into launches of at most kQuantMaxEntries entries.
struct Kv4Plan {
  std::vector<QuantTable> launches;   // tables (only .n entries used)
  std::vector<int> units;             // key groups per launch
  int64_t rows = 0, groups = 0;
};
int kv4_plan(const vc_params* p, const std::vector<RequestPlan>& plans, Kv4Plan* out) {
  const int gr = kv4_group_rows();
  out->launches.clear();
  out->units.clear();
  int64_t row = 0, groups = 0;
  QuantTable cur;
  cur.n = 0;
  cur.pad = 0;
  cur.unit_base = 0;
  int units = 0;
  auto flush = [&]() {
    if (cur.n == 0) return;
    out->launches.push_back(cur);
    out->units.push_back(units);
    cur.n = 0;
    cur.unit_base = groups;
    units = 0;
  };
  for (const RequestPlan& pl : plans) {
    for (int l = 0; l < p->L; ++l) {
      const int32_t b = pl.B[l];
      if (b == 0) continue;
      const int64_t u = (int64_t)p->Hkv * ((b + gr - 1) / gr);
      if (cur.n == kQuantMaxEntries || units + u > (int64_t)1 << 30) flush();
      QuantEntry& e = cur.e[cur.n++];
      e.row0 = row;
      e.B = b;
      e.unit0 = units;
      units += (int)u;
      groups += u;
      row += (int64_t)p->Hkv * b;
    }
  }
  flush();
  out->rows = row;
  out->groups = groups;
  return VC_OK;
}

}  // namespace
}  // namespace vc

using namespace vc;

extern "C" {

const char* viscache_version(void) { return "viscache-gb300 0.2 (sm_103a)"; }

int viscache_device_accessible(const void* ptr) {
  if (!ptr) return 0;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    cudaGetLastError();
    return -VC_ERR_CUDA;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return 1;
  if (a.type == cudaMemoryTypeHost) return a.devicePointer == ptr ? 1 : 0;
  return 0;
}

int viscache_test_inject_wait(int kernel_mask) {
  if (kernel_mask < 0 || kernel_mask > (VC_TEST_WAIT_SCORE_LSE | VC_TEST_WAIT_SCORE_COLSUM | VC_TEST_WAIT_FUSE))
    return VC_ERR_INVALID_ARG;
  g_test_wait.store(kernel_mask);
  return VC_OK;
}

int viscache_set_dependent_launch(int on) {
  if (on != 0 && on != 1) return VC_ERR_INVALID_ARG;
  vc::g_dependent_launch.store(on);
  return VC_OK;
}

int viscache_set_kernel_path(int path) {
  if (path != VC_PATH_AUTO && path != VC_PATH_SIMT) return VC_ERR_INVALID_ARG;
  g_path.store(path);
  return VC_OK;
}

size_t prunekv_score_workspace_size(int32_t L, int32_t Hq, int32_t W) {
  if (L < 1 || L > 256 || Hq < 1 || W < 1) return 0;
  // Hkv = Hq bounds the chunk padding of any Hkv dividing Hq
  return score_layout(L, Hq, Hq, 128, 1, W, VC_RANK_SHARED).total;
}

int prunekv_score(const void* Qw, const void* K, int dtype, int32_t L, int32_t Hq, int32_t Hkv,
                  int32_t d, int32_t n_vis, int32_t W, float scale, int rank_mode,
                  const float* row_lse, float* scores, void* ws, size_t ws_bytes, void* stream) {
  if (!valid_model(dtype, L, Hq, Hkv, d) || n_vis < 1 || n_vis > 65536 || W < 1)
    return VC_ERR_INVALID_ARG;
  if (rank_mode != VC_RANK_SHARED && rank_mode != VC_RANK_PER_LAYER) return VC_ERR_INVALID_ARG;
  if (!Qw || !K || !scores || !aligned16(Qw) || !aligned16(K) || !aligned16(scores))
    return VC_ERR_INVALID_ARG;
  if (!(scale >= 0.f)) return VC_ERR_INVALID_ARG;
  if (scale == 0.f) scale = 1.0f / sqrtf((float)d);
  Layout lay = score_layout(L, Hq, Hkv, d, n_vis, W, rank_mode);
  const int wc = check_ws(ws, ws_bytes, lay.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return cuda_status(launch_score(dtype, Qw, K, lay, scale, w, row_lse, scores, st));
}

size_t prunekv_select_workspace_size(int32_t L, int32_t Hkv, int32_t n_vis, int rank_mode) {
  if (L < 1 || L > 256 || Hkv < 1 || n_vis < 1) return 0;
  return select_layout(L, Hkv, n_vis, nullptr, 0, rank_mode).total;
}

int prunekv_select(const float* scores, int32_t L, int32_t Hkv, int32_t n_vis, const int32_t* B,
                   int32_t Nq, int rank_mode, int32_t* rank_out, int32_t* keep_idx,
                   int32_t* drop_idx, void* ws, size_t ws_bytes, void* stream) {
  if (L < 1 || L > 256 || Hkv < 1 || n_vis < 1 || n_vis > 65536) return VC_ERR_INVALID_ARG;
  if (rank_mode != VC_RANK_SHARED && rank_mode != VC_RANK_PER_LAYER) return VC_ERR_INVALID_ARG;
  if (!scores || !rank_out || !keep_idx || !drop_idx || !valid_budgets(B, L, Nq, n_vis))
    return VC_ERR_INVALID_ARG;
  Layout lay = select_layout(L, Hkv, n_vis, B, Nq, rank_mode);
  const int wc = check_ws(ws, ws_bytes, lay.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = lay.upload(w, st);
  if (e != cudaSuccess) return VC_ERR_CUDA;
  const int problems = rank_mode == VC_RANK_PER_LAYER ? L * Hkv : Hkv;
  e = launch_select(lay.shape(1.f), lay.tables(w), problems, lay.max_chunks, scores, rank_out,
                    reinterpret_cast<uint64_t*>(w + lay.o_chunks), keep_idx,
                    drop_idx, st);
  return cuda_status(e);
}

size_t prunekv_fuse_workspace_size(const int32_t* B, int32_t L, int32_t Hkv, int32_t d,
                                   int32_t n_vis, int32_t Nq) {
  if (L < 1 || L > 256 || Hkv < 1 || (d != 64 && d != 128) || !valid_budgets(B, L, Nq, n_vis)) return 0;
  return fuse_layout(L, Hkv, d, n_vis, B, Nq).total;
}

int prunekv_fuse_compact(const void* K, const void* V, int dtype, int32_t L, int32_t Hkv,
                         int32_t d, int32_t n_vis, const int32_t* B, int32_t Nq,
                         const int32_t* keep_idx, const int32_t* drop_idx, float mu, float tau,
                         void* K_out, void* V_out, void* ws, size_t ws_bytes, void* stream) {
  if (!valid_model(dtype, L, Hkv, Hkv, d) || n_vis < 1 || n_vis > 65536) return VC_ERR_INVALID_ARG;
  if (!valid_budgets(B, L, Nq, n_vis)) return VC_ERR_INVALID_ARG;
  if (!(mu >= 0.f && mu <= 1.f) || !(tau > 0.f)) return VC_ERR_INVALID_ARG;
  if (!K || !V || !keep_idx || !drop_idx || !K_out || !V_out) return VC_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V) || !aligned16(K_out) || !aligned16(V_out))
    return VC_ERR_INVALID_ARG;
  Layout lay = fuse_layout(L, Hkv, d, n_vis, B, Nq);
  const int wc = check_ws(ws, ws_bytes, lay.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = lay.upload(w, st);
  if (e != cudaSuccess) return VC_ERR_CUDA;
  const Shape sh = lay.shape(1.f);
  const Tables tb = lay.tables(w);
  e = launch_fuse(dtype, K, V, lay, sh, tb, keep_idx, drop_idx, mu, tau, K_out, V_out, w, st);
  return cuda_status(e);
}

size_t prunekv_workspace_size(const vc_batch* batch, const vc_params* p) {
  std::vector<RequestPlan> plans;
  if (plan_batch(batch, p, &plans) != VC_OK) return 0;
  return compress_layout(p, plans).total;
}

int prunekv_compress(const vc_batch* batch, const vc_params* p, const void* Qw, const void* K,
                     const void* V, void* K_out, void* V_out, int32_t* idx_out, void* ws,
                     size_t ws_bytes, void* stream) {
  std::vector<RequestPlan> plans;
  const int rc = plan_batch(batch, p, &plans);
  if (rc != VC_OK) return rc;
  if (!Qw || !K || !V || !K_out || !V_out || !idx_out) return VC_ERR_INVALID_ARG;
  if (!aligned16(Qw) || !aligned16(K) || !aligned16(V) || !aligned16(K_out) || !aligned16(V_out))
    return VC_ERR_INVALID_ARG;
  Layout lay = compress_layout(p, plans);
  const int wc = check_ws(ws, ws_bytes, lay.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const float scale = p->scale == 0.f ? 1.0f / sqrtf((float)p->d) : p->scale;
  float* scores = reinterpret_cast<float*>(w + lay.o_scores);
  int32_t* rank = reinterpret_cast<int32_t*>(w + lay.o_rank);
  int32_t* drop = reinterpret_cast<int32_t*>(w + lay.o_drop);
  cudaError_t e = launch_score(p->dtype, Qw, K, lay, scale, w, nullptr, scores, st);
  if (e != cudaSuccess) return VC_ERR_CUDA;
  const Shape sh = lay.shape(scale);
  const Tables tb = lay.tables(w);
  const int problems = lay.n_req * (p->rank_mode == VC_RANK_PER_LAYER ? p->L * p->Hkv : p->Hkv);
  e = launch_select(sh, tb, problems, lay.max_chunks, scores, rank,
                    reinterpret_cast<uint64_t*>(w + lay.o_chunks), idx_out, drop, st);
  if (e != cudaSuccess) return VC_ERR_CUDA;
  e = launch_fuse(p->dtype, K, V, lay, sh, tb, idx_out, drop, p->mu, p->tau, K_out, V_out, w, st);
  return cuda_status(e);
}

int prunekv_get_status(const void* ws, void* stream) {
  if (!ws) return VC_ERR_WORKSPACE;
  int32_t s = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&s, ws, sizeof(s), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return VC_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return VC_ERR_CUDA;
  return s;
}

size_t viscache_decode_workspace_size(const vc_batch* batch, const vc_params* p,
                                      const int32_t* n_text) {
  std::vector<RequestPlan> plans;
  if (plan_batch(batch, p, &plans) != VC_OK) return 0;
  static thread_local DecodeTable tb;
  if (decode_table(p, plans, 0, n_text, &tb) != VC_OK) return 0;   // checks the batch once
  // the largest layer's (KV head, split) units, counted as decode_table does
  const int64_t split = decode_split_keys(p->dtype);
  int64_t units = 0;
  for (int l = 0; l < p->L; ++l) {
    int64_t u = 0;
    for (size_t r = 0; r < plans.size(); ++r) {
      const int64_t keys = plans[r].B[l] + (int64_t)(n_text ? n_text[r] : 0);
      u += (int64_t)p->Hkv * std::max<int64_t>(1, (keys + split - 1) / split);
    }
    units = std::max(units, u);
  }
  return decode_ws(units, p->d, batch->n_req * p->Hkv).total;
}

int viscache_decode_attention(const vc_batch* batch, const vc_params* p, int32_t layer,
                              const void* q, const void* K_out, const void* V_out,
                              const void* K_text, const void* V_text, const int32_t* n_text,
                              void* out, void* ws, size_t ws_bytes, void* stream) {
  std::vector<RequestPlan> plans;
  const int rc = plan_batch(batch, p, &plans);
  if (rc != VC_OK) return rc;
  if (layer < 0 || layer >= p->L) return VC_ERR_INVALID_ARG;
  if (!q || !K_out || !V_out || !out || !aligned16(q) || !aligned16(K_out) || !aligned16(V_out) ||
      !aligned16(out))
    return VC_ERR_INVALID_ARG;
  if (n_text && (!K_text || !V_text || !aligned16(K_text) || !aligned16(V_text)))
    return VC_ERR_INVALID_ARG;
  static thread_local DecodeTable tb;
  const int tc = decode_table(p, plans, layer, n_text, &tb);
  if (tc != VC_OK) return tc;
  const DecodeWs dw = decode_ws(tb.units, p->d, tb.n_req * tb.Hkv);
  const int wc = check_ws(ws, ws_bytes, dw.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  return cuda_status(launch_decode(tb, p->dtype, p->d, q, K_out, V_out, K_text, V_text, out,
                                   reinterpret_cast<float*>(w + dw.o_o),
                                   reinterpret_cast<float2*>(w + dw.o_ml),
                                   reinterpret_cast<int32_t*>(w + dw.o_arr),
                                   static_cast<cudaStream_t>(stream)));
}

int viscache_decode_attention_kv4(const vc_batch* batch, const vc_params* p, int32_t layer,
                                  const void* q, const uint8_t* K_codes, const uint8_t* V_codes,
                                  const float* K_params, const float* V_params, const void* K_text,
                                  const void* V_text, const int32_t* n_text, void* out, void* ws,
                                  size_t ws_bytes, void* stream) {
  std::vector<RequestPlan> plans;
  const int rc = plan_batch(batch, p, &plans);
  if (rc != VC_OK) return rc;
  if (p->dtype != VC_BF16 || layer < 0 || layer >= p->L) return VC_ERR_INVALID_ARG;
  if (!q || !K_codes || !V_codes || !K_params || !V_params || !out || !aligned16(q) ||
      !aligned16(K_codes) || !aligned16(V_codes) || !aligned16(K_params) || !aligned16(V_params) ||
      !aligned16(out))
    return VC_ERR_INVALID_ARG;
  if (n_text && (!K_text || !V_text || !aligned16(K_text) || !aligned16(V_text)))
    return VC_ERR_INVALID_ARG;
  static thread_local DecodeTable tb;
  const int tc = decode_table(p, plans, layer, n_text, &tb);
  if (tc != VC_OK) return tc;
  const DecodeWs dw = decode_ws(tb.units, p->d, tb.n_req * tb.Hkv);
  const int wc = check_ws(ws, ws_bytes, dw.total);
  if (wc != VC_OK) return wc;
  uint8_t* w = static_cast<uint8_t*>(ws);
  return cuda_status(launch_decode_kv4(tb, p->d, q, K_codes, V_codes, K_params, V_params, K_text,
                                       V_text, out, reinterpret_cast<float*>(w + dw.o_o),
                                       reinterpret_cast<float2*>(w + dw.o_ml),
                                       reinterpret_cast<int32_t*>(w + dw.o_arr),
                                       static_cast<cudaStream_t>(stream)));
}

int viscache_kv4_sizes(const vc_batch* batch, const vc_params* p, int64_t* rows, int64_t* key_groups) {
  std::vector<RequestPlan> plans;
  const int rc = plan_batch(batch, p, &plans);
  if (rc != VC_OK) return rc;
  Kv4Plan kp;
  kv4_plan(p, plans, &kp);
  if (rows) *rows = kp.rows;
  if (key_groups) *key_groups = kp.groups;
  return VC_OK;
}

static int kv4_run(const vc_batch* batch, const vc_params* p, bool quantize, const void* K,
                   const void* V, uint8_t* Kc, uint8_t* Vc, float* Kp, float* Vp, void* Kh, void* Vh,
                   void* stream) {
  std::vector<RequestPlan> plans;
  const int rc = plan_batch(batch, p, &plans);
  if (rc != VC_OK) return rc;
  if (!Kc || !Vc || !Kp || !Vp || !aligned16(Kp) || !aligned16(Vp)) return VC_ERR_INVALID_ARG;
  if (quantize ? (!K || !V || !aligned16(K) || !aligned16(V)) : (!Kh || !Vh || !aligned16(Kh) || !aligned16(Vh)))
    return VC_ERR_INVALID_ARG;
  static thread_local Kv4Plan kp;
  kv4_plan(p, plans, &kp);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  for (size_t i = 0; i < kp.launches.size(); ++i) {
    const cudaError_t e = launch_kv4(kp.launches[i], kp.units[i], p->dtype, p->d, quantize, K, V, Kc,
                                     Vc, Kp, Vp, Kh, Vh, st);
    if (e != cudaSuccess) return VC_ERR_CUDA;
  }
  return VC_OK;
}

int viscache_kv4_quantize(const vc_batch* batch, const vc_params* p, const void* K_out,
                          const void* V_out, uint8_t* K_codes, uint8_t* V_codes, float* K_params,
                          float* V_params, void* stream) {
  return kv4_run(batch, p, true, K_out, V_out, K_codes, V_codes, K_params, V_params, nullptr, nullptr,
                 stream);
}

int viscache_kv4_dequantize(const vc_batch* batch, const vc_params* p, const uint8_t* K_codes,
                            const uint8_t* V_codes, const float* K_params, const float* V_params,
                            void* K_hat, void* V_hat, void* stream) {
  return kv4_run(batch, p, false, nullptr, nullptr, const_cast<uint8_t*>(K_codes),
                 const_cast<uint8_t*>(V_codes), const_cast<float*>(K_params),
                 const_cast<float*>(V_params), K_hat, V_hat, stream);
}

}  // extern "C"
