/*
 * viscache.h -- C ABI of libviscache, the GB300 (sm_103a) PruneKV visual-KV
 * compression pass of VisCache (Sec. 3.2 and Algorithm 1 of the paper).
 *
 * The pass runs once per request after prefill.  Per request it
 *   (a) scores every visual token by the attention the observation-window
 *       query rows pay it, summed over query heads and layers   -- Eq. (token_score);
 *   (b) keeps the top-B_l tokens of each KV head in layer l, B_l from the
 *       parabolic schedule, and evicts layers l > h            -- Eq. (parabolic);
 *   (c) drops the keys of the other survivors and fuses their values into
 *       the kept values                                         -- Eq. (redistribution),
 *                                                                  Eq. (weight_fusion);
 *   (d) writes the result as a dense variable-length cache.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every function returns an int status (VC_OK = 0 or a VC_ERR_* code).
 *   Nothing is printed; no C++ exception crosses the ABI.
 * - The caller owns every buffer.  The library never allocates device
 *   memory: scratch space comes from a caller workspace ("ws") whose size the
 *   matching *_workspace_size function returns.  ws must be 256-byte aligned.
 * - Device work is queued on the caller's stream (a cudaStream_t passed as
 *   void*, NULL = legacy default stream) and is asynchronous; after a stream
 *   synchronisation prunekv_get_status(ws) reports device-side errors
 *   (a bounded wait that timed out, an index out of range).
 * - Tensors are dense, row-major, passed as device pointers, element type
 *   VC_BF16 (bfloat16) or VC_F32 (float32); data pointers must be 16-byte
 *   aligned.  Layouts, per request (GQA: query head j reads KV head j / G,
 *   G = Hq / Hkv):
 *       Qw [L][Hq][W][d]    observation-window query rows (the last W rows)
 *       K  [L][Hkv][n][d]   visual keys   (n = n_vis)
 *       V  [L][Hkv][n][d]   visual values
 * - Compressed output ("dense varlen", D8): with P_l = sum_{j<l} B_j, layer l
 *   of a request is a [Hkv][B_l][d] block starting at row Hkv * P_l; the kept
 *   positions idx[Hkv][B_l] sit at the same row offsets.  Rows are in
 *   ascending original position.  Layers l > h (B_l = 0) are absent.
 *   Drop lists use the same scheme with D_l = Nq - B_l (l <= h, B_l > 0).
 * - Supported: d in {64, 128}; 1 <= n <= 65536; W >= 1; Hq % Hkv == 0;
 *   L <= 256.  The library is thread-safe.  Its only state is per host
 *   thread (the last batch's budget plans, reused when the next call repeats
 *   the batch and parameters; results never depend on it), the kernel-path
 *   switch and the profiling switch below, and the fixed scratch array of
 *   prunekv_score_static (VC_STATIC_SCRATCH_BYTES on every device that loads
 *   the library) with its process-wide cache of that array's device address
 *   per CUDA context.
 */
#ifndef VISCACHE_H_
#define VISCACHE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---- */
#define VC_OK                   0
#define VC_ERR_INVALID_ARG      1  /* bad size, mode, pointer alignment, mu/tau range */
#define VC_ERR_INFEASIBLE       2  /* retention target cannot be met (B_1 > n) */
#define VC_ERR_WORKSPACE        3  /* workspace NULL, misaligned or smaller than required */
#define VC_ERR_CUDA             4  /* a CUDA runtime call or kernel launch failed */
#define VC_ERR_DEVICE_TIMEOUT   5  /* a bounded device-side wait gave up */
#define VC_ERR_UNSUPPORTED      6  /* valid request outside what the library implements */
#define VC_ERR_DEVICE_INDEX     7  /* a kernel met an index out of range and skipped it */

/* ---- element types ---- */
#define VC_BF16 0
#define VC_F32  1

/* ---- ranking modes (Sec. 4.4: shared global vs. layer-specific ranking) ---- */
#define VC_RANK_SHARED    0  /* one order per KV head from the 1/L layer mean (default) */
#define VC_RANK_PER_LAYER 1  /* one order per (layer, KV head) */

/*
 * viscache_plan_budgets -- parabolic layer budgets, host only, exact integers.
 *
 * Paper: Eq. (parabolic) b_l = 1 - (l-1)^2 / (2 (h-1)^2) for l <= h, layers
 * l > h evicted, normalised to sum_l b_l = h*m; RR = p*q*(h/L)*m (Sec. 4,
 * Implementation Details) with p = 1.
 * Reading: T = round(RR * n * L) kept (token, layer) pairs per KV head,
 * split over layers 1..h in proportion to b_l by largest remainder (ties to
 * the lower layer); survivors Nq = round(T / (h*m)), at least B_1, at most n.
 * round() is round-half-up on exact rationals.
 *
 *   L, n_vis        layers, visual tokens (>= 1)
 *   rr_num/rr_den   overall retention RR in (0, 1]
 *   h               truncation layer in [1, L]; 0 selects round(3L/4)
 *                   clamped to [min(2, L), L]
 *   m_num/m_den     average layer budget m in (0, 1]; m_den = 0 selects 3/4
 *   B_out           host int32[L]: B_l (0 for l > h), non-increasing
 *   n_survive_out   host int32: Nq
 *   h_out           host int32 (nullable): the truncation layer used
 * Errors: VC_ERR_INVALID_ARG (ranges, NULL outputs), VC_ERR_INFEASIBLE (B_1 > n).
 */
int viscache_plan_budgets(int32_t L, int32_t n_vis, uint32_t rr_num, uint32_t rr_den,
                          int32_t h, uint32_t m_num, uint32_t m_den,
                          int32_t* B_out, int32_t* n_survive_out, int32_t* h_out);

/* Layer-budget schedules (the ablation axes of the paper's Table "ablation"). */
#define VC_SCHED_PARABOLA   0  /* Eq. (parabolic), the method's schedule (default) */
#define VC_SCHED_FIXED      1  /* uniform budget per kept layer */
#define VC_SCHED_ARITHMETIC 2  /* arithmetic progression (PyramidKV-style) */
#define VC_SCHED_GEOMETRIC  3  /* geometric progression over four layer blocks (PDrop-style) */

/* Drop set of each layer. */
#define VC_DROP_SURVIVORS 0    /* survivors of the top-q step minus the keep set (default) */
#define VC_DROP_ALL       1    /* every token not kept (n - B_l), i.e. Nq = n */

/*
 * viscache_plan_budgets_ex -- viscache_plan_budgets with a budget schedule
 * and a drop-set choice.  The table names the schedules only ("uniform",
 * "arithmetic progression", "geometric progression across four layer
 * blocks"); the readings keep everything else of the method fixed (layers
 * l > h evicted, T = round(RR*n*L), largest remainder, Nq = round(T/(h*m))
 * clamped to [B_1, n]) and give b_l for l = 1..h as:
 *   VC_SCHED_PARABOLA    1 - (l-1)^2 / (2 (h-1)^2)
 *   VC_SCHED_FIXED       1
 *   VC_SCHED_ARITHMETIC  1 - (l-1) / (2 (h-1))      (same end points 1 and 1/2)
 *   VC_SCHED_GEOMETRIC   (1/2)^k for block k = 0..min(4,h)-1 of a split of
 *                        layers 1..h into min(4, h) contiguous blocks whose
 *                        sizes differ by at most one (larger blocks first)
 * (b_l = 1 for every schedule when h = 1).  With VC_DROP_ALL the survivors
 * are all n tokens (Nq = n), so each layer's drop set is every token it does
 * not keep (the alternative reading of V_d's n - b_l rows in Sec. 3.2).
 *   schedule    one of VC_SCHED_*
 *   drop_mode   VC_DROP_SURVIVORS or VC_DROP_ALL
 * Other arguments and errors as viscache_plan_budgets; B_out is
 * non-increasing for every schedule.
 */
int viscache_plan_budgets_ex(int32_t L, int32_t n_vis, uint32_t rr_num, uint32_t rr_den,
                             int32_t h, uint32_t m_num, uint32_t m_den, int32_t schedule,
                             int32_t drop_mode, int32_t* B_out, int32_t* n_survive_out,
                             int32_t* h_out);

/*
 * prunekv_score -- token importance, Eq. (token_score) / Algorithm 1 step 1.
 *
 *   s[g][v]    = (1/L) sum_l sum_{j in group g} sum_i A^l_{j,i,v}   (VC_RANK_SHARED)
 *   s[l][g][v] =       sum_{j in group g} sum_i A^l_{j,i,v}         (VC_RANK_PER_LAYER)
 *   A^l_{j,i,v} = softmax over the n visual keys of scale * q^l_{j,i} . k^l_{j/G,v}
 *
 * With row_lse (device float[L][Hq][W], natural log, nullable) the
 * normaliser is taken from the caller instead: A = exp(scale*q.k - lse).
 *   Qw, K       device, dtype, layouts above
 *   scale       0 selects 1/sqrt(d)
 *   scores      device float32 output, [Hkv][n] or [L][Hkv][n]
 *   ws          workspace of prunekv_score_workspace_size(L, Hq, W) bytes
 * Arithmetic: bf16 inputs are multiplied exactly and accumulated in fp32;
 * softmax and sums in fp32.
 */
size_t prunekv_score_workspace_size(int32_t L, int32_t Hq, int32_t W);
int prunekv_score(const void* Qw, const void* K, int dtype, int32_t L, int32_t Hq,
                  int32_t Hkv, int32_t d, int32_t n_vis, int32_t W, float scale,
                  int rank_mode, const float* row_lse, float* scores,
                  void* ws, size_t ws_bytes, void* stream);

/*
 * prunekv_score_static -- prunekv_score for callers that cannot allocate
 * device memory (code running inside an allocator or memory-pool hook, where
 * a cudaMalloc would re-enter the allocator; a runtime that replays frozen
 * CUDA graphs and hands out no workspace; an embedding host without a device
 * allocator).  The paper has no counterpart: this is a deployment
 * convenience, not a step of the method.
 *
 * Same arguments, arithmetic and result as prunekv_score, minus the
 * workspace: the scratch (status word, plan tables, per-row log-sum-exp) is a
 * fixed device array of VC_STATIC_SCRATCH_BYTES inside the library, which
 * every GPU that loads the library holds until the process exits.  Nothing
 * is allocated: no cudaMalloc, cudaFree or allocating library routine.
 *   - Problems needing more scratch than that (prunekv_score_workspace_size
 *     (L, Hq, W) > VC_STATIC_SCRATCH_BYTES, i.e. roughly L*Hq*W > 460,000
 *     window rows: the 7B shape with up to 512 window rows fits, the 72B
 *     shape with 128 window rows, 655,360 rows, does not) are rejected with
 *     VC_ERR_WORKSPACE before any device work.
 *   - The first call in a CUDA context looks up the array's device address
 *     (cudaGetSymbolAddress) with that context's device current and caches
 *     it with the context's id; make that first call before capturing a
 *     stream.  After cudaDeviceReset (or when the primary context is
 *     released and created again) the array may move: the next call sees a
 *     new context id and looks the address up again, so it too should come
 *     before any capture.
 *   - All calls on a device share the array and it keeps the last call's
 *     contents; each call rewrites everything it reads (the status word is
 *     cleared when the call starts).  Calls whose kernels overlap on the GPU
 *     race on the array: serialise them.
 *   - Device-side errors (a bounded wait that gave up, an index out of
 *     range) land in the array's status word: prunekv_score_static_status
 *     reads it after the call, exactly as prunekv_get_status does for a
 *     workspace.
 */
#define VC_STATIC_SCRATCH_BYTES (16u << 20)
int prunekv_score_static(const void* Qw, const void* K, int dtype, int32_t L, int32_t Hq,
                         int32_t Hkv, int32_t d, int32_t n_vis, int32_t W, float scale,
                         int rank_mode, const float* row_lse, float* scores, void* stream);
/* Size in bytes of prunekv_score_static's scratch array (VC_STATIC_SCRATCH_BYTES). */
size_t prunekv_score_static_capacity(void);
/*
 * Device-side status of the last prunekv_score_static call on the current
 * device: synchronises `stream` (pass the stream the call used), then returns
 * VC_OK, the first device error the call recorded (VC_ERR_DEVICE_TIMEOUT,
 * VC_ERR_DEVICE_INDEX), or VC_ERR_CUDA if the word could not be read.
 * Allocates nothing.
 */
int prunekv_score_static_status(void* stream);

/*
 * prunekv_select -- rank, keep and drop sets, Algorithm 1 steps 1 and 3.
 *
 * Per KV head (per (layer, KV head) in VC_RANK_PER_LAYER) tokens are ordered
 * by descending score, the lower index first on exact ties.  The first Nq are
 * the survivors ("retain the q percent", the rest discarded); layer l keeps
 * the first B_l and drops survivors B_l .. Nq-1.
 *   scores      device float32 from prunekv_score
 *   B           HOST int32[L] budgets (from viscache_plan_budgets), B_l <= Nq <= n
 *   rank_out    device int32 [Hkv][n] (or [L][Hkv][n]): position of each token
 *   keep_idx    device int32, rows Hkv*P_l + g*B_l + r: kept positions, ascending
 *   drop_idx    device int32, rows Hkv*Q_l + g*D_l + r, D_l = Nq - B_l,
 *               Q_l = sum_{j<l, B_j>0} D_j: dropped survivors, ascending
 *   ws          workspace of prunekv_select_workspace_size(...) bytes
 */
size_t prunekv_select_workspace_size(int32_t L, int32_t Hkv, int32_t n_vis, int rank_mode);
int prunekv_select(const float* scores, int32_t L, int32_t Hkv, int32_t n_vis,
                   const int32_t* B, int32_t Nq, int rank_mode, int32_t* rank_out,
                   int32_t* keep_idx, int32_t* drop_idx, void* ws, size_t ws_bytes,
                   void* stream);

/*
 * prunekv_fuse_compact -- prune keys, fuse values, compact; Algorithm 1 step 3.
 *
 *   K_out = K[keep]                                  (bit-exact copy)
 *   V_out = mu * V_k + (1 - mu) * Phi V_d,  Phi = row-softmax(V_k V_d^T / tau)
 *           -- Eq. (redistribution), Eq. (weight_fusion); V_out = V_k when the
 *           drop set is empty.  fp32 arithmetic, rounded to dtype (RNE).
 *   K, V              [L][Hkv][n][d], dtype: device memory, or host memory the
 *                     device can read (viscache_device_accessible == 1; only the
 *                     kept rows of K and the survivors' rows of V are read)
 *   B, Nq             HOST budgets as for prunekv_select
 *   keep_idx/drop_idx device lists from prunekv_select
 *   mu in [0, 1], tau > 0
 *   K_out, V_out      device, dense varlen (rows Hkv * sum_l B_l, d columns)
 *   ws                workspace of prunekv_fuse_workspace_size(B, L, Hkv, d, n, Nq) bytes
 *                     (bf16, d = 128 also compacts the survivors' values there;
 *                     the tensor-core fusion then copies K_out itself while its
 *                     products run when K is device memory)
 */
size_t prunekv_fuse_workspace_size(const int32_t* B, int32_t L, int32_t Hkv, int32_t d,
                                   int32_t n_vis, int32_t Nq);
int prunekv_fuse_compact(const void* K, const void* V, int dtype, int32_t L, int32_t Hkv,
                         int32_t d, int32_t n_vis, const int32_t* B, int32_t Nq,
                         const int32_t* keep_idx, const int32_t* drop_idx, float mu,
                         float tau, void* K_out, void* V_out, void* ws, size_t ws_bytes,
                         void* stream);

/*
 * prunekv_compress -- the whole pass for a batch of requests in one call:
 * plan (host), score, select, fuse and compact, queued on one stream.
 *
 * Requests share the model shape (L, Hq, Hkv, d) and differ in n, W and RR.
 * Inputs are packed request after request, each request laid out exactly as
 * a single request:  K/V of request r start at element L*Hkv*d*sum_{r'<r} n_r',
 * Qw of request r at element L*Hq*d*sum_{r'<r} W_r'.  Outputs likewise: request
 * r's dense varlen cache starts at row Hkv * sum_{r'<r} T_r' (T_r = sum_l B_l).
 * Qw, K, the outputs and ws are device memory.  V may also be host memory the
 * device can read (viscache_device_accessible(V) == 1): only the rows of the
 * surviving tokens of layers with B_l > 0 are read, once, so V can stay on the
 * host while Qw and K are copied in.
 */
typedef struct {
    int32_t n_req;            /* number of requests, >= 1 */
    const int32_t* n_vis;     /* host [n_req] visual tokens per request */
    const int32_t* W;         /* host [n_req] window rows per request */
    const uint32_t* rr_num;   /* host [n_req] retention numerators */
    const uint32_t* rr_den;   /* host [n_req] retention denominators */
} vc_batch;

typedef struct {
    int32_t L, Hq, Hkv, d;    /* model shape */
    int32_t dtype;            /* VC_BF16 or VC_F32 */
    int32_t h;                /* truncation layer, 0 = round(3L/4) */
    uint32_t m_num, m_den;    /* average layer budget m, m_den = 0 -> 3/4 */
    float mu;                 /* fusion strength, paper default 0.7 */
    float tau;                /* redistribution temperature, paper default 1.0 */
    float scale;              /* logit scale, 0 -> 1/sqrt(d) */
    int32_t rank_mode;        /* VC_RANK_SHARED or VC_RANK_PER_LAYER */
    int32_t schedule;         /* VC_SCHED_* layer-budget schedule (0 = parabola) */
    int32_t drop_mode;        /* VC_DROP_SURVIVORS or VC_DROP_ALL */
} vc_params;

size_t prunekv_workspace_size(const vc_batch* batch, const vc_params* p);
int prunekv_compress(const vc_batch* batch, const vc_params* p, const void* Qw,
                     const void* K, const void* V, void* K_out, void* V_out,
                     int32_t* idx_out, void* ws, size_t ws_bytes, void* stream);

/*
 * viscache_scout_mmr -- keyframe selection of the scout stage, Eq. (mmr)
 * (Sec. 3.1): per video, frames join the selected set Omega greedily by
 *     lambda * sim(h_f, h_t) - (1 - lambda) * max_{f' in Omega} sim(h_f, h_f')
 * with sim the cosine similarity, until k = ceil(p * F) frames are chosen
 * (Sec. 4: lambda = 0.7, p = 0.75).  Readings: the redundancy term is 0 while
 * Omega is empty (the first pick is the most prompt-relevant frame), ties go
 * to the lower frame index, a zero vector has similarity 0.  fp32 arithmetic.
 *
 *   H             device fp32 [sum_r F_r][D] frame embeddings, video after video
 *   prompt        device fp32 [n_req][D] prompt embeddings
 *   n_req         videos, 1..64
 *   n_frames      host int32 [n_req]: F_r, 1..4096
 *   D             embedding width, 1..8192
 *   lambda        relevance weight in [0, 1]
 *   p_num/p_den   frame retention ratio p in (0, 1]
 *   order_out     device int32 [sum_r k_r]: picks in selection order, video r
 *                 at row sum_{r'<r} k_r'
 *   keyframes_out device int32, same rows: the picks in ascending frame order
 *   gains_out     device fp32, same rows (nullable): each pick's MMR score
 *   k_out         host int32 [n_req] (nullable): k_r
 *   ws            device workspace, 256-byte aligned, viscache_scout_workspace_size bytes
 * All outputs and ws are caller-owned; the call is asynchronous on `stream`.
 * Errors: VC_ERR_INVALID_ARG (sizes, ranges, NULL or misaligned inputs),
 * VC_ERR_WORKSPACE, VC_ERR_CUDA.
 */
size_t viscache_scout_workspace_size(int32_t n_req, const int32_t* n_frames, int32_t D);
/*
 * viscache_scout_sizes -- host only: the number of keyframes k_r = ceil(p * F_r)
 * viscache_scout_mmr picks for each video (the rows its outputs need), written
 * to k_out (host int32 [n_req]).  Same argument checks as viscache_scout_mmr.
 */
int viscache_scout_sizes(int32_t n_req, const int32_t* n_frames, uint32_t p_num, uint32_t p_den,
                         int32_t* k_out);
int viscache_scout_mmr(const float* H, const float* prompt, int32_t n_req, const int32_t* n_frames,
                       int32_t D, float lambda, uint32_t p_num, uint32_t p_den, int32_t* order_out,
                       int32_t* keyframes_out, float* gains_out, int32_t* k_out, void* ws,
                       size_t ws_bytes, void* stream);

/*
 * prunekv_get_status -- device-side status of the last call that used ws.
 * Synchronises the stream, returns VC_OK or the first device error code
 * recorded (VC_ERR_DEVICE_TIMEOUT, VC_ERR_DEVICE_INDEX), or VC_ERR_CUDA.
 * Every entry point clears the status word when it starts.
 */
int prunekv_get_status(const void* ws, void* stream);

/*
 * Benchmark support (not a step of the pass): per-kernel CUDA-event timing.
 * viscache_profile_enable(1) makes every later kernel launch record an event
 * pair on its stream (and clears what was recorded); viscache_profile_read
 * waits for the recorded events, writes up to max_kernels entries -- kernel
 * names joined by '\n' into names (name_bytes long), summed milliseconds and
 * launch counts -- clears the record and returns the number of entries, or
 * -VC_ERR_CUDA if an event could not be read.  Not thread-safe; off by default.
 */
int viscache_profile_enable(int on);
int viscache_profile_read(char* names, int name_bytes, float* total_ms, int* launches,
                          int max_kernels);

/*
 * viscache_decode_attention -- one decode step's attention in layer `layer`
 * over the cache that prunekv_compress left (Sec. 2 "VLLM Decoding"; after
 * PruneKV, Sec. 3.2, the visual part of layer l holds B_l rows per KV head):
 *     out[r][j] = softmax(q[r][j] . K_g^T * scale) V_g,   g = j / (Hq / Hkv),
 * over request r's B_l kept visual rows of KV head g followed by its T_r text
 * rows.  fp32 accumulation, out rounded once to the input type.
 *
 *   batch, p      the batch and parameters prunekv_compress ran with (they fix
 *                 every B_l); 1..256 requests, Hq / Hkv <= 8
 *   layer         0..L-1
 *   q             device [n_req][Hq][d], the step's query rows
 *   K_out, V_out  device [rows][d]: prunekv_compress's outputs; layer l, KV
 *                 head g of request r at row R_r + Hkv * P_l + g * B_l with
 *                 P_l = sum_{l'<l} B_l' and R_r = sum_{r'<r} Hkv * sum_l B_l
 *                 (a full cache in [L][Hkv][n][d] order per request is this
 *                 layout with every B_l = n)
 *   K_text, V_text device [sum_r Hkv * T_r][d], this layer's text rows, per
 *                 request [Hkv][T_r][d] packed; NULL when n_text is NULL
 *   n_text        host int32 [n_req] (nullable = no text): T_r, 0..2^24
 *   out           device [n_req][Hq][d]; a query with no keys gets zeros
 *   ws            device workspace, 256-byte aligned,
 *                 viscache_decode_workspace_size bytes (enough for any layer)
 * Types follow p->dtype (bf16 or fp32); every pointer 16-byte aligned.  All
 * buffers are caller-owned; the call is asynchronous on `stream`.
 * Errors: VC_ERR_INVALID_ARG (shapes, ranges, NULL or misaligned pointers),
 * VC_ERR_WORKSPACE, VC_ERR_CUDA.
 */
size_t viscache_decode_workspace_size(const vc_batch* batch, const vc_params* p,
                                      const int32_t* n_text);
/*
 * viscache_decode_attention_kv4 -- the same step over the 4-bit form of the
 * visual rows (viscache_kv4_quantize's outputs for the same batch and
 * parameters; bf16 only): each visual row is expanded to code * scale + min
 * rounded to bf16, exactly the rows viscache_kv4_dequantize writes, and the
 * attention is then the one above.  Text rows, queries and output are bf16;
 * the workspace is viscache_decode_workspace_size's.  Errors as above.
 */
int viscache_decode_attention_kv4(const vc_batch* batch, const vc_params* p, int32_t layer,
                                  const void* q, const uint8_t* K_codes, const uint8_t* V_codes,
                                  const float* K_params, const float* V_params, const void* K_text,
                                  const void* V_text, const int32_t* n_text, void* out, void* ws,
                                  size_t ws_bytes, void* stream);
int viscache_decode_attention(const vc_batch* batch, const vc_params* p, int32_t layer,
                              const void* q, const void* K_out, const void* V_out,
                              const void* K_text, const void* V_text, const int32_t* n_text,
                              void* out, void* ws, size_t ws_bytes, void* stream);

/*
 * viscache_kv4_* -- 4-bit quantisation of the compacted cache (Appendix
 * "Quantization": the compressed visual KV combined with a 4-bit KV cache
 * quantiser; the paper names KIVI-style quantisers without defining one).
 * Asymmetric round-to-nearest with a per-group scale and minimum:
 *     scale = (max - min) / 15,  code = clamp(rint((x - min) / scale), 0, 15)
 *     (code 0 when scale = 0),   x_hat = code * scale + min (fused multiply-add),
 * decided in fp32 (IEEE subtraction and division, rint to nearest even).
 * Keys: per channel over groups of 32 consecutive rows of one (request,
 * layer, KV head) segment of prunekv_compress's output (the last group of a
 * segment may be shorter).  Values: per row over groups of 32 channels.
 *
 *   batch, p      the batch and parameters prunekv_compress ran with (d = 64
 *                 or 128; bf16 or fp32 per p->dtype)
 *   K_out, V_out  device [rows][d], prunekv_compress's outputs
 *   K_codes, V_codes  device uint8 [rows][d/2]: two codes per byte, the even
 *                 channel in the low nibble
 *   K_params      device fp32 [key_groups][d][2]: (scale, min) per channel of
 *                 each key group, groups in row order
 *   V_params      device fp32 [rows][d/32][2]: (scale, min) per value group
 *   K_hat, V_hat  device [rows][d] (dequantize): the reconstruction, rounded
 *                 once to the input type
 * viscache_kv4_sizes gives rows and key_groups for a batch (host only; either
 * pointer may be NULL).  Float arrays 16-byte aligned.  All buffers are
 * caller-owned; the calls are asynchronous on `stream` and need no workspace.
 * Errors: VC_ERR_INVALID_ARG (shapes, NULL or misaligned pointers), the
 * planner's errors for the batch, VC_ERR_CUDA.
 */
int viscache_kv4_sizes(const vc_batch* batch, const vc_params* p, int64_t* rows,
                       int64_t* key_groups);
int viscache_kv4_quantize(const vc_batch* batch, const vc_params* p, const void* K_out,
                          const void* V_out, uint8_t* K_codes, uint8_t* V_codes, float* K_params,
                          float* V_params, void* stream);
int viscache_kv4_dequantize(const vc_batch* batch, const vc_params* p, const uint8_t* K_codes,
                            const uint8_t* V_codes, const float* K_params, const float* V_params,
                            void* K_hat, void* V_hat, void* stream);

/*
 * Kernel path selection (process-wide, default VC_PATH_AUTO): AUTO runs the
 * score (Eq. token_score) and the fusion (Eq. redistribution, weight_fusion)
 * of bf16, d = 128 problems on the tcgen05 tensor cores and everything else
 * on CUDA cores; VC_PATH_SIMT forces the CUDA-core kernels (fp32 FFMA) for
 * every problem.  Both compute the same quantities; used to cross-check.
 */
#define VC_PATH_AUTO 0
#define VC_PATH_SIMT 1
int viscache_set_kernel_path(int path);

/*
 * Launch ordering (process-wide, default 1): with 1 the kernels of a call
 * after its first are programmatic dependent launches -- each may be
 * scheduled while the kernel before it on the stream drains, and waits on
 * the device for that kernel's results before it reads them -- which hides
 * the gaps between them; with 0 every kernel is an ordinary launch and starts
 * only when the previous one has completed.  Results are the same either
 * way; 0 is for debugging and for timing the difference.  Calls are never
 * overlapped with work queued before them: a call's first kernel is always
 * an ordinary launch.  Errors: VC_ERR_INVALID_ARG unless on is 0 or 1.
 */
int viscache_set_dependent_launch(int on);

/*
 * viscache_test_inject_wait -- test support for the failure detection of the
 * tensor-core kernels (not a step of the pass).  For every later launch of
 * a kernel named in kernel_mask, one consumer warp first waits on an
 * mbarrier that nothing ever completes ("a flag that nothing sets"), bounded
 * like every wait of these kernels but with a short limit (~10^5 SM clocks).
 * When the wait gives up the kernel records VC_ERR_DEVICE_TIMEOUT in the
 * status word and then does its normal work (its own barriers and copies are
 * not touched), so the launch ends, the context stays usable, and the
 * caller's prunekv_get_status / prunekv_score_static_status reads the error.
 * kernel_mask 0 (the default) turns it off.  Process-wide; not thread-safe
 * against concurrent calls.  Errors: VC_ERR_INVALID_ARG for unknown bits.
 */
#define VC_TEST_WAIT_SCORE_LSE    1  /* score_lse_tc: the row log-sum-exp pass */
#define VC_TEST_WAIT_SCORE_COLSUM 2  /* score_colsum_tc: the column-sum pass */
#define VC_TEST_WAIT_FUSE         4  /* fuse_v_tc: the value fusion */
int viscache_test_inject_wait(int kernel_mask);

/*
 * viscache_device_accessible -- 1 if the current device can read `ptr`
 * directly (device memory, managed memory, or host memory mapped into the
 * device's address space, e.g. pinned with cudaHostAlloc under unified
 * addressing), 0 if not, -VC_ERR_CUDA if the query fails.  Not a step of the
 * pass: it tells a caller whether V may stay in host memory (see
 * prunekv_compress).  No device work, no synchronisation.
 */
int viscache_device_accessible(const void* ptr);

/* Version string of the library build. */
const char* viscache_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VISCACHE_H_ */
