/*
 * mmshift.h -- C ABI of the GB300 (sm_103a) prefill-only KV selection library.
 *
 * The library implements MM-ShiftKV's selection step (the paper's Section 3.2
 * and Algorithm 1 in Appendix B): after prefill, for every layer and KV head,
 *   1. build variance-expanded query proxies from the observation-window
 *      queries (Section 3.2.1, Appendix A.4);
 *   2. score every prompt key with the proxies' attention logits under GQA
 *      head grouping, 3. softmax over the whole prompt (Section 3.2.2);
 *   4. aggregate the attention mass per proxy group and vote with the
 *      tau-coverage rule, add the last-query anchor (Sections 3.2.2-3.2.3);
 *   5. keep the last token plus the top C-1 keys (Section 3.2.3);
 *   6. gather the kept K/V rows, in temporal order, into a compact cache
 *      (Appendix B).
 * Beyond the window-statistics path (mmshift_select and its steps):
 *   - proxy statistics over every prompt query (mmshift_prefill_stats,
 *     mmshift_select_with_stats) or over the prefill hidden states, with the
 *     proxies sampled in hidden space and projected by W_Q on the tensor
 *     cores (mmshift_hidden_stats, mmshift_build_hidden_proxies), as
 *     Section 3.2.1 writes them;
 *   - a budget per layer and KV head (mmshift_select_head_budgets,
 *     mmshift_topk_head_budgets; Section 3.1's C_{l,h});
 *   - the attention-mass coverage of a kept set for given decode queries
 *     (mmshift_coverage; Section 1, Fig. 1b).
 *
 * Conventions shared by every entry point:
 *   - All pointers except the ones marked "host" are device pointers. The
 *     caller owns every buffer; the library allocates no device memory and,
 *     apart from mmshift_poll_status, never synchronises. One exception:
 *     V, of which only the kept rows are read (by the gather), may also be
 *     page-locked host memory mapped into the device's address space at the
 *     same address (cudaHostAlloc / cudaHostRegister memory under unified
 *     addressing); the gather then reads just those rows across the
 *     host link. mmshift_select and mmshift_gather check K, Qwin and V
 *     with cudaPointerGetAttributes and refuse (MMSHIFT_ERR_INVALID_ARG)
 *     pageable host memory.
 *   - All work is enqueued on `stream` (a cudaStream_t; NULL is the legacy
 *     default stream) and is asynchronous.
 *   - Host-side validation runs first; on error nothing is enqueued and the
 *     outputs are untouched. Errors from the CUDA runtime are returned as
 *     MMSHIFT_ERR_CUDA (see mmshift_last_cuda_error).
 *   - Token data is "varlen packed": requests are concatenated along the token
 *     axis with host prefix offsets cu_seqlens[0..batch] (cu_seqlens[0] = 0).
 *   - A call covers n_layers layers; layer l reads K + l*layer_stride_kv,
 *     V + l*layer_stride_kv and Qwin + l*layer_stride_q (strides in elements)
 *     and uses the random-stream layer id params.layer_id + l. Every output
 *     and debug buffer is laid out [n_layers, ...] contiguously.
 *   - Results are deterministic for fixed inputs and (seed, layer_id).
 *
 * Shapes (T = total tokens = cu_seqlens[batch], R = sum_b min(C_b, T_b)):
 *   K, V        [T, Hkv, d]        dtype; rows contiguous (d elements)
 *   Qwin        [batch, W, Hq, d]  dtype; the W last prefill queries of each
 *                                  request, the last row being the last real
 *                                  prefill query (the anchor of Section 3.2.3)
 *   proxies     [batch, Hq, N, d]  dtype
 *   group_mass  [Hkv, G, T]        float32  (per layer)
 *   anchor, mass, scores [Hkv, T]  float32  (per layer)
 *   out_idx     [R, Hkv]           int32 token index within its request;
 *                                  request b owns rows [sum_{b'<b} C'_b', +C'_b),
 *                                  ascending in each column (temporal order)
 *   out_K/out_V [R, Hkv, d]        dtype; out_K[c, h] = K[cu_b + out_idx[c, h], h]
 */
#ifndef MMSHIFT_H
#define MMSHIFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* mmshift_stream_t; /* same type as cudaStream_t */

typedef enum {
  MMSHIFT_OK = 0,
  MMSHIFT_ERR_INVALID_ARG = 1, /* null pointer, bad shape, bad parameter */
  MMSHIFT_ERR_UNSUPPORTED = 2, /* valid but not implemented (dtype, head_dim) */
  MMSHIFT_ERR_WORKSPACE = 3,   /* workspace missing, too small or misaligned */
  MMSHIFT_ERR_CUDA = 4,        /* a CUDA runtime call failed */
  MMSHIFT_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
  MMSHIFT_ERR_DEVICE = 6       /* a device-side check failed */
} mmshift_status;

enum { MMSHIFT_BF16 = 0, MMSHIFT_F32 = 1 };

/* Importance score used by the budgeted top-k.
 * VOTE: S_t = vote(t) + lambda * anchor_t (Sections 3.2.2-3.2.3; the paper's
 *       method). MASS: S_t = sum_g group_mass[g, t] (the Table 5 ablation row
 *       with sampling and variance expansion but no group vote). */
enum { MMSHIFT_SCORE_VOTE = 0, MMSHIFT_SCORE_MASS = 1 };

#define MMSHIFT_MAX_BATCH 64
#define MMSHIFT_MAX_LAYERS 4096

/* Method hyper-parameters; defaults (mmshift_default_params) are the paper's
 * Section 4.1 values: N = 512 proxies in G = 32 groups, gamma = 10,
 * tau = 0.95, lambda = 1. */
typedef struct {
  int32_t n_proxies;      /* N per query head; 0 with n_groups = 0 = anchor only */
  int32_t n_groups;       /* G; n_proxies % n_groups == 0 */
  float gamma;            /* variance expansion, > 0 (Section 3.2.1) */
  float tau;              /* coverage threshold, 0 < tau <= 1 (Section 3.2.2) */
  float lambda;           /* anchor weight, >= 0 (Section 3.2.3) */
  int32_t score_mode;     /* MMSHIFT_SCORE_VOTE or MMSHIFT_SCORE_MASS */
  uint64_t seed;          /* key of the proxy random stream */
  int32_t layer_id;       /* layer id of the first layer of the call */
  float softmax_scale;    /* 0 => 1/sqrt(head_dim) */
  float rope_theta;       /* > 0 rotates proxies (RoPE base); 0 => no RoPE */
  int32_t rope_pos_offset;/* proxies sit at position T_b + rope_pos_offset */
} mmshift_params;

typedef struct {
  int32_t batch;            /* 1..MMSHIFT_MAX_BATCH requests */
  int32_t n_q_heads;        /* Hq, multiple of n_kv_heads */
  int32_t n_kv_heads;       /* Hkv */
  int32_t head_dim;         /* d: 64 or 128 */
  int32_t window;           /* W >= 2 observation-window queries */
  int32_t dtype;            /* MMSHIFT_BF16 or MMSHIFT_F32 */
  const int32_t* cu_seqlens;/* host [batch+1], T_b = cu[b+1]-cu[b] >= 1 */
  const int32_t* budgets;   /* host [batch], C_b >= 1 */
  int32_t n_layers;         /* 1..MMSHIFT_MAX_LAYERS */
  int64_t layer_stride_kv;  /* elements between layers of K and V (>= T*Hkv*d) */
  int64_t layer_stride_q;   /* elements between layers of Qwin (>= B*W*Hq*d) */
} mmshift_shape;

/* Optional intermediate outputs of mmshift_select (any may be NULL). */
typedef struct {
  void* proxies;     /* [L, batch, Hq, N, d] dtype: the sampled proxies */
  float* group_mass; /* [L, Hkv, G, T] attention mass of each proxy group */
  float* anchor;     /* [L, Hkv, T] last-query attention, mean over the GQA heads */
  float* mass;       /* [L, Hkv, T] sum_g group_mass */
  float* scores;     /* [L, Hkv, T] S_t used by the top-k */
  /* Stage timing: if n_stage_events >= MMSHIFT_N_STAGES + 1, stage_events
   * holds caller-created cudaEvent_t handles and event i is recorded on
   * `stream` just before stage i is enqueued (the last one after the last
   * stage). Stages: proxies, softmax pass, normaliser merge, mass pass,
   * anchor normalisation (tensor-core calls whose anchor rows stay out of the
   * softmax pass) and mass sum, coverage vote, top-k, gather; a stage that
   * does not run records its event next to its neighbour's. */
  void** stage_events;
  int32_t n_stage_events;
  int32_t launches;   /* out: number of kernels the call enqueued */
  int32_t score_path; /* out: 1 if steps 2-4 ran on the tensor cores (tcgen05),
                         0 if on the CUDA cores (fp32 FMA) */
  /* Test of the bounded device-side waits; 0 in normal use. Non-zero: on the
   * tensor-core path, one epilogue warp of the mass pass's first CTA waits
   * on a barrier that nothing arrives on; after 64 polls (a few ms) it gives
   * up and aborts its CTA, which waits for the copies and MMAs it already
   * issued and frees its tensor memory. The call's outputs are then
   * undefined and mmshift_poll_status returns MMSHIFT_ERR_TIMEOUT; the
   * context, the workspace and later calls are unaffected. */
  int32_t test_stuck_wait;
} mmshift_debug;

#define MMSHIFT_N_STAGES 8

/* Fill *p with the paper's default hyper-parameters (Section 4.1). */
void mmshift_default_params(mmshift_params* p);

/* Rows R = sum_b min(C_b, T_b) of out_idx / out_K / out_V per layer. */
mmshift_status mmshift_output_rows(const mmshift_shape* s, int64_t* rows);

/* Bytes of device workspace the calls below need for (s, p); 256-byte
 * alignment is required. The same workspace serves every entry point. */
mmshift_status mmshift_workspace_size(const mmshift_shape* s, const mmshift_params* p,
                                      size_t* bytes);

/* Step 1 alone (Section 3.2.1, Appendix A.4): per (request, query head,
 * dimension) mean and unbiased std over the W window queries, then
 * proxies[b, hq, i, j] = mu + gamma * sigma * z with z ~ N(0, 1): one
 * Philox4x64-10 draw (counter (i*d/8 + q, hq, b, layer_id), key (seed, 0))
 * gives, as eight 32-bit uniforms ((w >> 9) + 1/2) 2^-23 and Box-Muller on
 * consecutive pairs, dims 4q..4q+3 and d/2+4q..d/2+4q+3; then an optional
 * RoPE rotation to position T_b + rope_pos_offset and rounding to dtype.
 * proxies: [L, batch, Hq, N, d]. */
mmshift_status mmshift_build_proxies(const mmshift_shape* s, const void* Qwin,
                                     const mmshift_params* p, void* proxies,
                                     mmshift_stream_t stream);

/* Proxy statistics over the whole prefill (Section 3.2.1: the mean and the
 * standard deviation of the prompt's features are taken across all prompt
 * tokens; read in query space): for every layer l, request b, query head hq
 * and dimension j, over the T_b prompt queries of the request,
 *   stats[l][b][0][hq][j] = mean_t Qfull[l][cu_b + t][hq][j],
 *   stats[l][b][1][hq][j] = their standard deviation, T_b - 1 denominator
 *                           (0 for T_b = 1).
 * Qfull: [L][total_T][Hq][d] in the shape's dtype, 16-byte aligned; layers
 * `qfull_layer_stride` elements apart (0 = densely packed; a multiple of 8).
 * stats: [L][batch][2][Hq][d] float32. workspace: at least
 * mmshift_prefill_stats_workspace_size() bytes (per-chunk partial sums).
 * Reads every byte of Qfull once; deterministic (fixed merge order). */
mmshift_status mmshift_prefill_stats_workspace_size(const mmshift_shape* s, size_t* bytes);
mmshift_status mmshift_prefill_stats(const mmshift_shape* s, const void* Qfull,
                                     int64_t qfull_layer_stride, float* stats, void* workspace,
                                     size_t workspace_bytes, mmshift_stream_t stream);

/* Hidden-state statistics (Section 3.2.1: mu_pre, sigma_pre of the hidden
 * states entering layer l, per feature over all T_b prompt tokens of
 * request b, unbiased, 0 for T_b = 1): the reduction of mmshift_prefill_stats
 * over d_model columns. H: [L][T_total][d_model] in the shape's dtype, layers
 * `h_layer_stride` elements apart (0 = dense; a multiple of 8), 16-byte
 * aligned; d_model a multiple of 8. stats: [L][batch][2][d_model] float32
 * (mean, std). workspace: mmshift_hidden_stats_workspace_size() bytes. */
mmshift_status mmshift_hidden_stats_workspace_size(const mmshift_shape* s, int32_t d_model,
                                                  size_t* bytes);
mmshift_status mmshift_hidden_stats(const mmshift_shape* s, int32_t d_model, const void* H,
                                    int64_t h_layer_stride, float* stats, void* workspace,
                                    size_t workspace_bytes, mmshift_stream_t stream);

/* Step 1 in the hidden space (Section 3.2.1, the paper's construction):
 * N proxy hidden states H~_i = mu + gamma * sigma * z_i per (layer, request),
 * z from Philox4x64-10 with key (seed, 1) and counter
 * (i * d_model/8 + q, 0, b, layer_id + l) covering features [4q, 4q+4) and
 * [d_model/2 + 4q, +4) (Box-Muller on consecutive uniforms), rounded to
 * bf16, projected by the query projection on the tensor cores,
 * q~_i = W_Q H~_i + b_Q (fp32 accumulation), rotated by RoPE (rotate-half
 * pairs within each head, when params->rope_theta > 0) to position
 * rope_pos[b] (host array, nullable: T_b + rope_pos_offset; for M-RoPE
 * models pass the text position of the first decoded token, where the three
 * M-RoPE components coincide) and rounded to bf16.
 * hstats: [L][batch][2][d_model] float32 (mmshift_hidden_stats);
 * W_Q: [L][Hq*d][d_model] bf16 (row hq*d + j = output feature j of query
 * head hq), layers `wq_layer_stride` elements apart (0 = dense; a multiple
 * of 8), 16-byte aligned; bias_q: [L][Hq*d] bf16 or NULL. proxies:
 * [L, batch, Hq, N, d] bf16, for mmshift_select / mmshift_proxy_mass as
 * `proxies_in`. workspace: mmshift_hidden_proxies_workspace_size() bytes,
 * 256-byte aligned (its first word is the status mmshift_poll_status reads).
 * bf16 only (MMSHIFT_ERR_UNSUPPORTED otherwise); d_model a multiple of 64,
 * Hq*d a multiple of 128; needs the tensor-core path (sm_100 family). */
mmshift_status mmshift_hidden_proxies_workspace_size(const mmshift_shape* s, int32_t d_model,
                                                     const mmshift_params* p, size_t* bytes);
mmshift_status mmshift_build_hidden_proxies(const mmshift_shape* s, int32_t d_model,
                                            const float* hstats, const void* W_Q,
                                            int64_t wq_layer_stride, const void* bias_q,
                                            const int32_t* rope_pos, const mmshift_params* p,
                                            void* proxies, void* workspace,
                                            size_t workspace_bytes, mmshift_stream_t stream);

/* Step 1 from given statistics (e.g. mmshift_prefill_stats) instead of the
 * observation window's: q~ = mu + gamma * sigma * z with the same normals,
 * RoPE and rounding as mmshift_build_proxies. stats: [L][batch][2][Hq][d]
 * float32 (mean, std); proxies: [L, batch, Hq, N, d]. Pass the proxies to
 * mmshift_select / mmshift_proxy_mass to select with them, or pass the
 * statistics to mmshift_select_with_stats. */
mmshift_status mmshift_build_proxies_from_stats(const mmshift_shape* s, const float* stats,
                                                const mmshift_params* p, void* proxies,
                                                mmshift_stream_t stream);

/* Steps 2-4 (Section 3.2.2, Appendix B): softmax attention of every proxy over
 * all T_b keys of its KV head (h = hq / r), summed per proxy group over the r
 * query heads of that KV head; and the last-query anchor (mean over the r
 * heads). `proxies` ([L, batch, Hq, N, d]) may be NULL, in which case they
 * are sampled as in mmshift_build_proxies. Outputs are [L, ...] float32;
 * `mass` may be NULL. */
mmshift_status mmshift_proxy_mass(const mmshift_shape* s, const void* K, const void* Qwin,
                                  const void* proxies, const mmshift_params* p,
                                  float* group_mass, float* anchor, float* mass,
                                  void* workspace, size_t workspace_bytes,
                                  mmshift_stream_t stream);

/* Step 5 from masses (Sections 3.2.2-3.2.3): tau-coverage sets per (KV head,
 * group) -- the smallest prefix of keys by descending mass (ties: lower t
 * first) holding at least tau of the group's mass --, votes, S_t = vote +
 * lambda * anchor (or sum_g mass in MASS mode), then the kept indices.
 * group_mass [L, Hkv, G, T], anchor [L, Hkv, T] (unused in MASS mode);
 * scores (nullable: S_t is written there when given) [L, Hkv, T];
 * out_idx [L, R, Hkv]. */
mmshift_status mmshift_scores_topk(const mmshift_shape* s, const mmshift_params* p,
                                   const float* group_mass, const float* anchor,
                                   float* scores, int32_t* out_idx,
                                   void* workspace, size_t workspace_bytes,
                                   mmshift_stream_t stream);

/* Budgeted selection from given scores (Section 3.2.3): token T_b-1 always,
 * plus the C_b-1 largest S_t among t < T_b-1 (ties: lower t first), in
 * ascending order; C_b >= T_b keeps every token. scores [L, Hkv, T] float32,
 * finite; out_idx [L, R, Hkv]. */
mmshift_status mmshift_topk(const mmshift_shape* s, const float* scores, int32_t* out_idx,
                            void* workspace, size_t workspace_bytes,
                            mmshift_stream_t stream);

/* Step 6 (Appendix B): out_K[c, h] = K[cu_b + idx[c, h], h], same for V; a
 * bit copy. idx [L, R, Hkv] must hold indices in [0, T_b); out of range rows
 * are zero-filled and reported by mmshift_poll_status. */
mmshift_status mmshift_gather(const mmshift_shape* s, const void* K, const void* V,
                              const int32_t* idx, void* out_K, void* out_V,
                              void* workspace, size_t workspace_bytes,
                              mmshift_stream_t stream);

/* The whole selection (Algorithm 1): steps 1-6 for L layers. `proxies_in`
 * (nullable, [L, batch, Hq, N, d]) replaces the sampled proxies, e.g. for
 * proxies a caller projects from hidden states. `dbg` (nullable) receives
 * intermediate results. */
mmshift_status mmshift_select(const mmshift_shape* s, const void* K, const void* V,
                              const void* Qwin, const void* proxies_in,
                              const mmshift_params* p, int32_t* out_idx, void* out_K,
                              void* out_V, const mmshift_debug* dbg, void* workspace,
                              size_t workspace_bytes, mmshift_stream_t stream);

/* mmshift_select with the proxies' statistics given (Section 3.2.1: mean and
 * std over the whole prefill, e.g. from mmshift_prefill_stats) instead of
 * taken over the observation window; the sampled proxies use the same normals,
 * RoPE and rounding. stats: [L][batch][2][Hq][d] float32 (mean, std), read
 * only, must not be NULL. Qwin still supplies the anchor (its last row).
 * Same outputs, workspace and errors as mmshift_select. */
mmshift_status mmshift_select_with_stats(const mmshift_shape* s, const void* K, const void* V,
                                         const void* Qwin, const float* stats,
                                         const mmshift_params* p, int32_t* out_idx, void* out_K,
                                         void* out_V, const mmshift_debug* dbg, void* workspace,
                                         size_t workspace_bytes, mmshift_stream_t stream);

/* Budgets per layer and KV head (Section 3.1 defines the budget C_{l,h} per
 * layer and KV head; Section 4.3 pairs the selection with allocators that
 * spread budgets over layers and heads). head_budgets: device
 * [L][batch][Hkv] int32, C_{l,b,h} in [1, budgets[b]] (the shape's budgets
 * are each request's capacity: they size the output rows; values outside are
 * clamped and reported by mmshift_poll_status). Head h of request b keeps
 * min(C_{l,b,h}, T_b) rows of out_idx (T_b - 1 and the top others, in
 * ascending order); its remaining rows up to min(C_b, T_b) hold -1 and
 * gather zero K/V rows. out_count (nullable): device [L][batch][Hkv] int32,
 * the kept rows per head. Otherwise as mmshift_select / mmshift_topk. */
mmshift_status mmshift_select_head_budgets(const mmshift_shape* s, const void* K, const void* V,
                                           const void* Qwin, const void* proxies_in,
                                           const int32_t* head_budgets, const mmshift_params* p,
                                           int32_t* out_idx, int32_t* out_count, void* out_K,
                                           void* out_V, const mmshift_debug* dbg, void* workspace,
                                           size_t workspace_bytes, mmshift_stream_t stream);
mmshift_status mmshift_topk_head_budgets(const mmshift_shape* s, const float* scores,
                                         const int32_t* head_budgets, int32_t* out_idx,
                                         int32_t* out_count, void* workspace,
                                         size_t workspace_bytes, mmshift_stream_t stream);

/* Quality metric (Section 1, Fig. 1b): attention-mass coverage of a kept
 * set. For decode query g of query head hq (dec_q [L, batch, Hq, n_dec, d]
 * in the shape's dtype, the proxies_in layout), the softmax of
 * scale * q.k_t over the T_b prompt keys of KV head h = hq / r, summed over
 * the kept indices idx [L, R, Hkv] (e.g. mmshift_select's out_idx: indices
 * in [0, T_b); -1 marks padding rows and is skipped; other values are
 * skipped and reported by mmshift_poll_status) and
 * averaged over the r query heads of h: cov [L][batch][Hkv][n_dec] float32.
 * Steps 2-4 run with the decode queries as n_dec groups of one proxy (so the
 * masses come from the same kernels as the selection's); Qwin supplies the
 * anchor rows those kernels also compute. softmax_scale 0 = 1/sqrt(d);
 * 1 <= n_dec <= 1024; workspace: mmshift_coverage_workspace_size() bytes. */
mmshift_status mmshift_coverage_workspace_size(const mmshift_shape* s, int32_t n_dec,
                                               size_t* bytes);
mmshift_status mmshift_coverage(const mmshift_shape* s, const void* K, const void* Qwin,
                                const void* dec_q, int32_t n_dec, float softmax_scale,
                                const int32_t* idx, float* cov, void* workspace,
                                size_t workspace_bytes, mmshift_stream_t stream);

/* Allocation-free variant of mmshift_scores_topk.
 *
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory -- e.g. code running inside a runtime or
 * plugin host that owns every device allocation and hands out no workspace,
 * or a serving loop whose memory plan is frozen after start-up. Instead of a
 * caller workspace it uses a scratch array compiled into the library: a
 * file-scope __device__ array of MMSHIFT_NOALLOC_SCRATCH_BYTES (8 MiB) that
 * every GPU which loads the library holds until the process exits. It calls
 * no cudaMalloc/cudaFree and no allocating library routine.
 *
 *  - Inputs and outputs are the caller's, exactly as in mmshift_scores_topk
 *    (group_mass, anchor, nullable scores, out_idx).
 *  - Scratch use is L*Hkv*G*ceil32(T_b)/8 bytes of coverage bitmaps, plus
 *    L*Hkv*T*4 bytes of scores when `scores` is NULL (each part rounded up to
 *    256 bytes). Larger problems are rejected with MMSHIFT_ERR_WORKSPACE before
 *    anything is enqueued.
 *  - The first call on a device (with that device current) looks up the
 *    array's device address with cudaGetSymbolAddress; make that first call
 *    before any stream capture on that device. The address is kept for the
 *    life of the process, so destroying the device's primary context after
 *    that first call (cudaDeviceReset, which reloads the library's module
 *    and moves the array) is not supported.
 *  - Every call on a device shares the one array, which keeps the contents of
 *    the last call; nothing in it needs to start at zero (every byte read is
 *    first written by the same call). Calls whose work overlaps on the GPU --
 *    on different streams, or from different host threads without ordering --
 *    race on the array and must be serialised by the caller. */
#define MMSHIFT_NOALLOC_SCRATCH_BYTES (8u << 20)
mmshift_status mmshift_scores_topk_noalloc(const mmshift_shape* s, const mmshift_params* p,
                                           const float* group_mass, const float* anchor,
                                           float* scores, int32_t* out_idx,
                                           mmshift_stream_t stream);

/* Synchronise `stream`, read and clear the device status word kept in the
 * workspace: MMSHIFT_OK, MMSHIFT_ERR_TIMEOUT or MMSHIFT_ERR_DEVICE. */
mmshift_status mmshift_poll_status(void* workspace, mmshift_stream_t stream);

/* Human-readable name of a status code. */
const char* mmshift_status_string(mmshift_status st);

/* Text of the last CUDA runtime error seen on this host thread ("" if none). */
const char* mmshift_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* MMSHIFT_H */
