// Host side of the C ABI declared in include/mmshift.h: argument validation,
// problem description, workspace carve-up and kernel sequencing. Nothing here
// allocates device memory or synchronises (except mmshift_poll_status).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>

#include "common.cuh"

using namespace mmshift;

namespace {

thread_local std::string g_cuda_error;

mmshift_status cuda_fail(cudaError_t e) {
  g_cuda_error = cudaGetErrorString(e);
  return MMSHIFT_ERR_CUDA;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
int roundup(int x, int m) { return (x + m - 1) / m * m; }

mmshift_status check_shape(const mmshift_shape* s) {
  if (!s || !s->cu_seqlens || !s->budgets) return MMSHIFT_ERR_INVALID_ARG;
  if (s->batch < 1 || s->batch > MMSHIFT_MAX_BATCH) return MMSHIFT_ERR_INVALID_ARG;
  if (s->n_layers < 1 || s->n_layers > MMSHIFT_MAX_LAYERS) return MMSHIFT_ERR_INVALID_ARG;
  if (s->n_kv_heads < 1 || s->n_q_heads < s->n_kv_heads || s->n_q_heads % s->n_kv_heads)
    return MMSHIFT_ERR_INVALID_ARG;
  if (s->window < 2) return MMSHIFT_ERR_INVALID_ARG;
  if (s->dtype != MMSHIFT_BF16 && s->dtype != MMSHIFT_F32) return MMSHIFT_ERR_UNSUPPORTED;
  if (s->head_dim != 64 && s->head_dim != 128) return MMSHIFT_ERR_UNSUPPORTED;
  if (s->cu_seqlens[0] != 0) return MMSHIFT_ERR_INVALID_ARG;
  int64_t total = 0;
  for (int b = 0; b < s->batch; ++b) {
    const int64_t t = (int64_t)s->cu_seqlens[b + 1] - s->cu_seqlens[b];
    if (t < 1 || s->budgets[b] < 1) return MMSHIFT_ERR_INVALID_ARG;
    total += t;
  }
  if (total > (int64_t)1 << 30) return MMSHIFT_ERR_UNSUPPORTED;
  if (s->n_layers > 1) {
    if (s->layer_stride_kv < total * s->n_kv_heads * s->head_dim) return MMSHIFT_ERR_INVALID_ARG;
    if (s->layer_stride_q < (int64_t)s->batch * s->window * s->n_q_heads * s->head_dim)
      return MMSHIFT_ERR_INVALID_ARG;
  }
  return MMSHIFT_OK;
}

mmshift_status check_params(const mmshift_params* p) {
  if (!p) return MMSHIFT_ERR_INVALID_ARG;
  if (p->n_proxies < 0 || p->n_groups < 0) return MMSHIFT_ERR_INVALID_ARG;
  if ((p->n_proxies == 0) != (p->n_groups == 0)) return MMSHIFT_ERR_INVALID_ARG;
  if (p->n_groups && p->n_proxies % p->n_groups) return MMSHIFT_ERR_INVALID_ARG;
  if (p->n_groups > 1024) return MMSHIFT_ERR_UNSUPPORTED;
  if (!(p->gamma > 0.f) || !std::isfinite(p->gamma)) return MMSHIFT_ERR_INVALID_ARG;
  if (!(p->tau > 0.f) || p->tau > 1.f) return MMSHIFT_ERR_INVALID_ARG;
  if (!(p->lambda >= 0.f) || !std::isfinite(p->lambda)) return MMSHIFT_ERR_INVALID_ARG;
  if (p->score_mode != MMSHIFT_SCORE_VOTE && p->score_mode != MMSHIFT_SCORE_MASS)
    return MMSHIFT_ERR_INVALID_ARG;
  if (!(p->softmax_scale >= 0.f) || !std::isfinite(p->softmax_scale)) return MMSHIFT_ERR_INVALID_ARG;
  if (!(p->rope_theta >= 0.f) || !std::isfinite(p->rope_theta)) return MMSHIFT_ERR_INVALID_ARG;
  if (p->layer_id < 0) return MMSHIFT_ERR_INVALID_ARG;
  return MMSHIFT_OK;
}

// Key split length of the softmax pass. It is a constant, so the order in
// which a request's partial (max, sum) pairs are merged -- and with it every
// bit of the result -- does not depend on the other requests or layers of the
// call.
constexpr int kSplitLen = 1024;

mmshift_status build_problem(const mmshift_shape* s, const mmshift_params* p, Problem* P) {
  std::memset(P, 0, sizeof(*P));
  P->B = s->batch;
  P->L = s->n_layers;
  P->Hq = s->n_q_heads;
  P->Hkv = s->n_kv_heads;
  P->r = s->n_q_heads / s->n_kv_heads;
  P->d = s->head_dim;
  P->W = s->window;
  P->dtype = s->dtype;
  P->Np = p->n_proxies;
  P->G = p->n_groups;
  P->gs = P->G ? P->Np / P->G : 0;
  P->RG = roundup(P->r * P->gs, kChunk);
  P->n_group_rows = P->G * P->RG;
  P->anchor_rows = roundup(P->r, kChunk);
  P->Prows = P->n_group_rows + P->anchor_rows;
  P->Prows_pad = roundup(P->Prows, kRowTile);
  int64_t tot = 0, outr = 0, words = 0;
  for (int b = 0; b < P->B; ++b) {
    ReqInfo& R = P->req[b];
    R.t_len = s->cu_seqlens[b + 1] - s->cu_seqlens[b];
    R.tok_off = s->cu_seqlens[b];
    R.budget = s->budgets[b];
    R.keep = std::min(R.budget, R.t_len);
    R.out_off = (int32_t)outr;
    R.word_off = (int32_t)words;
    tot += R.t_len;
    outr += R.keep;
    words += (R.t_len + 31) / 32;
  }
  P->total_T = (int32_t)tot;
  P->R = (int32_t)outr;
  P->total_words = (int32_t)words;
  P->ls_kv = s->n_layers > 1 ? s->layer_stride_kv : 0;
  P->ls_q = s->n_layers > 1 ? s->layer_stride_q : 0;
  P->scale = p->softmax_scale > 0.f ? p->softmax_scale : 1.0f / std::sqrt((float)s->head_dim);
  P->alpha = P->scale * kLog2e;
  P->gamma = p->gamma;
  P->tau = p->tau;
  P->lambda = p->lambda;
  P->mode = p->score_mode;
  P->seed = p->seed;
  P->layer_id0 = p->layer_id;
  P->rope_theta = p->rope_theta;
  P->rope_off = p->rope_pos_offset;
  P->split_len = kSplitLen;
  int32_t so = 0;
  for (int b = 0; b < P->B; ++b) {
    ReqInfo& R = P->req[b];
    R.nsplit = (R.t_len + P->split_len - 1) / P->split_len;
    R.split_off = so;
    so += R.nsplit;
  }
  P->total_splits = so;
  return MMSHIFT_OK;
}

struct Layout {
  size_t status, packed, part, cvals, gmass, anchor, alog, apart, bits, scores, refine, refine_stats, total;
};

// The anchor rows start a 256-row block of their own: on the tensor-core
// path the softmax pass leaves them out (Problem::anchor_split).
bool anchor_spills(const Problem& P) {
  return P.G > 0 && P.n_group_rows % kRowTile == 0 && P.r <= kMaxSplitAnchor;
}

Layout layout_of(const Problem& P) {
  const size_t esz = P.dtype == MMSHIFT_BF16 ? 2 : 4;
  const size_t L = P.L;
  Layout w;
  size_t o = 0;
  w.status = o; o += 256;
  w.packed = o; o += align256(L * P.B * P.Hkv * (size_t)P.Prows_pad * P.d * esz);
  w.part = o;   o += align256(L * P.Hkv * (size_t)P.total_splits * kUmmaPartSlots * P.Prows_pad * sizeof(float2));
  w.cvals = o;  o += align256(L * P.B * P.Hkv * (size_t)P.Prows_pad * sizeof(float));
  w.gmass = o;  o += align256(L * P.Hkv * (size_t)P.G * P.total_T * sizeof(float));
  w.anchor = o; o += align256(L * P.Hkv * (size_t)P.total_T * sizeof(float));
  w.alog = o;   o += anchor_spills(P) ? align256(L * P.Hkv * (size_t)P.r * P.total_T * sizeof(float)) : 0;
  w.apart = o;  o += anchor_spills(P) ? align256(L * P.Hkv * (size_t)P.total_splits * kMaxSplitAnchor * sizeof(float2)) : 0;
  w.bits = o;   o += align256(L * P.Hkv * (size_t)P.G * P.total_words * sizeof(uint32_t));
  w.scores = o; o += align256(L * P.Hkv * (size_t)P.total_T * sizeof(float));
  // count word, the list of proxy elements to recompute in float64, then the
  // exact window sums they are recomputed from
  w.refine = o; o += 256 + align256((size_t)proxy_refine_capacity(P) * sizeof(int4));
  w.refine_stats = o; o += align256(L * P.B * P.Hq * (size_t)5 * P.d * sizeof(float));
  w.total = o;
  return w;
}

mmshift_status carve(const Problem& P, void* ws, size_t bytes, Buffers* bf) {
  const Layout w = layout_of(P);
  if (!ws || bytes < w.total) return MMSHIFT_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 255) return MMSHIFT_ERR_WORKSPACE;
  char* base = static_cast<char*>(ws);
  std::memset(bf, 0, sizeof(*bf));
  bf->status = reinterpret_cast<int*>(base + w.status);
  bf->packed = base + w.packed;
  bf->part = reinterpret_cast<float2*>(base + w.part);
  bf->cvals = reinterpret_cast<float*>(base + w.cvals);
  bf->gmass = reinterpret_cast<float*>(base + w.gmass);
  bf->anchor = reinterpret_cast<float*>(base + w.anchor);
  bf->alog = reinterpret_cast<float*>(base + w.alog);
  bf->apart = reinterpret_cast<float2*>(base + w.apart);
  bf->bits = reinterpret_cast<uint32_t*>(base + w.bits);
  bf->scores = reinterpret_cast<float*>(base + w.scores);
  bf->refine_count = reinterpret_cast<int*>(base + w.refine);
  bf->refine_items = reinterpret_cast<int4*>(base + w.refine + 256);
  bf->refine_cap = (int32_t)proxy_refine_capacity(P);
  bf->refine_stats = reinterpret_cast<float*>(base + w.refine_stats);
  return MMSHIFT_OK;
}

mmshift_status prepare(const mmshift_shape* s, const mmshift_params* p, Problem* P) {
  mmshift_status st = check_shape(s);
  if (st != MMSHIFT_OK) return st;
  mmshift_params dflt;
  if (!p) { mmshift_default_params(&dflt); p = &dflt; }
  if ((st = check_params(p)) != MMSHIFT_OK) return st;
  return build_problem(s, p, P);
}

// Records stage-boundary events when the caller asked for them.
struct StageMarks {
  cudaEvent_t* ev = nullptr;
  cudaStream_t st = nullptr;
  cudaError_t mark(int stage) const {
    return ev ? cudaEventRecord(ev[stage], st) : cudaSuccess;
  }
};

StageMarks marks_of(const mmshift_debug* dbg, cudaStream_t st) {
  StageMarks m;
  m.st = st;
  if (dbg && dbg->stage_events && dbg->n_stage_events >= MMSHIFT_N_STAGES + 1)
    m.ev = reinterpret_cast<cudaEvent_t*>(dbg->stage_events);
  return m;
}

// Tensor-core scoring when the device, dtype, shape and K's alignment (TMA
// needs a 16-byte aligned base) allow it; CUDA-core scoring otherwise.
int choose_umma(const Problem& P, const void* K) {
  return (umma_supported(P) && (reinterpret_cast<uintptr_t>(K) & 15) == 0) ? 1 : 0;
}

// Scoring path of a call: tensor or CUDA cores, and the softmax partials
// and anchor handling that go with it.
void set_score_path(Problem& P, const void* K) {
  P.use_umma = choose_umma(P, K);
  P.part_slots = P.use_umma ? kUmmaPartSlots : 1;
  P.anchor_split = P.use_umma && anchor_spills(P) ? 1 : 0;
}

// Kernels one mmshift_select call enqueues (reported through mmshift_debug).
int count_launches(const Problem& P, const Buffers& bf) {
  int n = proxy_launches(P, bf);               // proxies (+ float64 refinement)
  n += P.use_umma ? umma_launches(P) : 3;      // softmax pass, merge, mass pass
  if (bf.mass && P.total_T) n += 1;            // mass sum
  if (P.mode == MMSHIFT_SCORE_VOTE && P.G) n += 1;  // coverage vote
  n += 1;                                      // top-k
  if (P.R) n += 1;                             // gather
  return n;
}

// Proxies (sampled or given) packed into the workspace, then steps 2-4.
mmshift_status run_mass(const Problem& P, const Buffers& bf, const void* K, const void* qwin,
                        cudaStream_t st, const StageMarks& mk = StageMarks()) {
  cudaError_t e;
  if ((e = mk.mark(0)) != cudaSuccess) return cuda_fail(e);
  if ((e = launch_proxy_pack(P, bf, st, qwin)) != cudaSuccess) return cuda_fail(e);
  e = P.use_umma ? launch_score_umma(P, bf, st, K, mk.ev)
                 : launch_score_simt(P, bf, st, K, mk.ev);
  if (e != cudaSuccess) return cuda_fail(e);
  if ((e = mk.mark(4)) != cudaSuccess) return cuda_fail(e);
  if ((e = launch_anchor_split(P, bf, st)) != cudaSuccess) return cuda_fail(e);
  if ((e = launch_mass_sum(P, bf, st)) != cudaSuccess) return cuda_fail(e);
  return MMSHIFT_OK;
}

}  // namespace

namespace mmshift {
// Shared with the allocation-free entry point (noalloc.cu).
mmshift_status noalloc_prepare(const mmshift_shape* s, const mmshift_params* p, Problem* P) {
  return prepare(s, p, P);
}
mmshift_status noalloc_cuda_fail(cudaError_t e) { return cuda_fail(e); }
}  // namespace mmshift

// Whole-prefill statistics job of a shape (no hyper-parameters involved).
static mmshift_status stats_job(const mmshift_shape* s, int64_t qfull_layer_stride, StatsJob* J,
                                int32_t ncol = 0) {
  mmshift_status st = check_shape(s);
  if (st != MMSHIFT_OK) return st;
  std::memset(J, 0, sizeof(*J));
  J->L = s->n_layers;
  J->B = s->batch;
  J->ncol = ncol ? ncol : s->n_q_heads * s->head_dim;
  if (J->ncol % 8) return MMSHIFT_ERR_INVALID_ARG;
  const int64_t total = s->cu_seqlens[s->batch];
  int maxc = 0;
  for (int b = 0; b < s->batch; ++b) {
    J->tok_off[b] = s->cu_seqlens[b];
    J->t_len[b] = s->cu_seqlens[b + 1] - s->cu_seqlens[b];
    maxc = std::max(maxc, (J->t_len[b] + kStatsChunk - 1) / kStatsChunk);
  }
  J->nchunk = maxc;
  const int64_t dense = total * J->ncol;
  J->ls = qfull_layer_stride ? qfull_layer_stride : dense;
  if (J->L > 1 && J->ls < dense) return MMSHIFT_ERR_INVALID_ARG;
  if (J->ls % 8) return MMSHIFT_ERR_INVALID_ARG;   // 16-byte rows for the vector loads
  return MMSHIFT_OK;
}

// Whether kernels may read `p` with plain loads: device or managed memory,
// or page-locked host memory mapped at the same address (unified
// addressing). Pageable host memory is refused.
static bool device_readable(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();   // clear the sticky error of a failed query
    return false;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return true;
  return a.type == cudaMemoryTypeHost && a.devicePointer == p;
}
static bool device_memory(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// The hidden-space proxy job of a call: shapes, tiles and RoPE positions.
static mmshift_status hidden_job(const mmshift_shape* s, int32_t d_model, const mmshift_params* p,
                                 const int32_t* rope_pos, HiddenJob* J) {
  mmshift_status st = check_shape(s);
  if (st != MMSHIFT_OK) return st;
  if ((st = check_params(p)) != MMSHIFT_OK) return st;
  if (s->dtype != MMSHIFT_BF16) return MMSHIFT_ERR_UNSUPPORTED;
  if (d_model < 64 || d_model % 64) return MMSHIFT_ERR_UNSUPPORTED;
  const int F = s->n_q_heads * s->head_dim;
  if (F % 128) return MMSHIFT_ERR_UNSUPPORTED;
  std::memset(J, 0, sizeof(*J));
  J->L = s->n_layers;
  J->B = s->batch;
  J->Hq = s->n_q_heads;
  J->d = s->head_dim;
  J->F = F;
  J->DM = d_model;
  J->N = p->n_proxies;
  J->Npad = (p->n_proxies + 127) / 128 * 128;
  J->NT = F % 256 == 0 ? 256 : 128;
  J->MT = J->Npad / 128;
  J->NTL = F / J->NT;
  J->tiles = J->L * J->B * J->MT * J->NTL;
  J->gamma = p->gamma;
  J->rope_theta = p->rope_theta;
  J->seed = p->seed;
  J->layer_id0 = p->layer_id;
  for (int b = 0; b < s->batch; ++b)
    J->pos[b] = rope_pos ? rope_pos[b] : (s->cu_seqlens[b + 1] - s->cu_seqlens[b]) + p->rope_pos_offset;
  return MMSHIFT_OK;
}

// Steps 1-6 of Algorithm 1 for every layer; proxies from the window
// statistics, from given statistics (stats_in) or given outright (proxies_in).
static mmshift_status select_impl(const mmshift_shape* s, const void* K, const void* V,
                                  const void* Qwin, const void* proxies_in, const float* stats_in,
                                  const mmshift_params* p, int32_t* out_idx, void* out_K,
                                  void* out_V, const mmshift_debug* dbg, void* workspace,
                                  size_t workspace_bytes, mmshift_stream_t stream,
                                  const int32_t* head_budgets = nullptr,
                                  int32_t* out_count = nullptr) {
  Problem P;
  mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !K || !V || !Qwin || !out_idx || !out_K || !out_V) return MMSHIFT_ERR_INVALID_ARG;
  set_score_path(P, K);
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  // K and Qwin are streamed by every pass: device memory; V is read only for
  // the kept rows and may also be mapped page-locked host memory
  if (!device_memory(K) || !device_memory(Qwin) || !device_readable(V))
    return MMSHIFT_ERR_INVALID_ARG;
  bf.proxies_in = proxies_in;
  bf.stats_in = stats_in;
  bf.head_budget = head_budgets;
  bf.out_count = out_count;
  if (dbg) {
    P.test_stuck_wait = dbg->test_stuck_wait;
    bf.proxies_out = dbg->proxies;
    if (dbg->group_mass && P.G) bf.gmass = dbg->group_mass;
    if (dbg->anchor) bf.anchor = dbg->anchor;
    if (dbg->scores) { bf.scores = dbg->scores; bf.scores_out = 1; }
    bf.mass = dbg->mass;
  }
  const cudaStream_t cs = (cudaStream_t)stream;
  const StageMarks mk = marks_of(dbg, cs);
  P.cover_hint = (float)(P.r * P.gs);   // the masses below are softmax sums over r * gs rows
  if ((st = run_mass(P, bf, K, Qwin, cs, mk)) != MMSHIFT_OK) return st;
  cudaError_t e = mk.mark(5);
  if (e == cudaSuccess && P.mode == MMSHIFT_SCORE_VOTE) e = launch_cover(P, bf, cs);
  if (e == cudaSuccess) e = mk.mark(6);
  if (e == cudaSuccess) e = launch_topk(P, bf, cs, out_idx, false);
  if (e == cudaSuccess) e = mk.mark(7);
  if (e == cudaSuccess) e = launch_gather(P, bf, cs, K, V, out_idx, out_K, out_V);
  if (e == cudaSuccess) e = mk.mark(8);
  if (dbg) {
    const_cast<mmshift_debug*>(dbg)->launches = count_launches(P, bf);
    const_cast<mmshift_debug*>(dbg)->score_path = P.use_umma ? 1 : 0;
  }
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

extern "C" {

void mmshift_default_params(mmshift_params* p) {
  if (!p) return;
  std::memset(p, 0, sizeof(*p));
  p->n_proxies = 512;
  p->n_groups = 32;
  p->gamma = 10.0f;
  p->tau = 0.95f;
  p->lambda = 1.0f;
  p->score_mode = MMSHIFT_SCORE_VOTE;
  p->seed = 0;
  p->layer_id = 0;
  p->softmax_scale = 0.0f;
  p->rope_theta = 0.0f;
  p->rope_pos_offset = 0;
}

mmshift_status mmshift_output_rows(const mmshift_shape* s, int64_t* rows) {
  if (!rows) return MMSHIFT_ERR_INVALID_ARG;
  const mmshift_status st = check_shape(s);
  if (st != MMSHIFT_OK) return st;
  int64_t r = 0;
  for (int b = 0; b < s->batch; ++b)
    r += std::min<int64_t>(s->budgets[b], (int64_t)s->cu_seqlens[b + 1] - s->cu_seqlens[b]);
  *rows = r;
  return MMSHIFT_OK;
}

mmshift_status mmshift_workspace_size(const mmshift_shape* s, const mmshift_params* p,
                                      size_t* bytes) {
  if (!bytes) return MMSHIFT_ERR_INVALID_ARG;
  Problem P;
  const mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  *bytes = layout_of(P).total;
  return MMSHIFT_OK;
}


mmshift_status mmshift_prefill_stats_workspace_size(const mmshift_shape* s, size_t* bytes) {
  if (!bytes) return MMSHIFT_ERR_INVALID_ARG;
  StatsJob J;
  const mmshift_status st = stats_job(s, 0, &J);
  if (st != MMSHIFT_OK) return st;
  *bytes = align256((size_t)J.L * J.B * J.nchunk * 3 * J.ncol * sizeof(float));
  return MMSHIFT_OK;
}

mmshift_status mmshift_prefill_stats(const mmshift_shape* s, const void* Qfull,
                                     int64_t qfull_layer_stride, float* stats, void* workspace,
                                     size_t workspace_bytes, mmshift_stream_t stream) {
  StatsJob J;
  mmshift_status st = stats_job(s, qfull_layer_stride, &J);
  if (st != MMSHIFT_OK) return st;
  if (!Qfull || !stats || !workspace) return MMSHIFT_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(Qfull) & 15) return MMSHIFT_ERR_INVALID_ARG;
  size_t need = 0;
  if ((st = mmshift_prefill_stats_workspace_size(s, &need)) != MMSHIFT_OK) return st;
  if (workspace_bytes < need) return MMSHIFT_ERR_WORKSPACE;
  const cudaError_t e = launch_prefill_stats(J, Qfull, static_cast<float*>(workspace), stats,
                                             (cudaStream_t)stream, s->dtype == MMSHIFT_BF16);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_hidden_stats_workspace_size(const mmshift_shape* s, int32_t d_model,
                                                  size_t* bytes) {
  if (!bytes || d_model < 8) return MMSHIFT_ERR_INVALID_ARG;
  StatsJob J;
  const mmshift_status st = stats_job(s, 0, &J, d_model);
  if (st != MMSHIFT_OK) return st;
  *bytes = align256((size_t)J.L * J.B * J.nchunk * 3 * J.ncol * sizeof(float));
  return MMSHIFT_OK;
}

mmshift_status mmshift_hidden_stats(const mmshift_shape* s, int32_t d_model, const void* H,
                                    int64_t h_layer_stride, float* stats, void* workspace,
                                    size_t workspace_bytes, mmshift_stream_t stream) {
  if (d_model < 8) return MMSHIFT_ERR_INVALID_ARG;
  StatsJob J;
  mmshift_status st = stats_job(s, h_layer_stride, &J, d_model);
  if (st != MMSHIFT_OK) return st;
  if (!H || !stats || !workspace) return MMSHIFT_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(H) & 15) return MMSHIFT_ERR_INVALID_ARG;
  size_t need = 0;
  if ((st = mmshift_hidden_stats_workspace_size(s, d_model, &need)) != MMSHIFT_OK) return st;
  if (workspace_bytes < need) return MMSHIFT_ERR_WORKSPACE;
  const cudaError_t e = launch_prefill_stats(J, H, static_cast<float*>(workspace), stats,
                                             (cudaStream_t)stream, s->dtype == MMSHIFT_BF16);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_hidden_proxies_workspace_size(const mmshift_shape* s, int32_t d_model,
                                                     const mmshift_params* p, size_t* bytes) {
  if (!bytes) return MMSHIFT_ERR_INVALID_ARG;
  HiddenJob J;
  const mmshift_status st = hidden_job(s, d_model, p, nullptr, &J);
  if (st != MMSHIFT_OK) return st;
  *bytes = 256 + hidden_scratch_bytes(J);
  return MMSHIFT_OK;
}

mmshift_status mmshift_build_hidden_proxies(const mmshift_shape* s, int32_t d_model,
                                            const float* hstats, const void* W_Q,
                                            int64_t wq_layer_stride, const void* bias_q,
                                            const int32_t* rope_pos, const mmshift_params* p,
                                            void* proxies, void* workspace,
                                            size_t workspace_bytes, mmshift_stream_t stream) {
  HiddenJob J;
  mmshift_status st = hidden_job(s, d_model, p, rope_pos, &J);
  if (st != MMSHIFT_OK) return st;
  if (J.N == 0) return MMSHIFT_OK;
  if (!hstats || !W_Q || !proxies || !workspace) return MMSHIFT_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(W_Q) & 15) || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return MMSHIFT_ERR_INVALID_ARG;
  const int64_t dense = (int64_t)J.F * J.DM;
  if (wq_layer_stride % 8 || (J.L > 1 && wq_layer_stride && wq_layer_stride < dense))
    return MMSHIFT_ERR_INVALID_ARG;
  if (J.L > 1 && wq_layer_stride == 0) wq_layer_stride = dense;
  if (workspace_bytes < 256 + hidden_scratch_bytes(J)) return MMSHIFT_ERR_WORKSPACE;
  if (!tmap_encoder_available()) return MMSHIFT_ERR_UNSUPPORTED;
  J.hstats = hstats;
  J.bias = static_cast<const __nv_bfloat16*>(bias_q);
  J.out = static_cast<__nv_bfloat16*>(proxies);
  J.status = static_cast<int*>(workspace);
  const cudaError_t e = launch_hidden_proxies(J, static_cast<unsigned char*>(workspace) + 256, W_Q,
                                              wq_layer_stride, (cudaStream_t)stream);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_build_proxies_from_stats(const mmshift_shape* s, const float* stats,
                                                const mmshift_params* p, void* proxies,
                                                mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !stats || !proxies) return MMSHIFT_ERR_INVALID_ARG;
  if (P.Np == 0) return MMSHIFT_OK;
  Buffers bf;
  std::memset(&bf, 0, sizeof(bf));
  bf.proxies_out = proxies;
  bf.stats_in = stats;
  const cudaError_t e = launch_proxy_pack(P, bf, (cudaStream_t)stream, nullptr);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_build_proxies(const mmshift_shape* s, const void* Qwin,
                                     const mmshift_params* p, void* proxies,
                                     mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !Qwin || !proxies) return MMSHIFT_ERR_INVALID_ARG;
  if (P.Np == 0) return MMSHIFT_OK;
  Buffers bf;
  std::memset(&bf, 0, sizeof(bf));
  bf.proxies_out = proxies;
  const cudaError_t e = launch_proxy_pack(P, bf, (cudaStream_t)stream, Qwin);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_proxy_mass(const mmshift_shape* s, const void* K, const void* Qwin,
                                  const void* proxies, const mmshift_params* p,
                                  float* group_mass, float* anchor, float* mass,
                                  void* workspace, size_t workspace_bytes,
                                  mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !K || !Qwin || !anchor || (P.G && !group_mass)) return MMSHIFT_ERR_INVALID_ARG;
  set_score_path(P, K);
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  bf.proxies_in = proxies;
  if (P.G) bf.gmass = group_mass;
  bf.anchor = anchor;
  bf.mass = mass;
  return run_mass(P, bf, K, Qwin, (cudaStream_t)stream);
}

mmshift_status mmshift_scores_topk(const mmshift_shape* s, const mmshift_params* p,
                                   const float* group_mass, const float* anchor,
                                   float* scores, int32_t* out_idx,
                                   void* workspace, size_t workspace_bytes,
                                   mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !out_idx || (P.G && !group_mass)) return MMSHIFT_ERR_INVALID_ARG;
  if (P.mode == MMSHIFT_SCORE_VOTE && !anchor) return MMSHIFT_ERR_INVALID_ARG;
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  if (P.G) bf.gmass = const_cast<float*>(group_mass);
  if (anchor) bf.anchor = const_cast<float*>(anchor);
  if (scores) { bf.scores = scores; bf.scores_out = 1; }
  const cudaStream_t cs = (cudaStream_t)stream;
  cudaError_t e = cudaSuccess;
  if (P.mode == MMSHIFT_SCORE_VOTE) e = launch_cover(P, bf, cs);
  if (e == cudaSuccess) e = launch_topk(P, bf, cs, out_idx, false);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_topk(const mmshift_shape* s, const float* scores, int32_t* out_idx,
                            void* workspace, size_t workspace_bytes, mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, nullptr, &P);
  if (st != MMSHIFT_OK) return st;
  if (!scores || !out_idx) return MMSHIFT_ERR_INVALID_ARG;
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  bf.scores = const_cast<float*>(scores);
  const cudaError_t e = launch_topk(P, bf, (cudaStream_t)stream, out_idx, true);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_topk_head_budgets(const mmshift_shape* s, const float* scores,
                                         const int32_t* head_budgets, int32_t* out_idx,
                                         int32_t* out_count, void* workspace,
                                         size_t workspace_bytes, mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, nullptr, &P);
  if (st != MMSHIFT_OK) return st;
  if (!scores || !head_budgets || !out_idx) return MMSHIFT_ERR_INVALID_ARG;
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  bf.scores = const_cast<float*>(scores);
  bf.head_budget = head_budgets;
  bf.out_count = out_count;
  const cudaError_t e = launch_topk(P, bf, (cudaStream_t)stream, out_idx, true);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_gather(const mmshift_shape* s, const void* K, const void* V,
                              const int32_t* idx, void* out_K, void* out_V,
                              void* workspace, size_t workspace_bytes,
                              mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = prepare(s, nullptr, &P);
  if (st != MMSHIFT_OK) return st;
  if (!K || !V || !idx || !out_K || !out_V) return MMSHIFT_ERR_INVALID_ARG;
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  if (!device_readable(K) || !device_readable(V)) return MMSHIFT_ERR_INVALID_ARG;
  const cudaError_t e = launch_gather(P, bf, (cudaStream_t)stream, K, V, idx, out_K, out_V);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_select(const mmshift_shape* s, const void* K, const void* V,
                              const void* Qwin, const void* proxies_in,
                              const mmshift_params* p, int32_t* out_idx, void* out_K,
                              void* out_V, const mmshift_debug* dbg, void* workspace,
                              size_t workspace_bytes, mmshift_stream_t stream) {
  return select_impl(s, K, V, Qwin, proxies_in, nullptr, p, out_idx, out_K, out_V, dbg,
                     workspace, workspace_bytes, stream);
}

mmshift_status mmshift_select_head_budgets(const mmshift_shape* s, const void* K, const void* V,
                                           const void* Qwin, const void* proxies_in,
                                           const int32_t* head_budgets, const mmshift_params* p,
                                           int32_t* out_idx, int32_t* out_count, void* out_K,
                                           void* out_V, const mmshift_debug* dbg, void* workspace,
                                           size_t workspace_bytes, mmshift_stream_t stream) {
  if (!head_budgets) return MMSHIFT_ERR_INVALID_ARG;
  return select_impl(s, K, V, Qwin, proxies_in, nullptr, p, out_idx, out_K, out_V, dbg, workspace,
                     workspace_bytes, stream, head_budgets, out_count);
}

mmshift_status mmshift_select_with_stats(const mmshift_shape* s, const void* K, const void* V,
                                         const void* Qwin, const float* stats,
                                         const mmshift_params* p, int32_t* out_idx, void* out_K,
                                         void* out_V, const mmshift_debug* dbg, void* workspace,
                                         size_t workspace_bytes, mmshift_stream_t stream) {
  if (!stats) return MMSHIFT_ERR_INVALID_ARG;
  return select_impl(s, K, V, Qwin, nullptr, stats, p, out_idx, out_K, out_V, dbg, workspace,
                     workspace_bytes, stream);
}

// Hyper-parameters under which steps 2-4 give the coverage masses: the
// decode queries are the proxies, one per group.
static mmshift_status coverage_params(int32_t n_dec, float softmax_scale, mmshift_params* p) {
  if (n_dec < 1 || n_dec > 1024) return MMSHIFT_ERR_INVALID_ARG;
  if (!(softmax_scale >= 0.f) || !std::isfinite(softmax_scale)) return MMSHIFT_ERR_INVALID_ARG;
  mmshift_default_params(p);
  p->n_proxies = n_dec;
  p->n_groups = n_dec;
  p->softmax_scale = softmax_scale;
  p->score_mode = MMSHIFT_SCORE_MASS;
  return MMSHIFT_OK;
}

mmshift_status mmshift_coverage_workspace_size(const mmshift_shape* s, int32_t n_dec,
                                               size_t* bytes) {
  mmshift_params p;
  const mmshift_status st = coverage_params(n_dec, 0.f, &p);
  if (st != MMSHIFT_OK) return st;
  return mmshift_workspace_size(s, &p, bytes);
}

mmshift_status mmshift_coverage(const mmshift_shape* s, const void* K, const void* Qwin,
                                const void* dec_q, int32_t n_dec, float softmax_scale,
                                const int32_t* idx, float* cov, void* workspace,
                                size_t workspace_bytes, mmshift_stream_t stream) {
  mmshift_params p;
  mmshift_status st = coverage_params(n_dec, softmax_scale, &p);
  if (st != MMSHIFT_OK) return st;
  Problem P;
  if ((st = prepare(s, &p, &P)) != MMSHIFT_OK) return st;
  if (!K || !Qwin || !dec_q || !idx || !cov) return MMSHIFT_ERR_INVALID_ARG;
  set_score_path(P, K);
  Buffers bf;
  if ((st = carve(P, workspace, workspace_bytes, &bf)) != MMSHIFT_OK) return st;
  bf.proxies_in = dec_q;
  bf.mass = nullptr;
  const cudaStream_t cs = (cudaStream_t)stream;
  if ((st = run_mass(P, bf, K, Qwin, cs)) != MMSHIFT_OK) return st;
  const cudaError_t e = launch_coverage(P, bf, idx, cov, cs);
  return e == cudaSuccess ? MMSHIFT_OK : cuda_fail(e);
}

mmshift_status mmshift_poll_status(void* workspace, mmshift_stream_t stream) {
  if (!workspace) return MMSHIFT_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e);
  int word = 0;
  if ((e = cudaMemcpy(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e);
  if ((e = cudaMemset(workspace, 0, sizeof(int))) != cudaSuccess) return cuda_fail(e);
  if (word & kStatusTimeout) return MMSHIFT_ERR_TIMEOUT;
  if (word) return MMSHIFT_ERR_DEVICE;
  return MMSHIFT_OK;
}

const char* mmshift_status_string(mmshift_status st) {
  switch (st) {
    case MMSHIFT_OK: return "ok";
    case MMSHIFT_ERR_INVALID_ARG: return "invalid argument";
    case MMSHIFT_ERR_UNSUPPORTED: return "unsupported configuration";
    case MMSHIFT_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case MMSHIFT_ERR_CUDA: return "CUDA runtime error";
    case MMSHIFT_ERR_TIMEOUT: return "device-side wait timed out";
    case MMSHIFT_ERR_DEVICE: return "device-side check failed";
  }
  return "unknown status";
}

const char* mmshift_last_cuda_error(void) { return g_cuda_error.c_str(); }

}  // extern "C"
