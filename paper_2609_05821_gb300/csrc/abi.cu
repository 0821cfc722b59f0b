// C ABI: host-side argument checks, workspace sizing and launch sequencing.
// Every check runs before anything is enqueued; nothing here allocates.
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <string>

#include "internal.cuh"

using namespace conduit;

namespace {

std::atomic<int64_t> g_launches{0};

thread_local std::string g_last_error;

conduit_status fail(conduit_status code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

conduit_status cuda_fail(cudaError_t err, const char* what) {
  return fail(CONDUIT_ERR_CUDA, "%s: %s", what, cudaGetErrorString(err));
}

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

conduit_status check_batch(const conduit_batch* b) {
  if (!b) return fail(CONDUIT_ERR_INVALID_ARG, "batch is NULL");
  if (b->num_requests < 1) return fail(CONDUIT_ERR_INVALID_ARG, "num_requests must be >= 1");
  if (b->num_images < b->num_requests)
    return fail(CONDUIT_ERR_INVALID_ARG, "num_images must be >= num_requests");
  if (!b->tok_off || !b->img_off || !b->req_img_off || !b->q_off)
    return fail(CONDUIT_ERR_INVALID_ARG, "a host offset array is NULL");
  if (!b->tok_off_dev || !b->img_off_dev || !b->req_img_off_dev || !b->q_off_dev)
    return fail(CONDUIT_ERR_INVALID_ARG, "a device offset array is NULL");
  const int R = b->num_requests, K = b->num_images;
  if (b->tok_off[0] != 0 || b->q_off[0] != 0 || b->req_img_off[0] != 0)
    return fail(CONDUIT_ERR_INVALID_ARG, "tok_off, q_off and req_img_off must start at 0");
  if (b->req_img_off[R] != K)
    return fail(CONDUIT_ERR_INVALID_ARG, "req_img_off[R] must equal num_images");
  for (int r = 0; r < R; ++r) {
    if (b->tok_off[r + 1] <= b->tok_off[r])
      return fail(CONDUIT_ERR_INVALID_ARG, "request %d has no visual tokens", r);
    if (b->q_off[r + 1] < b->q_off[r])
      return fail(CONDUIT_ERR_INVALID_ARG, "q_off must be non-decreasing (request %d)", r);
    const int j0 = b->req_img_off[r], j1 = b->req_img_off[r + 1];
    if (j1 <= j0) return fail(CONDUIT_ERR_INVALID_ARG, "request %d has no images", r);
    if (j1 - j0 > kMaxImagesPerRequest)
      return fail(CONDUIT_ERR_UNSUPPORTED, "request %d has more than %d images", r,
                  kMaxImagesPerRequest);
    if (b->img_off[j0] != b->tok_off[r] || b->img_off[j1] != b->tok_off[r + 1])
      return fail(CONDUIT_ERR_INVALID_ARG, "images of request %d do not tile its tokens", r);
    for (int j = j0; j < j1; ++j)
      if (b->img_off[j + 1] <= b->img_off[j])
        return fail(CONDUIT_ERR_INVALID_ARG, "image %d is empty or out of order", j);
  }
  return CONDUIT_OK;
}

conduit_status check_kv(const conduit_kv* kv, const conduit_batch* b) {
  if (!kv) return fail(CONDUIT_ERR_INVALID_ARG, "kv is NULL");
  if (kv->num_layers < 1 || kv->num_q_heads < 1 || kv->num_kv_heads < 1)
    return fail(CONDUIT_ERR_INVALID_ARG, "layer and head counts must be >= 1");
  if (kv->num_q_heads % kv->num_kv_heads)
    return fail(CONDUIT_ERR_INVALID_ARG, "num_q_heads must be a multiple of num_kv_heads");
  if (kv->head_dim < 8 || kv->head_dim > 256 || kv->head_dim % 8)
    return fail(CONDUIT_ERR_UNSUPPORTED, "head_dim must be a multiple of 8 in [8, 256]");
  if (kv->dtype != CONDUIT_F32 && kv->dtype != CONDUIT_BF16)
    return fail(CONDUIT_ERR_INVALID_ARG, "dtype must be CONDUIT_F32 or CONDUIT_BF16");
  if (!kv->k || !kv->v) return fail(CONDUIT_ERR_INVALID_ARG, "kv->k or kv->v is NULL");
  if (!aligned16(kv->k) || !aligned16(kv->v))
    return fail(CONDUIT_ERR_INVALID_ARG, "kv->k and kv->v must be 16-byte aligned");
  if ((kv->num_q_heads / kv->num_kv_heads) * kv->head_dim > 4096)
    return fail(CONDUIT_ERR_UNSUPPORTED, "(Hq/Hkv) * head_dim must be <= 4096");
  if (kv->page_size < 0) return fail(CONDUIT_ERR_INVALID_ARG, "page_size must be >= 0");
  if (kv->page_size > 0) {
    if (!kv->page_table || kv->num_pages < 1 || kv->max_pages_per_req < 1)
      return fail(CONDUIT_ERR_INVALID_ARG, "paged cache needs page_table, num_pages, max_pages_per_req");
    for (int r = 0; r < b->num_requests; ++r) {
      const int64_t n = b->tok_off[r + 1] - b->tok_off[r];
      if (n > int64_t(kv->max_pages_per_req) * kv->page_size)
        return fail(CONDUIT_ERR_INVALID_ARG, "request %d has more tokens than its page-table row holds", r);
    }
  }
  return CONDUIT_OK;
}

KvDev make_kv(const conduit_kv* kv, const conduit_batch* b) {
  KvDev d{};
  d.k = kv->k;
  d.v = kv->v;
  d.L = kv->num_layers;
  d.Hq = kv->num_q_heads;
  d.Hkv = kv->num_kv_heads;
  d.d = kv->head_dim;
  d.G = kv->num_q_heads / kv->num_kv_heads;
  d.dtype = kv->dtype;
  d.page_size = kv->page_size;
  d.num_pages = kv->num_pages;
  d.max_pages = kv->max_pages_per_req;
  d.page_table = kv->page_table;
  d.n_tot = b->tok_off[b->num_requests];
  return d;
}

BatchDev make_batch(const conduit_batch* b) {
  return BatchDev{b->num_requests, b->num_images, b->tok_off_dev, b->img_off_dev,
                  b->req_img_off_dev, b->q_off_dev};
}

conduit_status make_layers(const conduit_kv* kv, const int32_t* layers, int32_t n_layers,
                           LayerList* out) {
  if (!layers) {
    if (n_layers != 0 && n_layers != kv->num_layers)
      return fail(CONDUIT_ERR_INVALID_ARG, "layers == NULL needs n_layers == 0 or num_layers");
    if (kv->num_layers > CONDUIT_MAX_LAYERS)
      return fail(CONDUIT_ERR_UNSUPPORTED, "more than %d layers", CONDUIT_MAX_LAYERS);
    out->n = kv->num_layers;
    for (int i = 0; i < kv->num_layers; ++i) out->ids[i] = i;
    return CONDUIT_OK;
  }
  if (n_layers < 1 || n_layers > CONDUIT_MAX_LAYERS)
    return fail(CONDUIT_ERR_INVALID_ARG, "n_layers must be in [1, %d]", CONDUIT_MAX_LAYERS);
  for (int i = 0; i < n_layers; ++i) {
    if (layers[i] < 0 || layers[i] >= kv->num_layers)
      return fail(CONDUIT_ERR_INVALID_ARG, "layer id %d out of range", layers[i]);
    if (i && layers[i] <= layers[i - 1])
      return fail(CONDUIT_ERR_INVALID_ARG, "layer ids must be strictly increasing");
    out->ids[i] = layers[i];
  }
  out->n = n_layers;
  return CONDUIT_OK;
}

struct ScoreLayout {
  bool tc;     // tensor-core kernel (bf16, head_dim 128) or the CUDA-core ones
  int rg_max;  // row groups per slab (column-sum partials per KV head)
  int group_rows;
  int parts;   // partials per row group and per value norm (2 for the tensor-core kernel)
  size_t stats, pa, pa2, ss, attn, total;
};

// What a scoring call computes (conduit_score_opts with its defaults filled in).
struct ScoreMode {
  bool rms;                // RMS statistic in s (Eq. 4) instead of the mean (Eq. 6)
  int vmode;               // 0 value norms from V, 1 from the side cache, 2 none
  const float* vnorm;
  const float* extra_lse;  // full-context softmax denominators, or NULL
};

conduit_status read_opts(const conduit_score_opts* o, ScoreMode* m) {
  *m = ScoreMode{false, 0, nullptr, nullptr};
  if (!o) return CONDUIT_OK;
  if (o->statistic != CONDUIT_STAT_MEAN && o->statistic != CONDUIT_STAT_RMS)
    return fail(CONDUIT_ERR_INVALID_ARG, "opts->statistic must be CONDUIT_STAT_MEAN or _RMS");
  if (o->value_norm < CONDUIT_VNORM_FROM_V || o->value_norm > CONDUIT_VNORM_NONE)
    return fail(CONDUIT_ERR_INVALID_ARG, "opts->value_norm must be a CONDUIT_VNORM_* value");
  if ((o->value_norm == CONDUIT_VNORM_SIDE_CACHE) != (o->vnorm != nullptr))
    return fail(CONDUIT_ERR_INVALID_ARG,
                "opts->vnorm is required with CONDUIT_VNORM_SIDE_CACHE and must be NULL otherwise");
  if (o->extra_lse && reinterpret_cast<uintptr_t>(o->extra_lse) % 4)
    return fail(CONDUIT_ERR_INVALID_ARG, "opts->extra_lse must be 4-byte aligned");
  *m = ScoreMode{o->statistic == CONDUIT_STAT_RMS, o->value_norm, o->vnorm, o->extra_lse};
  return CONDUIT_OK;
}

// Without value partials (vmode != 0) there is no ss region; the RMS
// statistic adds a pa2 region of the size of pa.
ScoreLayout score_layout(const conduit_kv* kv, const conduit_batch* b, int n_layers,
                         const ScoreMode& mode) {
  const bool normed = mode.vmode != 0;
  const int R = b->num_requests;
  const size_t n_tot = size_t(b->tok_off[R]);
  const size_t q_tot = size_t(b->q_off[R]);
  ScoreLayout s{};
  s.tc = score_tc_supported(make_kv(kv, b));
  s.rg_max = 1;
  s.parts = s.tc ? 2 : 1;
  if (s.tc) {
    s.group_rows = kScoreGroupRows;
    const int G = kv->num_q_heads / kv->num_kv_heads;
    for (int r = 0; r < R; ++r)
      s.rg_max = std::max(s.rg_max, score_tc_groups(G * (b->q_off[r + 1] - b->q_off[r])));
  }
  const int64_t total_rows = int64_t(n_layers) * kv->num_q_heads * int64_t(q_tot);
  size_t off = 0;
  s.stats = off;
  if (!s.tc) off += align_up(size_t(total_rows) * sizeof(float2));  // (max, sum) per row
  const size_t pa_bytes =
      align_up(size_t(n_layers) * kv->num_kv_heads * s.rg_max * s.parts * n_tot * sizeof(float));
  s.pa = off;
  off += pa_bytes;
  s.pa2 = off;
  if (mode.rms) off += pa_bytes;
  s.ss = off;
  if (!normed) off += align_up(size_t(n_layers) * kv->num_kv_heads * s.parts * n_tot * sizeof(float));
  s.attn = off;
  off += align_up(n_tot * sizeof(float));
  s.total = off;
  return s;
}

int max_tokens(const conduit_batch* b) {
  int m = 0;
  for (int r = 0; r < b->num_requests; ++r) m = std::max(m, b->tok_off[r + 1] - b->tok_off[r]);
  return m;
}

conduit_status check_workspace(void* ws, size_t have, size_t need) {
  if (need == 0) return CONDUIT_OK;
  if (!ws) return fail(CONDUIT_ERR_WORKSPACE, "workspace is NULL but %zu bytes are needed", need);
  if (reinterpret_cast<uintptr_t>(ws) % kAlign)
    return fail(CONDUIT_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (have < need)
    return fail(CONDUIT_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", have, need);
  return CONDUIT_OK;
}

conduit_status check_selection(const conduit_batch* b, const int32_t* idx_off,
                               const int32_t* idx_off_dev, bool need_idx, const int32_t* idx) {
  if (!idx_off || !idx_off_dev)
    return fail(CONDUIT_ERR_INVALID_ARG, "idx_off (host) and idx_off_dev (device) are required");
  if (idx_off[0] != 0) return fail(CONDUIT_ERR_INVALID_ARG, "idx_off[0] must be 0");
  for (int r = 0; r < b->num_requests; ++r) {
    const int kr = idx_off[r + 1] - idx_off[r];
    if (kr < 0 || kr > b->tok_off[r + 1] - b->tok_off[r])
      return fail(CONDUIT_ERR_INVALID_ARG, "budget of request %d is outside [0, N_r]", r);
  }
  if (need_idx && idx_off[b->num_requests] > 0 && !idx)
    return fail(CONDUIT_ERR_INVALID_ARG, "idx is NULL");
  return CONDUIT_OK;
}

int max_budget(const conduit_batch* b, const int32_t* idx_off) {
  int m = 0;
  for (int r = 0; r < b->num_requests; ++r) m = std::max(m, idx_off[r + 1] - idx_off[r]);
  return m;
}

conduit_status check_norm_cache(const conduit_kv* kv, const float* vnorm) {
  if (!vnorm) return fail(CONDUIT_ERR_INVALID_ARG, "vnorm is NULL");
  if (reinterpret_cast<uintptr_t>(vnorm) % 4)
    return fail(CONDUIT_ERR_INVALID_ARG, "vnorm must be 4-byte aligned");
  if (kv->num_layers > 65535)
    return fail(CONDUIT_ERR_UNSUPPORTED, "the norm cache takes at most 65535 layers");
  return CONDUIT_OK;
}

// Every scoring entry point: conduit_score_ex with the options read into `mode`.
// The selection that conduit_score_select_topk appends to a scoring call.
struct SelectTail {
  float lambda;
  const int32_t* idx_off;      // host prefix sums of the budgets
  const int32_t* idx_off_dev;  // the same on the device
  int32_t* idx;
  uint8_t* mask;
  float* s_hat;
  float* coeff;
};

// Workspace of conduit_score_select_topk: the scoring call's, then one
// arrival counter per request (fused tail) and the selection's keys (the
// separate launches, for requests of more than 8192 tokens).
struct FusedLayout {
  ScoreLayout score;
  size_t arrivals, keys, total;
};

FusedLayout fused_layout(const conduit_kv* kv, const conduit_batch* b, int n_layers, const ScoreMode& mode) {
  FusedLayout f;
  f.score = score_layout(kv, b, n_layers, mode);
  f.arrivals = f.score.total;
  f.keys = f.arrivals + align_up(size_t(b->num_requests) * sizeof(int32_t));
  f.total = f.keys + align_up(size_t(b->tok_off[b->num_requests]) * sizeof(uint32_t));
  return f;
}

conduit_status score_impl(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                          const int32_t* layers, int32_t n_layers, const ScoreMode& mode, float* s,
                          float* attn_sum, float* g, void* workspace, size_t workspace_bytes,
                          int32_t* status, void* stream, const SelectTail* tail = nullptr) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if (!q || !s || !g) return fail(CONDUIT_ERR_INVALID_ARG, "q, s and g are required");
  if (tail) {
    if (!(tail->lambda >= 0.f && tail->lambda <= 1.f))
      return fail(CONDUIT_ERR_INVALID_ARG, "lambda must lie in [0, 1]");
    if ((st = check_selection(batch, tail->idx_off, tail->idx_off_dev, true, tail->idx))) return st;
  }
  if (!aligned16(q)) return fail(CONDUIT_ERR_INVALID_ARG, "q must be 16-byte aligned");
  for (int r = 0; r < batch->num_requests; ++r)
    if (batch->q_off[r + 1] == batch->q_off[r])
      return fail(CONDUIT_ERR_INVALID_ARG, "request %d has an empty scoring span", r);
  static thread_local LayerList ll;
  if ((st = make_layers(kv, layers, n_layers, &ll))) return st;
  const bool normed = mode.vmode != 0;
  if (mode.vmode == 1 && (st = check_norm_cache(kv, mode.vnorm))) return st;
  const FusedLayout flay = fused_layout(kv, batch, ll.n, mode);
  const ScoreLayout& lay = flay.score;
  if ((st = check_workspace(workspace, workspace_bytes, tail ? flay.total : lay.total))) return st;

  const KvDev kd = make_kv(kv, batch);
  const BatchDev bd = make_batch(batch);
  const int R = batch->num_requests;
  int max_tok = 0, max_rows = 0;
  for (int r = 0; r < R; ++r) {
    max_tok = std::max(max_tok, batch->tok_off[r + 1] - batch->tok_off[r]);
    max_rows = std::max(max_rows, kd.G * (batch->q_off[r + 1] - batch->q_off[r]));
  }
  char* ws = static_cast<char*>(workspace);
  float2* stats = reinterpret_cast<float2*>(ws + lay.stats);
  float* pa = reinterpret_cast<float*>(ws + lay.pa);
  float* ss = normed ? nullptr : reinterpret_cast<float*>(ws + lay.ss);
  float* pa2 = mode.rms ? reinterpret_cast<float*>(ws + lay.pa2) : nullptr;
  float* attn = attn_sum ? attn_sum : reinterpret_cast<float*>(ws + lay.attn);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  cudaError_t err;
  const bool fused = tail && finalize_select_supported(max_tok, kd.n_tot);
  int32_t* arrivals = reinterpret_cast<int32_t*>(ws + flay.arrivals);
  if (fused && (err = cudaMemsetAsync(arrivals, 0, size_t(R) * sizeof(int32_t), cs)))
    return cuda_fail(err, "score_select");
  if (lay.tc) {  // the tensor-core kernel also streams V for the value norms (unless normed)
    err = launch_score_tc(kd, bd, batch->q_off, q, batch->q_off[R], ll, lay.rg_max, pa, ss, pa2,
                          mode.extra_lse, status, cs);
  } else {
    if (!normed && (err = launch_value_sumsq(kd, bd, ll, max_tok, ss, cs)))
      return cuda_fail(err, "value_sumsq");
    err = launch_score_simt(kd, bd, q, batch->q_off[R], ll, max_rows, max_tok, stats, pa, pa2,
                            mode.extra_lse, cs);
  }
  if (err) return cuda_fail(err, "score");
  if (fused) {
    if ((err = launch_finalize_select(pa, pa2, ss, mode.vnorm, mode.vmode, ll, bd, ll.n, kd.Hkv, kd.Hq,
                                      lay.rg_max, lay.group_rows, lay.parts, kd.n_tot, max_tok, s, attn, g,
                                      tail->lambda, tail->idx_off_dev, tail->idx, tail->mask, tail->s_hat,
                                      tail->coeff, arrivals, status, cs)))
      return cuda_fail(err, "finalize_select");
    return CONDUIT_OK;
  }
  if ((err = launch_finalize(pa, pa2, ss, mode.vnorm, mode.vmode, ll, bd, ll.n, kd.Hkv, kd.Hq,
                             lay.rg_max, lay.group_rows, lay.parts, kd.n_tot, s, attn, g, status, cs)))
    return cuda_fail(err, "finalize");
  if (tail &&
      (err = launch_select(bd, max_tok, s, g, tail->lambda, tail->idx_off_dev, tail->idx, tail->mask,
                           tail->s_hat, tail->coeff, reinterpret_cast<uint32_t*>(ws + flay.keys), status, cs)))
    return cuda_fail(err, "select");
  return CONDUIT_OK;
}

}  // namespace

namespace conduit {
void count_launches(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace conduit

extern "C" {

int32_t conduit_version(void) { return CONDUIT_VERSION; }

int64_t conduit_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char* conduit_last_error_string(void) { return g_last_error.c_str(); }

int32_t conduit_budget(double r, int64_t n_vis) {
  if (!(r >= 0.0 && r <= 1.0) || n_vis < 0) return -1;
  const double k = std::floor(r * double(n_vis) + 1e-9);
  return int32_t(std::min<double>(k, double(n_vis)));
}

conduit_status conduit_score_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                            int32_t n_layers, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  const int nl = n_layers > 0 ? n_layers : kv->num_layers;
  *bytes = score_layout(kv, batch, nl, ScoreMode{false, 0, nullptr, nullptr}).total;
  return CONDUIT_OK;
}

conduit_status conduit_score(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                             const int32_t* layers, int32_t n_layers, float* s, float* attn_sum,
                             float* g, void* workspace, size_t workspace_bytes, int32_t* status,
                             void* stream) {
  return score_impl(kv, batch, q, layers, n_layers, ScoreMode{false, 0, nullptr, nullptr}, s,
                    attn_sum, g, workspace, workspace_bytes, status, stream);
}

conduit_status conduit_score_ex_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                               int32_t n_layers, const conduit_score_opts* opts,
                                               size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  ScoreMode mode;
  if ((st = read_opts(opts, &mode))) return st;
  const int nl = n_layers > 0 ? n_layers : kv->num_layers;
  *bytes = score_layout(kv, batch, nl, mode).total;
  return CONDUIT_OK;
}

conduit_status conduit_score_ex(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                                const int32_t* layers, int32_t n_layers,
                                const conduit_score_opts* opts, float* s, float* attn_sum,
                                float* g, void* workspace, size_t workspace_bytes,
                                int32_t* status, void* stream) {
  conduit_status st;
  ScoreMode mode;
  if ((st = read_opts(opts, &mode))) return st;
  return score_impl(kv, batch, q, layers, n_layers, mode, s, attn_sum, g, workspace,
                    workspace_bytes, status, stream);
}

conduit_status conduit_score_select_topk_workspace_size(const conduit_kv* kv,
                                                        const conduit_batch* batch,
                                                        int32_t n_layers,
                                                        const conduit_score_opts* opts,
                                                        size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  ScoreMode mode;
  if ((st = read_opts(opts, &mode))) return st;
  const int nl = n_layers > 0 ? n_layers : kv->num_layers;
  *bytes = fused_layout(kv, batch, nl, mode).total;
  return CONDUIT_OK;
}

conduit_status conduit_score_select_topk(const conduit_kv* kv, const conduit_batch* batch,
                                         const void* q, const int32_t* layers, int32_t n_layers,
                                         const conduit_score_opts* opts, float lambda,
                                         const int32_t* idx_off, const int32_t* idx_off_dev,
                                         float* s, float* attn_sum, float* g, int32_t* idx,
                                         uint8_t* mask, float* s_hat, float* coeff,
                                         void* workspace, size_t workspace_bytes, int32_t* status,
                                         void* stream) {
  conduit_status st;
  ScoreMode mode;
  if ((st = read_opts(opts, &mode))) return st;
  const SelectTail tail{lambda, idx_off, idx_off_dev, idx, mask, s_hat, coeff};
  return score_impl(kv, batch, q, layers, n_layers, mode, s, attn_sum, g, workspace, workspace_bytes,
                    status, stream, &tail);
}

conduit_status conduit_value_norms(const conduit_kv* kv, const conduit_batch* batch, float* vnorm,
                                   void* stream) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if ((st = check_norm_cache(kv, vnorm))) return st;
  cudaError_t err = launch_value_norms(make_kv(kv, batch), make_batch(batch), nullptr, nullptr,
                                       batch->tok_off[batch->num_requests], vnorm,
                                       static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "value_norms");
  return CONDUIT_OK;
}

conduit_status conduit_value_norms_update(const conduit_kv* kv, const conduit_batch* batch,
                                          const int32_t* idx, const int32_t* idx_off,
                                          const int32_t* idx_off_dev, float* vnorm, void* stream) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  if ((st = check_norm_cache(kv, vnorm))) return st;
  cudaError_t err = launch_value_norms(make_kv(kv, batch), make_batch(batch), idx, idx_off_dev,
                                       idx_off[batch->num_requests], vnorm,
                                       static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "value_norms_update");
  return CONDUIT_OK;
}

conduit_status conduit_score_with_norms_workspace_size(const conduit_kv* kv,
                                                       const conduit_batch* batch,
                                                       int32_t n_layers, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  const int nl = n_layers > 0 ? n_layers : kv->num_layers;
  *bytes = score_layout(kv, batch, nl, ScoreMode{false, 1, nullptr, nullptr}).total;
  return CONDUIT_OK;
}

conduit_status conduit_score_with_norms(const conduit_kv* kv, const conduit_batch* batch,
                                        const void* q, const int32_t* layers, int32_t n_layers,
                                        const float* vnorm, float* s, float* attn_sum, float* g,
                                        void* workspace, size_t workspace_bytes, int32_t* status,
                                        void* stream) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if ((st = check_norm_cache(kv, vnorm))) return st;
  return score_impl(kv, batch, q, layers, n_layers, ScoreMode{false, 1, vnorm, nullptr}, s,
                    attn_sum, g, workspace, workspace_bytes, status, stream);
}

conduit_status conduit_select_workspace_size(const conduit_batch* batch, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch))) return st;
  *bytes = align_up(size_t(batch->tok_off[batch->num_requests]) * sizeof(uint32_t));
  return CONDUIT_OK;
}

conduit_status conduit_select_topk(const conduit_batch* batch, const float* s, const float* g,
                                   float lambda, const int32_t* idx_off,
                                   const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                   float* s_hat, float* coeff, void* workspace,
                                   size_t workspace_bytes, int32_t* status, void* stream) {
  conduit_status st;
  if ((st = check_batch(batch))) return st;
  if (!s || !g) return fail(CONDUIT_ERR_INVALID_ARG, "s and g are required");
  if (!(lambda >= 0.f && lambda <= 1.f))
    return fail(CONDUIT_ERR_INVALID_ARG, "lambda must lie in [0, 1]");
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  size_t need = 0;
  conduit_select_workspace_size(batch, &need);
  if ((st = check_workspace(workspace, workspace_bytes, need))) return st;
  cudaError_t err = launch_select(make_batch(batch), max_tokens(batch), s, g, lambda, idx_off_dev, idx, mask, s_hat,
                                  coeff, static_cast<uint32_t*>(workspace), status,
                                  static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "select");
  return CONDUIT_OK;
}

conduit_status conduit_select_topk_noalloc(const conduit_batch* batch, const float* s,
                                           const float* g, float lambda, const int32_t* idx_off,
                                           const int32_t* idx_off_dev, int32_t* idx,
                                           uint8_t* mask, float* s_hat, float* coeff,
                                           int32_t* status, void* stream) {
  conduit_status st;
  if ((st = check_batch(batch))) return st;
  if (!s || !g) return fail(CONDUIT_ERR_INVALID_ARG, "s and g are required");
  if (!(lambda >= 0.f && lambda <= 1.f))
    return fail(CONDUIT_ERR_INVALID_ARG, "lambda must lie in [0, 1]");
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  const int64_t n_tot = batch->tok_off[batch->num_requests];
  if (n_tot > select_noalloc_max_tokens() || n_tot > CONDUIT_NOALLOC_MAX_TOKENS)
    return fail(CONDUIT_ERR_UNSUPPORTED,
                "batch has %lld tokens; the static scratch of conduit_select_topk_noalloc holds %d",
                static_cast<long long>(n_tot), CONDUIT_NOALLOC_MAX_TOKENS);
  cudaError_t err = launch_select_noalloc(make_batch(batch), max_tokens(batch), s, g, lambda, idx_off_dev, idx, mask,
                                          s_hat, coeff, status, static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "select_noalloc");
  return CONDUIT_OK;
}

conduit_status conduit_select_quota_workspace_size(const conduit_batch* batch, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch))) return st;
  *bytes = align_up(size_t(batch->tok_off[batch->num_requests]) * sizeof(uint32_t)) +
           align_up(quota_scratch_bytes(batch->num_images));
  return CONDUIT_OK;
}

conduit_status conduit_select_quota(const conduit_batch* batch, const float* s, const float* g,
                                    float lambda, const int32_t* idx_off,
                                    const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                    float* s_hat, float* coeff, int32_t* quota, void* workspace,
                                    size_t workspace_bytes, int32_t* status, void* stream) {
  conduit_status st;
  if ((st = check_batch(batch))) return st;
  if (!s || !g) return fail(CONDUIT_ERR_INVALID_ARG, "s and g are required");
  if (!(lambda >= 0.f && lambda <= 1.f))
    return fail(CONDUIT_ERR_INVALID_ARG, "lambda must lie in [0, 1]");
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  size_t need = 0;
  conduit_select_quota_workspace_size(batch, &need);
  if ((st = check_workspace(workspace, workspace_bytes, need))) return st;
  int max_images = 0, max_image_tokens = 0;
  for (int r = 0; r < batch->num_requests; ++r)
    max_images = std::max(max_images, batch->req_img_off[r + 1] - batch->req_img_off[r]);
  for (int j = 0; j < batch->num_images; ++j)
    max_image_tokens = std::max(max_image_tokens, batch->img_off[j + 1] - batch->img_off[j]);
  char* ws = static_cast<char*>(workspace);
  const size_t keys_bytes = align_up(size_t(batch->tok_off[batch->num_requests]) * sizeof(uint32_t));
  cudaError_t err = launch_select_quota(make_batch(batch), max_images, max_image_tokens, s, g, lambda,
                                        idx_off_dev, idx, mask, s_hat, coeff, quota,
                                        reinterpret_cast<uint32_t*>(ws), ws + keys_bytes, status,
                                        static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "select_quota");
  return CONDUIT_OK;
}

static conduit_status kv_copy(const conduit_kv* kv, const conduit_batch* batch,
                              const int32_t* idx, const int32_t* idx_off,
                              const int32_t* idx_off_dev, void* rows_k, void* rows_v,
                              const void* new_k, const void* new_v, int mode, void* stream) {
  static const char* names[3] = {"kv_gather", "kv_scatter", "kv_exchange"};
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  const int n_sel = idx_off[batch->num_requests];
  if (n_sel > 0 && (!rows_k || !rows_v))
    return fail(CONDUIT_ERR_INVALID_ARG, "the K and V row buffers are required");
  if (n_sel > 0 && (!aligned16(rows_k) || !aligned16(rows_v)))
    return fail(CONDUIT_ERR_INVALID_ARG, "the K and V row buffers must be 16-byte aligned");
  if (mode == 2 && n_sel > 0) {
    if (!new_k || !new_v) return fail(CONDUIT_ERR_INVALID_ARG, "k_rows and v_rows are required");
    if (!aligned16(new_k) || !aligned16(new_v))
      return fail(CONDUIT_ERR_INVALID_ARG, "k_rows and v_rows must be 16-byte aligned");
  }
  cudaError_t err = launch_kv_copy(make_kv(kv, batch), make_batch(batch), idx, idx_off_dev, n_sel,
                                   max_budget(batch, idx_off), mode, rows_k, rows_v, new_k, new_v,
                                   static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, names[mode]);
  return CONDUIT_OK;
}

conduit_status conduit_kv_gather(const conduit_kv* kv, const conduit_batch* batch,
                                 const int32_t* idx, const int32_t* idx_off,
                                 const int32_t* idx_off_dev, void* k_rows, void* v_rows,
                                 void* stream) {
  return kv_copy(kv, batch, idx, idx_off, idx_off_dev, k_rows, v_rows, nullptr, nullptr, 0, stream);
}

conduit_status conduit_kv_scatter(const conduit_kv* kv, const conduit_batch* batch,
                                  const int32_t* idx, const int32_t* idx_off,
                                  const int32_t* idx_off_dev, const void* k_rows,
                                  const void* v_rows, void* stream) {
  return kv_copy(kv, batch, idx, idx_off, idx_off_dev, const_cast<void*>(k_rows),
                 const_cast<void*>(v_rows), nullptr, nullptr, 1, stream);
}

conduit_status conduit_kv_exchange(const conduit_kv* kv, const conduit_batch* batch,
                                   const int32_t* idx, const int32_t* idx_off,
                                   const int32_t* idx_off_dev, void* k_old, void* v_old,
                                   const void* k_rows, const void* v_rows, void* stream) {
  return kv_copy(kv, batch, idx, idx_off, idx_off_dev, k_old, v_old, k_rows, v_rows, 2, stream);
}

conduit_status conduit_refresh_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                              const int32_t* idx_off, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  (void)idx_off;
  // the tensor-core kernel takes its work items from a counter in the workspace
  *bytes = refresh_tc_supported(make_kv(kv, batch)) ? kAlign : 0;
  return CONDUIT_OK;
}

conduit_status conduit_refresh_attn(const conduit_kv* kv, const conduit_batch* batch,
                                    const int32_t* idx, const int32_t* idx_off,
                                    const int32_t* idx_off_dev, const void* q_rows, void* out,
                                    void* workspace, size_t workspace_bytes, int32_t* status,
                                    void* stream) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if ((st = check_selection(batch, idx_off, idx_off_dev, true, idx))) return st;
  const int n_sel = idx_off[batch->num_requests];
  if (n_sel == 0) return CONDUIT_OK;
  if (!q_rows || !out) return fail(CONDUIT_ERR_INVALID_ARG, "q_rows and out are required");
  const KvDev kd = make_kv(kv, batch);
  const bool tc = refresh_tc_supported(kd);
  if ((st = check_workspace(workspace, workspace_bytes, tc ? kAlign : 0))) return st;
  cudaError_t err =
      tc ? launch_refresh_tc(kd, make_batch(batch), idx, idx_off_dev, idx_off, n_sel, q_rows, out,
                             static_cast<int32_t*>(workspace), status,
                             static_cast<cudaStream_t>(stream))
         : launch_refresh_simt(kd, make_batch(batch), idx, idx_off_dev, n_sel, q_rows, out,
                               static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "refresh_attn");
  return CONDUIT_OK;
}

conduit_status conduit_staleness_iso_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                                   int32_t M, size_t* bytes) {
  conduit_status st;
  if (!bytes) return fail(CONDUIT_ERR_INVALID_ARG, "bytes is NULL");
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if (M < 1) return fail(CONDUIT_ERR_INVALID_ARG, "M must be >= 1");
  *bytes = stale_layout(make_kv(kv, batch), make_batch(batch), batch->q_off[batch->num_requests], M).total;
  return CONDUIT_OK;
}

conduit_status conduit_staleness_iso(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                                     const uint8_t* refreshed, const void* z, int32_t M, float kappa,
                                     double* err, double* err_layers, void* workspace,
                                     size_t workspace_bytes, int32_t* status, void* stream) {
  conduit_status st;
  if ((st = check_batch(batch)) || (st = check_kv(kv, batch))) return st;
  if (!q || !refreshed || !z || !err)
    return fail(CONDUIT_ERR_INVALID_ARG, "q, refreshed, z and err are required");
  if (!aligned16(q) || !aligned16(z)) return fail(CONDUIT_ERR_INVALID_ARG, "q and z must be 16-byte aligned");
  if (M < 1) return fail(CONDUIT_ERR_INVALID_ARG, "M must be >= 1");
  if (!(kappa >= 0.f) || !std::isfinite(kappa))
    return fail(CONDUIT_ERR_INVALID_ARG, "kappa must be finite and >= 0");
  const KvDev kd = make_kv(kv, batch);
  const BatchDev bd = make_batch(batch);
  const int32_t q_tot = batch->q_off[batch->num_requests];
  if ((st = check_workspace(workspace, workspace_bytes, stale_layout(kd, bd, q_tot, M).total))) return st;
  cudaError_t err_c = launch_staleness_iso(kd, bd, batch->q_off, q_tot, q, refreshed, z, M, kappa, err,
                                           err_layers, workspace, status,
                                           static_cast<cudaStream_t>(stream));
  if (err_c) return cuda_fail(err_c, "staleness_iso");
  return CONDUIT_OK;
}

conduit_status conduit_clear_status(int32_t* status, void* stream) {
  if (!status) return fail(CONDUIT_ERR_INVALID_ARG, "status is NULL");
  cudaError_t err = cudaMemsetAsync(status, 0, sizeof(int32_t), static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "clear_status");
  return CONDUIT_OK;
}

conduit_status conduit_read_status(const int32_t* status, void* stream, int32_t* word) {
  if (!status || !word) return fail(CONDUIT_ERR_INVALID_ARG, "status and word are required");
  cudaError_t err = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (err) return cuda_fail(err, "read_status (synchronize)");
  err = cudaMemcpy(word, status, sizeof(int32_t), cudaMemcpyDeviceToHost);
  if (err) return cuda_fail(err, "read_status (copy)");
  if (*word & CONDUIT_FLAG_TIMEOUT) return CONDUIT_ERR_TIMEOUT;
  if (*word & CONDUIT_FLAG_NONFINITE) return CONDUIT_ERR_NONFINITE;
  return CONDUIT_OK;
}

}  // extern "C"
