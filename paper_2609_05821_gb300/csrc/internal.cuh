// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "conduit.h"

namespace conduit {

constexpr int kMaxImagesPerRequest = 4096;  // selection keeps c_j of one request in shared memory

// Scored layer ids, passed to kernels by value.
struct LayerList {
  int32_t n;
  int32_t ids[CONDUIT_MAX_LAYERS];
};

// Device view of the batch offsets.
struct BatchDev {
  int32_t R;
  int32_t K;
  const int32_t* tok_off;
  const int32_t* img_off;
  const int32_t* req_img_off;
  const int32_t* q_off;
};

// Device view of the KV cache with its addressing rule (contiguous or paged).
struct KvDev {
  void* k;
  void* v;
  int32_t L, Hq, Hkv, d, G;
  int32_t dtype;
  int32_t page_size, num_pages, max_pages;
  const int32_t* page_table;
  int64_t n_tot;  // rows per (layer, head) of a contiguous cache

  // Element offset of row (layer l, KV head g) of request r's token t
  // (request-local t, global row tg = tok_off[r] + t).
  __device__ __forceinline__ int64_t row(int l, int g, int r, int64_t tg, int t) const {
    if (page_size == 0) return ((int64_t(l) * Hkv + g) * n_tot + tg) * d;
    const int page = page_table[int64_t(r) * max_pages + t / page_size];
    return (((int64_t(l) * num_pages + page) * Hkv + g) * page_size + (t % page_size)) * int64_t(d);
  }
};

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T>
__device__ __forceinline__ T from_float(float x);
template <>
__device__ __forceinline__ float from_float<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ void flag_status(int32_t* status, int32_t bits) {
  if (status) atomicOr(status, bits);
}

// Index of the request owning global token row tg (binary search over tok_off).
__device__ __forceinline__ int request_of(const int32_t* tok_off, int R, int64_t tg) {
  int lo = 0, hi = R - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tok_off[mid] <= tg) lo = mid; else hi = mid - 1;
  }
  return lo;
}

constexpr float kLog2e = 1.4426950408889634f;

// log2(2^x + 2^y); x or y may be -inf (then the other is returned unchanged).
// Joins the visual keys' log-sum-exp of a scoring row with that of the keys
// outside the visual span (full-context softmax).
__device__ __forceinline__ float log2_add(float x, float y) {
  const float hi = fmaxf(x, y), lo = fminf(x, y);
  if (lo == -INFINITY) return hi;
  return hi + log2f(1.f + exp2f(lo - hi));
}

// ----------------------------------------------------- value sums of squares
// The value norm v_t^(l) is sqrt of a sum of per-head partial sums of squares.
// The scoring kernels and the norm side cache (conduit_value_norms) both build
// these partials with the helpers below, so the side cache holds bitwise the
// norm the scoring pass would compute from V itself.

// One 16-byte chunk (8 bf16) of a 64-element half row into four running sums
// (one per bf16 pair of the chunk); eight chunks make a half row.
__device__ __forceinline__ void sumsq_bf16_chunk(const uint4& x, float (&sq)[4]) {
  const __nv_bfloat162* hv = reinterpret_cast<const __nv_bfloat162*>(&x);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 f = __bfloat1622float2(hv[e]);
    sq[e] = fmaf(f.x, f.x, fmaf(f.y, f.y, sq[e]));
  }
}
__device__ __forceinline__ float sumsq_combine(const float (&sq)[4]) {
  return (sq[0] + sq[1]) + (sq[2] + sq[3]);
}

// Sum of squares of one head row of d elements by a whole warp: lane c takes
// 16-byte chunks c, c+32, ..., then a butterfly reduction (every lane ends
// with the same value).
template <typename T>
__device__ __forceinline__ float warp_row_sumsq(const T* row, int d, int lane) {
  constexpr int VEC = 16 / sizeof(T);
  const int cpr = d / VEC;
  float acc = 0.f;
  for (int c = lane; c < cpr; c += 32) {
    const uint4 raw = *reinterpret_cast<const uint4*>(row + c * VEC);
    const T* vals = reinterpret_cast<const T*>(&raw);
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
      const float x = to_float(vals[u]);
      acc = fmaf(x, x, acc);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

// Host-side count of kernels enqueued by this library (conduit_launch_count).
void count_launches(int n);

// ------------------------------------------------------------------ launchers
// Each returns a cudaError_t from the launch (cudaGetLastError) and enqueues
// on `stream`.
cudaError_t launch_value_sumsq(const KvDev& kv, const BatchDev& b, const LayerList& layers,
                               int max_tokens, float* ss, cudaStream_t stream);
// pa2 (sums of alpha^2, RMS statistic) and extra_lse ([L][Hq][q_tot] natural-log
// log-sum-exp of each scoring row over keys outside the visual span) may be NULL.
cudaError_t launch_score_simt(const KvDev& kv, const BatchDev& b, const void* q, int32_t q_tot,
                              const LayerList& layers, int max_rows, int max_tokens,
                              float2* stats, float* pa, float* pa2, const float* extra_lse,
                              cudaStream_t stream);
// Tensor-core scoring (bf16, head_dim 128): one kernel, row statistics then
// column sums per (slab, group of at most 256 scoring rows); it writes two
// partials per row group into pa and two half-row partials into ss (ss NULL:
// V is not read, the norms come from the side cache).
constexpr int kScoreGroupRows = 256;
bool score_tc_supported(const KvDev& kv);
int score_tc_groups(int rows);
cudaError_t launch_score_tc(const KvDev& kv, const BatchDev& b, const int32_t* q_off_host,
                            const void* q, int32_t q_tot, const LayerList& layers, int rg_max,
                            float* pa, float* ss, float* pa2, const float* extra_lse,
                            int32_t* status, cudaStream_t stream);
// pa is [n_layers][Hkv][rg_max][parts][n_tot] and ss [n_layers][Hkv][parts][n_tot]
// (partial sums of squares of V per KV head); request r contributes
// ceil(G n_q_r / group_rows) row groups (one when group_rows == 0).
// Value norms: vmode 0 from ss, 1 from the side cache vnorm [L][n_tot] (read
// at layers.ids[li]), 2 none (v = 1, attention alone). pa2 (same layout as pa,
// sums of alpha^2) switches the statistic in s to the RMS of Eq. 4; attn_sum
// and g always take the mean of Eq. 6.
cudaError_t launch_finalize(const float* pa, const float* pa2, const float* ss, const float* vnorm,
                            int vmode, const LayerList& layers, const BatchDev& b, int n_layers, int Hkv,
                            int Hq, int rg_max, int group_rows, int parts, int64_t n_tot, float* s,
                            float* attn_sum, float* g, int32_t* status, cudaStream_t stream);
// Value-norm side cache: vnorm[l][tg] for every layer and for rows i < n_rows,
// row i being global token i (idx == NULL) or request r's selected token
// idx[i] (idx_off_dev: device prefix sums of the budgets).
cudaError_t launch_value_norms(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                               const int32_t* idx_off_dev, int64_t n_rows, float* vnorm,
                               cudaStream_t stream);
// Isotropic Monte Carlo staleness estimator (App. D): workspace carving and
// the launcher (M draws of refresh attention over (K, xi^(m)), then ||O||^2).
struct StaleLayout {
  size_t xi, rows, out, pos, part, scale, counter, total;
  size_t xi_bytes;
};
StaleLayout stale_layout(const KvDev& kv, const BatchDev& b, int32_t q_tot, int M);
cudaError_t launch_staleness_iso(const KvDev& kv, const BatchDev& b, const int32_t* q_off_host,
                                 int32_t q_tot, const void* q, const uint8_t* refreshed,
                                 const void* z, int M, float kappa, double* err, double* err_rl,
                                 void* workspace, int32_t* status, cudaStream_t stream);
// max_tokens: the largest request (picks how many keys a thread keeps in
// registers). Requests of more than 8 x 1024 tokens take one cluster of CTAs
// each (keys in registers) when cluster_ok, else one CTA with its keys in
// `keys`.
cudaError_t launch_select(const BatchDev& b, int max_tokens, const float* s, const float* g,
                          float lambda, const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                          float* s_hat, float* coeff, uint32_t* keys, int32_t* status,
                          cudaStream_t stream, bool cluster_ok = true);
// The scoring tail and the global selection in one launch
// (conduit_score_select_topk): launch_finalize's reductions followed by
// launch_select's top-k, for batches whose largest request has at most
// 8 x 1024 tokens and whose 32-token blocks fit one wave of the current
// device's SMs (finalize_select_supported). arrivals: one int per request,
// zero when the kernel starts.
bool finalize_select_supported(int max_tokens, int64_t n_tot);
cudaError_t launch_finalize_select(const float* pa, const float* pa2, const float* ss, const float* vnorm,
                                   int vmode, const LayerList& layers, const BatchDev& b, int n_layers,
                                   int Hkv, int Hq, int rg_max, int group_rows, int parts, int64_t n_tot,
                                   int max_tokens, float* s, float* attn_sum, float* g, float lambda,
                                   const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask, float* s_hat,
                                   float* coeff, int32_t* arrivals, int32_t* status, cudaStream_t stream);
// Explicit per-image quotas (App. D.3): quota_kernel per request, then one
// selection CTA per image. scratch holds quota_scratch_bytes(K) bytes.
size_t quota_scratch_bytes(int total_images);
cudaError_t launch_select_quota(const BatchDev& b, int max_images, int max_image_tokens,
                                const float* s, const float* g, float lambda,
                                const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                float* s_hat, float* coeff, int32_t* quota, uint32_t* keys,
                                void* scratch, int32_t* status, cudaStream_t stream);
// Same selection with the keys in the library's static device array.
int64_t select_noalloc_max_tokens();
cudaError_t launch_select_noalloc(const BatchDev& b, int max_tokens, const float* s, const float* g,
                                  float lambda,
                                  const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                  float* s_hat, float* coeff, int32_t* status,
                                  cudaStream_t stream);
// mode 0: rows <- cache (gather); 1: cache <- rows (scatter); 2: rows <- cache,
// then cache <- new (exchange).
cudaError_t launch_kv_copy(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                           const int32_t* idx_off_dev, int32_t n_sel, int max_sel, int mode,
                           void* k_rows, void* v_rows, const void* k_new, const void* v_new,
                           cudaStream_t stream);
bool refresh_tc_supported(const KvDev& kv);
cudaError_t launch_refresh_tc(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                              const int32_t* idx_off_dev, const int32_t* idx_off_host, int32_t n_sel,
                              const void* q_rows, void* out, int32_t* work_counter, int32_t* status,
                              cudaStream_t stream);
cudaError_t launch_refresh_simt(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                                const int32_t* idx_off_dev, int32_t n_sel, const void* q_rows,
                                void* out, cudaStream_t stream);

}  // namespace conduit
