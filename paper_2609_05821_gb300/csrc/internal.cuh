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

// Host-side count of kernels enqueued by this library (conduit_launch_count).
void count_launches(int n);

// ------------------------------------------------------------------ launchers
// Each returns a cudaError_t from the launch (cudaGetLastError) and enqueues
// on `stream`.
cudaError_t launch_value_sumsq(const KvDev& kv, const BatchDev& b, const LayerList& layers,
                               int max_tokens, float* ss, cudaStream_t stream);
cudaError_t launch_score_simt(const KvDev& kv, const BatchDev& b, const void* q, int32_t q_tot,
                              const LayerList& layers, int max_rows, int max_tokens,
                              float2* stats, float* pa, cudaStream_t stream);
// Tensor-core scoring (bf16, head_dim 128): one kernel, row statistics then
// column sums per (slab, group of at most 256 scoring rows); it writes two
// partials per row group into pa and two half-row partials into ss.
constexpr int kScoreGroupRows = 256;
bool score_tc_supported(const KvDev& kv);
int score_tc_groups(int rows);
cudaError_t launch_score_tc(const KvDev& kv, const BatchDev& b, const int32_t* q_off_host,
                            const void* q, int32_t q_tot, const LayerList& layers, int rg_max,
                            float* pa, float* ss, int32_t* status, cudaStream_t stream);
// pa is [n_layers][Hkv][rg_max][parts][n_tot] and ss [n_layers][Hkv][parts][n_tot]
// (partial sums of squares of V per KV head); request r contributes
// ceil(G n_q_r / group_rows) row groups (one when group_rows == 0).
cudaError_t launch_finalize(const float* pa, const float* ss, const BatchDev& b, int n_layers,
                            int Hkv, int Hq, int rg_max, int group_rows, int parts, int64_t n_tot, float* s,
                            float* attn_sum, float* g, int32_t* status, cudaStream_t stream);
// max_tokens: the largest request (picks how many keys a thread keeps in registers).
cudaError_t launch_select(const BatchDev& b, int max_tokens, const float* s, const float* g,
                          float lambda, const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                          float* s_hat, float* coeff, uint32_t* keys, int32_t* status,
                          cudaStream_t stream);
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
                              const void* q_rows, void* out, int32_t* status, cudaStream_t stream);
cudaError_t launch_refresh_simt(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                                const int32_t* idx_off_dev, int32_t n_sel, const void* q_rows,
                                void* out, cudaStream_t stream);

}  // namespace conduit
