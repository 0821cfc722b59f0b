/*
 * conduit.h - C ABI of the GB300 library for Conduit's query-conditioned
 * scoring pass and budgeted selective refresh (Conduit, Sec. 3 and
 * Algorithm 1).
 *
 * Conventions shared by every entry point:
 *  - Every call returns a conduit_status. No exception crosses the ABI.
 *  - Arguments are checked on the host before anything is enqueued; a call
 *    that returns CONDUIT_ERR_INVALID_ARG, _UNSUPPORTED or _WORKSPACE has
 *    launched nothing and touched no device memory.
 *  - Pointers marked "device" are caller-owned device memory; pointers
 *    marked "host" are caller-owned host memory read during the call only.
 *    The library never allocates device memory: scratch space comes from a
 *    caller workspace whose size the matching *_workspace_size call returns.
 *  - All device work is enqueued on the caller's stream (a cudaStream_t
 *    passed as void*; NULL means the legacy default stream) and is
 *    asynchronous. No call synchronises, except conduit_read_status.
 *  - Conditions found on the device (a non-finite score, a bounded wait that
 *    ran out) are OR-ed into a caller-provided device int32 status word as
 *    CONDUIT_FLAG_* bits; conduit_read_status turns the word into a status.
 *  - conduit_last_error_string() describes the last failure of the calling
 *    thread.
 *
 * Token positions are request-local indices 0 .. N_r-1 of the request's
 * visual tokens. Image spans are contiguous, non-empty and tile each
 * request's tokens (Sec. 3.1, Eq. 1).
 */
#ifndef CONDUIT_H
#define CONDUIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define CONDUIT_VERSION 100 /* 1.0.0 */
#define CONDUIT_MAX_LAYERS 512

typedef int32_t conduit_status;
enum {
  CONDUIT_OK = 0,
  CONDUIT_ERR_INVALID_ARG = 1, /* a pointer, size, span or budget is wrong */
  CONDUIT_ERR_UNSUPPORTED = 2, /* valid, but a shape or dtype the library does not implement */
  CONDUIT_ERR_CUDA = 3,        /* a CUDA runtime call failed */
  CONDUIT_ERR_NONFINITE = 4,   /* device found a NaN / Inf score (status word) */
  CONDUIT_ERR_TIMEOUT = 5,     /* a bounded device wait ran out (status word) */
  CONDUIT_ERR_WORKSPACE = 6    /* workspace pointer missing, misaligned or short */
};

/*
 * Bits of the device status word. A bounded wait that ran out sets
 * CONDUIT_FLAG_TIMEOUT together with one site bit naming what never arrived:
 * a TMA tile (CONDUIT_SITE_LOAD), an MMA completion (CONDUIT_SITE_MMA) or an
 * item's final MMA completion (CONDUIT_SITE_FINAL).
 */
enum {
  CONDUIT_FLAG_NONFINITE = 1,
  CONDUIT_FLAG_TIMEOUT = 2,
  CONDUIT_SITE_LOAD = 1 << 8,
  CONDUIT_SITE_MMA = 1 << 9,
  CONDUIT_SITE_FINAL = 1 << 10
};

/* Element type of K, V, queries, fresh rows and refresh outputs. */
enum { CONDUIT_F32 = 0, CONDUIT_BF16 = 1 };

/*
 * The reused visual KV cache (Sec. 3.1; paged storage as in the serving
 * engine of Sec. 4.3).
 *  contiguous (page_size == 0): k, v are [L][Hkv][N_tot][d]; request r's
 *    tokens are rows tok_off[r] .. tok_off[r+1]-1.
 *  paged (page_size > 0): k, v are pools [L][P][Hkv][page_size][d];
 *    request r's token t lives in physical page
 *    page_table[r * max_pages_per_req + t / page_size] at row t % page_size.
 * k and v are 16-byte aligned device pointers of dtype `dtype`.
 */
typedef struct conduit_kv {
  int32_t num_layers;        /* L */
  int32_t num_q_heads;       /* Hq */
  int32_t num_kv_heads;      /* Hkv, Hq % Hkv == 0 (grouped-query attention) */
  int32_t head_dim;          /* d, a multiple of 8 in [8, 256] */
  int32_t dtype;             /* CONDUIT_F32 or CONDUIT_BF16 */
  int32_t page_size;         /* 0 = contiguous, else rows per page */
  int32_t num_pages;         /* P (paged only) */
  int32_t max_pages_per_req; /* row length of page_table (paged only) */
  void* k;                   /* device */
  void* v;                   /* device */
  const int32_t* page_table; /* device [R][max_pages_per_req] (paged only) */
} conduit_kv;

/*
 * A batch of requests, each with its visual-token span, its image spans
 * (Eq. 1: V_j, n_j, pi(t)) and its scoring query span Q (App. A.2: the text
 * block after the last image). Every offset array exists twice, on the host
 * (for checks and launch sizing) and on the device (for the kernels), with
 * equal contents.
 *  tok_off    [R+1]  request r owns global token rows tok_off[r] .. tok_off[r+1]-1
 *  img_off    [K+1]  image j owns global token rows img_off[j] .. img_off[j+1]-1
 *  req_img_off[R+1]  request r owns images req_img_off[r] .. req_img_off[r+1]-1
 *  q_off      [R+1]  request r owns query rows q_off[r] .. q_off[r+1]-1
 */
typedef struct conduit_batch {
  int32_t num_requests; /* R >= 1 */
  int32_t num_images;   /* K (total over requests) >= R */
  const int32_t* tok_off;         /* host */
  const int32_t* img_off;         /* host */
  const int32_t* req_img_off;     /* host */
  const int32_t* q_off;           /* host */
  const int32_t* tok_off_dev;     /* device */
  const int32_t* img_off_dev;     /* device */
  const int32_t* req_img_off_dev; /* device */
  const int32_t* q_off_dev;       /* device */
} conduit_batch;

/* Library version, CONDUIT_VERSION of the build. */
int32_t conduit_version(void);

/* Text of the calling thread's last error ("" if none). Never NULL. */
const char* conduit_last_error_string(void);

/*
 * Refresh budget k = floor(r * N_vis), Eq. 2 and Algorithm 1 (first step).
 * A guard of 1e-9 makes decimal ratios land on integers (0.3 * 10 -> 3).
 * Returns -1 if r is outside [0, 1] or NaN, or n_vis is negative.
 */
int32_t conduit_budget(double r, int64_t n_vis);

/*
 * Query-conditioned scoring pass (Sec. 3.3, Eqs. 6-8; Algorithm 1 scoring
 * loops). For every request, scored layer l and token t:
 *   alpha_{q,t,l,h} = softmax over the request's N_r visual keys of
 *                     <q_{l,h,q}, k_{l,h/G,t}> / sqrt(d)            (fp32)
 *   a_t^(l)  = sum_q sum_h alpha / (|Q| Hq)                          Eq. 6
 *   v_t^(l)  = || concat_g V_{l,g,t} ||_2                            Sec. 3.3
 *   s[t]     = (1/|L|) sum_l a_t^(l) v_t^(l)                         Eq. 7
 *   attn_sum[t] = sum_l a_t^(l)
 *   g[j]     = (1/(|L| n_j)) sum_l sum_{t in V_j} a_t^(l)            Eq. 8
 *  q         device [L][Hq][Q_tot][d], dtype of kv (post-RoPE queries)
 *  layers    host [n_layers] strictly increasing scored layer ids, or NULL
 *            for all L layers (App. A.2 default); n_layers <= CONDUIT_MAX_LAYERS
 *  s, attn_sum  device fp32 [N_tot] (attn_sum may be NULL)
 *  g         device fp32 [K]
 *  workspace device, 256-byte aligned, conduit_score_workspace_size bytes
 *  status    device int32 status word or NULL (NONFINITE if a score is NaN/Inf)
 * Results are deterministic: the same inputs give bitwise-equal outputs.
 */
conduit_status conduit_score_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                            int32_t n_layers, size_t* bytes);
conduit_status conduit_score(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                             const int32_t* layers, int32_t n_layers, float* s, float* attn_sum,
                             float* g, void* workspace, size_t workspace_bytes, int32_t* status,
                             void* stream);

/*
 * Scoring variants (conduit_score_ex). The defaults (all fields zero, or a
 * NULL options pointer) are conduit_score.
 *  statistic   CONDUIT_STAT_MEAN: s uses a_t^(l) of Eq. 6 (the deployed policy).
 *              CONDUIT_STAT_RMS: s uses the RMS attention of Eq. 4,
 *                abar_t^(l) = sqrt( sum_q sum_h alpha^2 / (|Q| Hq) ),
 *              over the same query rows and heads. attn_sum and g (Eq. 8) keep
 *              the mean of Eq. 6 in both cases.
 *  value_norm  CONDUIT_VNORM_FROM_V: v_t^(l) from V (Sec. 3.3).
 *              CONDUIT_VNORM_SIDE_CACHE: v_t^(l) = vnorm[l][t], the side cache
 *                of conduit_value_norms (V is not read).
 *              CONDUIT_VNORM_NONE: v_t^(l) = 1, the score is attention alone
 *                (the factor ablation that drops the value norm, Sec. 4.4).
 *  vnorm       device fp32 [L][tok_off[R]]; required with SIDE_CACHE, else NULL.
 *  extra_lse   device fp32 [L][Hq][Q_tot] (layout of q without d), or NULL.
 *              When given, alpha_{q,t} is normalised over the whole context
 *              rather than the visual keys alone: extra_lse[l][h][q] is the
 *              natural-log log-sum-exp of <q_{l,h,q}, k_j> / sqrt(d) over the
 *              keys j outside the request's visual span (text, query span),
 *              -inf where there are none, as a flash-attention pass over those
 *              keys returns it. The softmax denominator of row (l, h, q)
 *              becomes sum_{t visual} exp(x_t) + exp(extra_lse), so the alphas
 *              of a row sum to less than 1.
 */
enum { CONDUIT_STAT_MEAN = 0, CONDUIT_STAT_RMS = 1 };
enum { CONDUIT_VNORM_FROM_V = 0, CONDUIT_VNORM_SIDE_CACHE = 1, CONDUIT_VNORM_NONE = 2 };

typedef struct conduit_score_opts {
  int32_t statistic;     /* CONDUIT_STAT_* */
  int32_t value_norm;    /* CONDUIT_VNORM_* */
  const float* vnorm;    /* side cache (value_norm == CONDUIT_VNORM_SIDE_CACHE) or NULL */
  const float* extra_lse; /* full-context softmax denominators or NULL */
} conduit_score_opts;

/*
 * conduit_score with the variants of `opts` (NULL: the defaults). Arguments,
 * results and errors are otherwise those of conduit_score; INVALID_ARG also
 * for an unknown statistic or value_norm, a vnorm that does not match
 * value_norm, or a misaligned extra_lse. The workspace depends on opts (RMS
 * adds one partial-sum array, any value_norm but FROM_V drops one).
 */
conduit_status conduit_score_ex_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                               int32_t n_layers, const conduit_score_opts* opts,
                                               size_t* bytes);
conduit_status conduit_score_ex(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                                const int32_t* layers, int32_t n_layers,
                                const conduit_score_opts* opts, float* s, float* attn_sum,
                                float* g, void* workspace, size_t workspace_bytes,
                                int32_t* status, void* stream);

/*
 * Value-norm side cache (Sec. 4.3 and App. C.2: v_t^(l) depends only on the
 * cached content, so one scalar per token and layer stored when the cache is
 * built keeps the scores exact and takes the value rows off the scoring
 * pass).
 *   vnorm[l][t] = || concat_g V_{l,g,t} ||_2   for every layer l < L and
 *                 global token row t < tok_off[R]
 * The norm is computed with the operations, in the order, that conduit_score
 * uses for this cache, so conduit_score_with_norms over this side cache
 * returns bitwise the s, attn_sum and g of conduit_score.
 *  vnorm  device fp32 [L][tok_off[R]], 4-byte aligned (written); caller-owned
 * Errors: INVALID_ARG for a NULL or misaligned vnorm, UNSUPPORTED for more
 * than 65535 layers, otherwise as for conduit_score.
 */
conduit_status conduit_value_norms(const conduit_kv* kv, const conduit_batch* batch, float* vnorm,
                                   void* stream);

/*
 * Keep the side cache exact after conduit_kv_scatter or conduit_kv_exchange
 * rewrote rows: recompute vnorm[l][tok_off[r] + idx_i] for every layer l and
 * every selected row i (idx, idx_off, idx_off_dev as for conduit_kv_scatter).
 * The other entries are left as they are.
 */
conduit_status conduit_value_norms_update(const conduit_kv* kv, const conduit_batch* batch,
                                          const int32_t* idx, const int32_t* idx_off,
                                          const int32_t* idx_off_dev, float* vnorm, void* stream);

/*
 * conduit_score with v_t^(l) read from the side cache at vnorm[l][t] (l the
 * scored layer id) instead of from V: the scoring pass reads K, Q and 4 bytes
 * per token and layer. All other arguments, results and errors are those of
 * conduit_score; the workspace is smaller (no value partial sums). Same as
 * conduit_score_ex with value_norm = CONDUIT_VNORM_SIDE_CACHE.
 *  vnorm  device fp32 [L][tok_off[R]] from conduit_value_norms (read)
 */
conduit_status conduit_score_with_norms_workspace_size(const conduit_kv* kv,
                                                       const conduit_batch* batch,
                                                       int32_t n_layers, size_t* bytes);
conduit_status conduit_score_with_norms(const conduit_kv* kv, const conduit_batch* batch,
                                        const void* q, const int32_t* layers, int32_t n_layers,
                                        const float* vnorm, float* s, float* attn_sum, float* g,
                                        void* workspace, size_t workspace_bytes, int32_t* status,
                                        void* stream);

/*
 * Image-level amplification and one global top-k per request (Sec. 3.4-3.5,
 * Eqs. 9-11; Algorithm 1 last loops).
 *   c_j    = (1 - lambda) + lambda g_j / g_bar, g_bar = mean of the request's g_j;
 *            exactly 1 when the request has one image (Sec. 3.5) or g_bar == 0;
 *            binary32, one rounding per operation, g_bar = (((g_0 + g_1) + ...) / K
 *   s_hat_t = s_t c_{pi(t)}                                          Eq. 10
 *   T_r    = TopK_t(s_hat, k_r), ties to the lowest index            Eq. 11
 *  s, g       device fp32 [N_tot], [K] (outputs of conduit_score)
 *  lambda     in [0, 1]
 *  idx_off    host [R+1], idx_off_dev device [R+1]: prefix sums of the
 *             budgets, k_r = idx_off[r+1] - idx_off[r], 0 <= k_r <= N_r
 *  idx        device int32 [idx_off[R]]: request r's selected request-local
 *             token indices at idx[idx_off[r] ..], ascending
 *  mask       device uint8 [N_tot] refresh mask (1 = recompute) or NULL
 *  s_hat      device fp32 [N_tot] or NULL;  coeff device fp32 [K] c_j or NULL
 *  status     NONFINITE if an s_hat is NaN / Inf
 */
conduit_status conduit_select_workspace_size(const conduit_batch* batch, size_t* bytes);
conduit_status conduit_select_topk(const conduit_batch* batch, const float* s, const float* g,
                                   float lambda, const int32_t* idx_off, const int32_t* idx_off_dev,
                                   int32_t* idx, uint8_t* mask, float* s_hat, float* coeff,
                                   void* workspace, size_t workspace_bytes, int32_t* status,
                                   void* stream);

/*
 * Scoring and the global selection in one call (Sec. 3.3-3.5, Eqs. 6-11;
 * Algorithm 1 from the scoring loops to the top-k): the results of
 * conduit_score_ex(kv, batch, q, layers, n_layers, opts, s, attn_sum, g, ...)
 * followed by conduit_select_topk(batch, s, g, lambda, idx_off, idx_off_dev,
 * idx, mask, s_hat, coeff, ...), bit for bit, with fewer launches: when every
 * request holds at most 8192 tokens and the batch at most 32 tokens per SM of
 * the device (4 864 on a 152-SM GPU), the per-token reductions (s_t, A_t),
 * the image means g_j, c_j, s_hat and the top-k run as one launch after the
 * scoring kernel (the last block to finish a request's tokens selects that
 * request); other batches take the separate launches of the two calls.
 * Arguments, layouts and ownership are those of the two calls (opts may be
 * NULL: the defaults; attn_sum may be NULL).
 *  workspace  device, 256-byte aligned,
 *             conduit_score_select_topk_workspace_size bytes
 * Errors: the union of the two calls' (INVALID_ARG, UNSUPPORTED, WORKSPACE,
 * CUDA); nothing is enqueued when the arguments are rejected. status: the
 * bits either call sets (NONFINITE; TIMEOUT from the scoring kernel).
 */
conduit_status conduit_score_select_topk_workspace_size(const conduit_kv* kv,
                                                        const conduit_batch* batch,
                                                        int32_t n_layers,
                                                        const conduit_score_opts* opts,
                                                        size_t* bytes);
conduit_status conduit_score_select_topk(const conduit_kv* kv, const conduit_batch* batch,
                                         const void* q, const int32_t* layers, int32_t n_layers,
                                         const conduit_score_opts* opts, float lambda,
                                         const int32_t* idx_off, const int32_t* idx_off_dev,
                                         float* s, float* attn_sum, float* g, int32_t* idx,
                                         uint8_t* mask, float* s_hat, float* coeff,
                                         void* workspace, size_t workspace_bytes, int32_t* status,
                                         void* stream);

/*
 * Explicit per-image quotas instead of the global ranking (App. D.3: the
 * "explicit" variant of the cross-image diagnostic, compared there with the
 * deployed global rule). Per request, with c_j of conduit_select_topk:
 *   k_j proportional to c_j n_j, sum_j k_j = k_r, 0 <= k_j <= n_j
 * by the largest remainder: w_j = c_j n_j (float64), W summed left to right
 * over the open images, ideal_j = (kk w_j) / W; an image whose ideal exceeds
 * n_j is closed at n_j and the rest kk of the budget is shared again over
 * the others; otherwise k_j = floor(ideal_j) plus one unit for the
 * k_r - sum floor largest remainders, ties to the lower image index. If every
 * open weight is 0 (lambda = 1 and g_j = 0), the weights become n_j.
 * Then T_r = union over j of the k_j tokens of image j with the largest s_t
 * (c_j is constant inside an image), ties to the lowest index.
 * Arguments as for conduit_select_topk, plus
 *  quota  device int32 [K] k_j, or NULL
 * idx holds request r's indices ascending (image by image); s_hat = s c_pi(t)
 * is written for reference. status: NONFINITE for a NaN / Inf or negative s,
 * or a non-finite c_j (that request's budget is then shared by image size).
 */
conduit_status conduit_select_quota_workspace_size(const conduit_batch* batch, size_t* bytes);
conduit_status conduit_select_quota(const conduit_batch* batch, const float* s, const float* g,
                                    float lambda, const int32_t* idx_off,
                                    const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                    float* s_hat, float* coeff, int32_t* quota, void* workspace,
                                    size_t workspace_bytes, int32_t* status, void* stream);

/*
 * conduit_select_topk without a caller workspace. The paper has no
 * counterpart: this is a convenience of this library for callers that cannot
 * hand it device scratch memory, for instance a serving engine that has
 * given all free device memory to its paged KV pool and keeps no allocator
 * handle on this path, or plain C code with no device allocator at all.
 * Arguments and results are those of conduit_select_topk, minus workspace.
 *  - Scratch comes from one static device array of the library, sized for
 *    CONDUIT_NOALLOC_MAX_TOKENS tokens (4 MiB), which every GPU that loads
 *    the library keeps until the process exits. A batch with more tokens
 *    (tok_off[R]) is rejected with CONDUIT_ERR_UNSUPPORTED.
 *  - The first call on a device looks up the array's device address with
 *    that device current; make that first call before any stream capture.
 *    The CUDA runtime may load the library's device code onto a device only
 *    at that lookup (or at the library's first launch there), so that first
 *    use needs about 4 MiB of free device memory; a caller that hands all
 *    free memory to its KV pool should make one call (or any other library
 *    call) first. If the lookup fails, for lack of memory or otherwise, the
 *    call returns CONDUIT_ERR_CUDA with the runtime's message.
 *  - The call allocates nothing: no cudaMalloc, cudaFree or other
 *    allocating routine.
 *  - All calls share the array and it keeps the last call's contents. Each
 *    call rewrites the part it reads, but calls whose work overlaps on the
 *    GPU (other streams, other host threads) race on it: order them.
 */
#define CONDUIT_NOALLOC_MAX_TOKENS (1 << 20)
conduit_status conduit_select_topk_noalloc(const conduit_batch* batch, const float* s,
                                           const float* g, float lambda, const int32_t* idx_off,
                                           const int32_t* idx_off_dev, int32_t* idx,
                                           uint8_t* mask, float* s_hat, float* coeff,
                                           int32_t* status, void* stream);

/*
 * Gather of the selected rows of every layer (selective recompute, Sec. 3.1
 * and 3.5): k_rows[l][i][g][:] = K[l][g][idx_i][:] (same for V), where i runs
 * over all requests' selections in idx order.
 *  k_rows, v_rows  device [L][idx_off[R]][Hkv][d], dtype of kv
 */
conduit_status conduit_kv_gather(const conduit_kv* kv, const conduit_batch* batch,
                                 const int32_t* idx, const int32_t* idx_off,
                                 const int32_t* idx_off_dev, void* k_rows, void* v_rows,
                                 void* stream);

/*
 * Scatter of recomputed K/V rows into the cache, all layers in one launch
 * (Sec. 3.5: selected entries are recomputed, the rest are reused):
 * K[l][g][idx_i][:] = k_rows[l][i][g][:] (same for V). In place in kv->k, kv->v.
 *  k_rows, v_rows  device [L][idx_off[R]][Hkv][d], dtype of kv
 */
conduit_status conduit_kv_scatter(const conduit_kv* kv, const conduit_batch* batch,
                                  const int32_t* idx, const int32_t* idx_off,
                                  const int32_t* idx_off_dev, const void* k_rows,
                                  const void* v_rows, void* stream);

/*
 * Gather and scatter in one launch (Sec. 3.5: the stale entries of the
 * selected tokens are read out and replaced by their recomputed K/V): for
 * every layer l, selected row i and KV head g,
 *   k_old[l][i][g][:] = K[l][g][idx_i][:], then K[l][g][idx_i][:] = k_rows[l][i][g][:]
 * (same for V). Equal to conduit_kv_gather followed by conduit_kv_scatter;
 * the indices of a request must be distinct (conduit_select_topk's are),
 * and k_old / v_old must not overlap k_rows / v_rows or the cache.
 *  k_old, v_old    device [L][idx_off[R]][Hkv][d], dtype of kv (written)
 *  k_rows, v_rows  device [L][idx_off[R]][Hkv][d], dtype of kv (read)
 * Buffers are 16-byte aligned; errors as for conduit_kv_gather.
 */
conduit_status conduit_kv_exchange(const conduit_kv* kv, const conduit_batch* batch,
                                   const int32_t* idx, const int32_t* idx_off,
                                   const int32_t* idx_off_dev, void* k_old, void* v_old,
                                   const void* k_rows, const void* v_rows, void* stream);

/*
 * Causal attention of the refreshed rows over the patched cache (Sec. 3.1
 * and 4.3, selective recompute): for every layer l, selected row i at
 * position p_i = idx_i and query head h,
 *   out[l][i][h] = sum_{j <= p_i} softmax_j(<q_rows[l][i][h], K'[l][h/G][j]> / sqrt(d)) V'[l][h/G][j]
 * where K', V' are the cache after conduit_kv_scatter (call it first).
 * Softmax and accumulation in fp32; out is written in the cache dtype.
 *  q_rows, out  device [L][idx_off[R]][Hq][d], dtype of kv
 *  idx must be ascending within each request (conduit_select_topk's order).
 *  workspace    device, 256-byte aligned, conduit_refresh_workspace_size
 *               bytes (256 for bf16 caches with head_dim 128: the work
 *               counter of the persistent kernel; 0 otherwise); calls that
 *               overlap on the GPU need workspaces of their own.
 */
conduit_status conduit_refresh_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                              const int32_t* idx_off, size_t* bytes);
conduit_status conduit_refresh_attn(const conduit_kv* kv, const conduit_batch* batch,
                                    const int32_t* idx, const int32_t* idx_off,
                                    const int32_t* idx_off_dev, const void* q_rows, void* out,
                                    void* workspace, size_t workspace_bytes, int32_t* status,
                                    void* stream);

/*
 * Isotropic Monte Carlo staleness estimator (App. D): the residual error a
 * refresh set T leaves under sampled stale value displacements, per request
 *   E_r = sum_{l, h, q in Q_r} (1/M) sum_m || sum_{t not in T} alpha_{q,t} xi_t^(m) ||^2
 *   xi_{l,g,t}^(m) = kappa ||V_{l,g,t}|| / sqrt(d) z_{l,g,t}^(m)
 * with alpha the cached-key softmax over the request's N_r visual keys (Eq. 6's
 * alpha), query head h reading KV head h / G, ||V_{l,g,t}|| that head's value
 * norm and z standard normal draws. Comparing E for the sets of different
 * selection rules (and a uniform random set) under the same z is the
 * cross-image diagnostic of App. D.3.
 *  q          device [L][Hq][Q_tot][d], dtype of kv (the scoring queries)
 *  refreshed  device uint8 [N_tot], 1 = token in T (e.g. conduit_select_topk's mask)
 *  z          device [M][L][Hkv][N_tot][d], dtype of kv (the random draws; the
 *             caller generates them)
 *  M >= 1, kappa >= 0
 *  err        device double [R] E_r (written)
 *  err_layers device double [R][L] the per-layer terms of E_r, or NULL
 *  workspace  conduit_staleness_iso_workspace_size bytes (it holds one draw of
 *             xi in the cache's layout and the per-draw attention outputs)
 * Attention runs with the refresh kernels (bf16 P and outputs for bf16
 * caches); the reduction of ||O||^2 is in a fixed order.
 */
conduit_status conduit_staleness_iso_workspace_size(const conduit_kv* kv, const conduit_batch* batch,
                                                   int32_t M, size_t* bytes);
conduit_status conduit_staleness_iso(const conduit_kv* kv, const conduit_batch* batch, const void* q,
                                     const uint8_t* refreshed, const void* z, int32_t M, float kappa,
                                     double* err, double* err_layers, void* workspace,
                                     size_t workspace_bytes, int32_t* status, void* stream);

/*
 * Number of kernels this library has enqueued in this process (launched, or
 * recorded into a stream capture) since it was loaded. Diagnostic only.
 */
int64_t conduit_launch_count(void);

/* Zero the device status word (enqueued on stream). */
conduit_status conduit_clear_status(int32_t* status, void* stream);

/*
 * Synchronise `stream`, copy the status word to *word (host) and return
 * CONDUIT_OK, CONDUIT_ERR_NONFINITE or CONDUIT_ERR_TIMEOUT (timeout wins).
 */
conduit_status conduit_read_status(const int32_t* status, void* stream, int32_t* word);

#ifdef __cplusplus
}
#endif

#endif /* CONDUIT_H */
