// Image-level amplification and exact global top-k (Conduit Eqs. 9-11).
//
// One CTA per request:
//   c_j = (1 - lambda) + lambda g_j / g_bar  (c = 1 for one image or g_bar = 0)
//   s_hat_t = s_t c_{pi(t)}
//   radix select over the float bit patterns (s_hat >= 0, so unsigned order
//   equals value order; -0 is canonicalised to +0) finds the k-th largest
//   key exactly; every key above it is taken, and keys equal to it are taken
//   in ascending token order until k are chosen (ties to the lowest index).
//   Selected indices are written in ascending order together with the mask.
//
// Explicit per-image quotas (App. D.3, the variant the paper compares with the
// global rule): quota_kernel (one CTA per request) turns the same c_j into
// quotas k_j proportional to c_j n_j (largest remainder, float64), and the
// selection kernel runs one CTA per image with budget k_j over the keys s_t,
// writing its indices after those of the request's earlier images.
#include <mutex>

#include "internal.cuh"
#include "token_reduce.cuh"

namespace conduit {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kQuotaThreads = 256;

// Eq. 9 with one rounding per operation (no contraction), so that the
// coefficient that decides integer quotas is reproducible:
//   g_bar = (((g_0 + g_1) + g_2) + ...) / K,  c_j = (1 - lambda) + lambda (g_j / g_bar).
__device__ __forceinline__ float image_mean_f32(const float* g, int K) {
  float sum = 0.f;
  for (int j = 0; j < K; ++j) sum = __fadd_rn(sum, __ldcg(g + j));
  return __fdiv_rn(sum, float(K));
}
__device__ __forceinline__ float image_coefficient(float gj, float gbar, float lambda, int K) {
  if (K == 1 || gbar == 0.f) return 1.f;
  return __fadd_rn(__fsub_rn(1.f, lambda), __fmul_rn(lambda, __fdiv_rn(gj, gbar)));
}

// Block-wide exclusive scan of one int per thread; returns the prefix and
// stores the block total in *total.
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_s, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_s[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < (kSelThreads >> 5) ? warp_s[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < (kSelThreads >> 5)) warp_s[lane] = w;  // inclusive warp prefixes
  }
  __syncthreads();
  const int before = (warp > 0 ? warp_s[warp - 1] : 0) + x - v;
  if (total) *total = warp_s[(kSelThreads >> 5) - 1];
  __syncthreads();
  return before;
}

// Segment selection by one CTA of kSelThreads threads. kQuota = false:
// segment = request `seg`, keys s_hat = s c_pi(t), budget k_r (Eqs. 10-11).
// kQuota = true: segment = image `seg`, keys s_t, budget quota[j], output at
// the request's slice + qoff[j] (App. D.3). s and g are read through L2, so
// the fused scoring tail can select a request whose scores other blocks of
// the same launch wrote.
template <int kRegKeys, bool kQuota>  // keys a thread keeps in registers (0: keys in the workspace)
__device__ __forceinline__ void select_segment(int seg, const BatchDev& b, const float* s,
                                               const float* g, float lambda, const int32_t* idx_off,
                                               int32_t* idx, uint8_t* mask, float* s_hat,
                                               float* coeff, uint32_t* keys, int32_t* status,
                                               const float* seg_coeff, const int32_t* seg_quota,
                                               const int32_t* seg_qoff, const float* mean_attn = nullptr,
                                               float* mean_g = nullptr, int mean_layers = 0) {
  __shared__ float c_s[kMaxImagesPerRequest];
  __shared__ int img_s[kMaxImagesPerRequest + 1];
  __shared__ unsigned hist[256];
  __shared__ float mean_s[kMeanThreads / 32];
  __shared__ int warp_s[32];
  __shared__ uint32_t prefix_s;
  __shared__ int remaining_s;
  __shared__ float gbar_s;

  int t0, N, k, K, base_t;
  int32_t* out;
  float c_seg = 1.f;
  if (kQuota) {  // segment = image seg
    const int j = seg;
    const int r = request_of(b.req_img_off, b.R, j);
    t0 = b.img_off[j];
    N = b.img_off[j + 1] - t0;
    k = min(max(seg_quota[j], 0), N);  // quota_kernel keeps 0 <= k_j <= n_j
    K = 1;
    base_t = t0 - b.tok_off[r];  // request-local index of the image's first token
    out = idx + idx_off[r] + seg_qoff[j];
    c_seg = seg_coeff[j];
  } else {       // segment = request seg
    const int r = seg;
    t0 = b.tok_off[r];
    N = b.tok_off[r + 1] - t0;
    K = b.req_img_off[r + 1] - b.req_img_off[r];
    k = idx_off[r + 1] - idx_off[r];
    base_t = 0;
    out = idx + idx_off[r];
  }

  // s_hat (Eq. 10) and its sortable key (s itself in quota mode, where c_j is
  // constant over the segment and decides only the quota). Each thread owns the contiguous
  // tokens [lo, hi); up to kRegKeys of them stay in registers for the radix
  // passes (requests of up to 1024 x kRegKeys tokens), otherwise the keys go
  // through the workspace. The scores held in registers are loaded before
  // c_j is formed, so the two loads overlap.
  const int per = (N + kSelThreads - 1) / kSelThreads;
  const int lo = min(N, int(threadIdx.x) * per), hi = min(N, lo + per);
  const bool in_regs = kRegKeys > 0 && per <= kRegKeys;
  float sv[kRegKeys > 0 ? kRegKeys : 1];
  if (in_regs) {
#pragma unroll
    for (int j = 0; j < kRegKeys; ++j) sv[j] = lo + j < hi ? __ldcg(s + t0 + lo + j) : 0.f;
  }
  if (!kQuota && K == 1) {  // one image: c = 1 exactly (Sec. 3.5), the span is the request
    // With mean_attn, g of the image (Eq. 8) is formed here too, in the order
    // of image_mean_group, its loads in flight with the scores' above.
    float macc = 0.f;
    if (mean_attn && threadIdx.x < kMeanThreads) {
      for (int t = int(threadIdx.x); t < N; t += kMeanThreads) macc += __ldcg(mean_attn + t0 + t);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) macc += __shfl_xor_sync(0xffffffffu, macc, o);
      if ((threadIdx.x & 31) == 0) mean_s[threadIdx.x >> 5] = macc;
    }
    if (threadIdx.x == 0) {
      img_s[0] = 0;
      img_s[1] = N;
      c_s[0] = 1.f;
      if (coeff) coeff[b.req_img_off[seg]] = 1.f;
    }
    __syncthreads();
    if (mean_attn && threadIdx.x == 0) {
      float tot = 0.f;
      for (int w = 0; w < kMeanThreads / 32; ++w) tot += mean_s[w];
      *mean_g = tot / (float(mean_layers) * float(N));
    }
  } else if (!kQuota) {
    // c_j (Eq. 9): g_bar in a fixed order by one thread
    const int j0 = b.req_img_off[seg];
    for (int j = threadIdx.x; j <= K; j += blockDim.x) img_s[j] = b.img_off[j0 + j] - t0;
    if (threadIdx.x == 0) gbar_s = image_mean_f32(g + j0, K);
    __syncthreads();
    const float gbar = gbar_s;
    for (int j = threadIdx.x; j < K; j += blockDim.x) {
      const float c = image_coefficient(__ldcg(g + j0 + j), gbar, lambda, K);
      c_s[j] = c;
      if (coeff) coeff[j0 + j] = c;
    }
    __syncthreads();
  }
  uint32_t kr[kRegKeys > 0 ? kRegKeys : 1];
  bool bad = false;
  {
    int img = 0;  // image of token lo
    if (!kQuota) {
      int a0 = 0, a1 = K - 1;
      while (a0 < a1) {
        const int mid = (a0 + a1 + 1) >> 1;
        if (img_s[mid] <= lo) a0 = mid; else a1 = mid - 1;
      }
      img = a0;
    }
    auto key_of = [&](int t, float st) -> uint32_t {  // st = s[t0 + t]
      float key;
      if (kQuota) {
        key = st;
        const float sh = key * c_seg;
        if (!isfinite(sh) || sh < 0.f || !isfinite(key) || key < 0.f) bad = true;
        if (s_hat) s_hat[t0 + t] = sh == 0.f ? 0.f : sh;
      } else {
        while (img + 1 < K && img_s[img + 1] <= t) ++img;
        key = st * c_s[img];
        if (!isfinite(key) || key < 0.f) bad = true;
        if (s_hat) s_hat[t0 + t] = key == 0.f ? 0.f : key;
      }
      if (key == 0.f) key = 0.f;  // -0 -> +0
      return __float_as_uint(key);
    };
    if (in_regs) {
#pragma unroll
      for (int j = 0; j < kRegKeys; ++j) kr[j] = (lo + j < hi) ? key_of(lo + j, sv[j]) : 0u;
    } else {
      for (int t = lo; t < hi; ++t) keys[t0 + t] = key_of(t, __ldcg(s + t0 + t));
    }
  }
  if (bad) flag_status(status, CONDUIT_FLAG_NONFINITE);
  __syncthreads();

  if (k == 0) {
    if (mask)
      for (int t = threadIdx.x; t < N; t += blockDim.x) mask[t0 + t] = 0;
    return;
  }

  // Radix select of the k-th largest key: four 8-bit digits, MSB first.
  if (threadIdx.x == 0) {
    prefix_s = 0u;
    remaining_s = k;
  }
  uint32_t pmask = 0u;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0u;
    __syncthreads();
    const uint32_t prefix = prefix_s;
    if (in_regs) {
#pragma unroll
      for (int j = 0; j < kRegKeys; ++j)
        if (lo + j < hi && (kr[j] & pmask) == prefix) atomicAdd(&hist[(kr[j] >> shift) & 255u], 1u);
    } else {
      for (int t = lo; t < hi; ++t) {
        const uint32_t key = keys[t0 + t];
        if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // Lane l holds digits 255-8l .. 248-8l (highest first); a warp scan of
      // the lane totals finds the lane whose bins reach the remaining count.
      const int lane = threadIdx.x;
      int cnt[8], lsum = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        cnt[q] = int(hist[255 - 8 * lane - q]);
        lsum += cnt[q];
      }
      int incl = lsum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int rem = remaining_s, excl = incl - lsum;
      const unsigned hit = __ballot_sync(0xffffffffu, excl < rem && rem <= incl);
      if (lane == __ffs(hit) - 1) {
        int r2 = rem - excl, q = 0;
        for (; q < 7; ++q) {
          if (cnt[q] >= r2) break;
          r2 -= cnt[q];
        }
        remaining_s = r2;
        prefix_s = prefix | (uint32_t(255 - 8 * lane - q) << shift);
      }
    }
    pmask |= 255u << shift;
    __syncthreads();
  }
  const uint32_t kth = prefix_s;
  const int need = remaining_s;  // keys equal to kth still to take, >= 1

  // Contiguous token ranges per thread keep the output in ascending order.
  int gt = 0, eq = 0;
  if (in_regs) {
#pragma unroll
    for (int j = 0; j < kRegKeys; ++j)
      if (lo + j < hi) {
        gt += kr[j] > kth;
        eq += kr[j] == kth;
      }
  } else {
    for (int t = lo; t < hi; ++t) {
      const uint32_t key = keys[t0 + t];
      gt += key > kth;
      eq += key == kth;
    }
  }
  const int eq_base = block_exclusive_scan(eq, warp_s, nullptr);
  const int take_eq = max(0, min(eq, need - eq_base));
  const int pos0 = block_exclusive_scan(gt + take_eq, warp_s, nullptr);
  int pos = pos0, seen_eq = 0;
  auto emit = [&](int t, uint32_t key) {
    bool sel = key > kth;
    if (key == kth) {
      sel = seen_eq < take_eq;
      ++seen_eq;
    }
    if (sel) out[pos++] = base_t + t;
    if (mask) mask[t0 + t] = sel ? 1 : 0;
  };
  if (in_regs) {
#pragma unroll
    for (int j = 0; j < kRegKeys; ++j)
      if (lo + j < hi) emit(lo + j, kr[j]);
  } else {
    for (int t = lo; t < hi; ++t) emit(t, keys[t0 + t]);
  }
}

template <int kRegKeys, bool kQuota>
__global__ void __launch_bounds__(kSelThreads) select_kernel(BatchDev b, const float* s,
                                                             const float* g, float lambda,
                                                             const int32_t* idx_off, int32_t* idx,
                                                             uint8_t* mask, float* s_hat,
                                                             float* coeff, uint32_t* keys,
                                                             int32_t* status,
                                                             const float* seg_coeff,
                                                             const int32_t* seg_quota,
                                                             const int32_t* seg_qoff) {
  select_segment<kRegKeys, kQuota>(int(blockIdx.x), b, s, g, lambda, idx_off, idx, mask, s_hat, coeff, keys,
                                   status, seg_coeff, seg_quota, seg_qoff);
}

// ------------------------------------------- scoring tail + selection, fused
// conduit_score_select_topk's one launch after the scoring kernel, for
// batches whose requests each fit one CTA's registers (at most 8 x 1024
// tokens): block i first reduces tokens [32 i, 32 i + 32) over the layers
// exactly as finalize_tokens_kernel does (s_t, A_t); then it counts itself in
// on each request its tokens belong to (one arrival counter per request,
// zeroed before the scoring kernel), and the block that arrives last for a
// request takes that request's image means g_j (Eq. 8, each image by a group
// of 256 threads in image_means_kernel's order), then c_j, s_hat and the
// top-k exactly as select_kernel does. The selection of early requests runs
// while later requests are still being reduced, and the results equal those
// of the three separate launches bit for bit.
template <int kRegKeys>
__global__ void __launch_bounds__(kSelThreads) finalize_select_kernel(
    TokenReduceArgs f, const __grid_constant__ LayerList layers, BatchDev b, float lambda,
    const int32_t* idx_off, int32_t* idx, uint8_t* mask, float* s_hat, float* coeff, float* g,
    int32_t* arrivals) {
  __shared__ float part_s[kLayerSlots][33];
  __shared__ float part_a[kLayerSlots][33];
  __shared__ float mean_s[kSelThreads / kMeanThreads][kMeanThreads / 32];
  __shared__ int done_s[kTokBlock + 1];  // requests this block completes, then their count
  const int64_t tok0 = int64_t(blockIdx.x) * kTokBlock;
  token_reduce_block(f, layers, b, tok0, part_s, part_a);
  __syncthreads();  // this block's s and A are written
  if (threadIdx.x == 0) {
    // Each arrival releases this block's s and A (written before the barrier
    // above) at device scope; the last arrival also acquires every other
    // block's, and the barrier below passes them on to the block's threads.
    const int64_t tok1 = min(tok0 + kTokBlock, f.n_tot);
    int nd = 0;
    for (int r = request_of(b.tok_off, b.R, tok0); r < b.R && b.tok_off[r] < tok1; ++r) {
      const int blocks = (b.tok_off[r + 1] - 1) / kTokBlock - b.tok_off[r] / kTokBlock + 1;
      int old;
      asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(arrivals + r) : "memory");
      if (old == blocks - 1) done_s[nd++] = r;
    }
    done_s[kTokBlock] = nd;
  }
  __syncthreads();
  const int nd = done_s[kTokBlock];
  const int grp = threadIdx.x / kMeanThreads, gt = threadIdx.x % kMeanThreads;
  for (int i = 0; i < nd; ++i) {
    const int r = done_s[i];
    const int j0 = b.req_img_off[r], j1 = b.req_img_off[r + 1];
    if (j1 - j0 == 1) {  // one image: c = 1, so g is formed inside the selection, alongside its loads
      select_segment<kRegKeys, false>(r, b, f.s, g, lambda, idx_off, idx, mask, s_hat, coeff, nullptr,
                                      f.status, nullptr, nullptr, nullptr, f.attn_sum, &g[j0], f.n_layers);
    } else {
      // group grp takes images j0 + grp, j0 + grp + 4, ...; its 256 threads
      // walk the same images, so its named barrier (id grp + 1) always completes
      for (int j = j0 + grp; j < j1; j += kSelThreads / kMeanThreads)
        image_mean_group(f.attn_sum, b.img_off[j], b.img_off[j + 1], f.n_layers, gt, mean_s[grp], &g[j],
                         [grp] { asm volatile("bar.sync %0, %1;" ::"r"(grp + 1), "n"(kMeanThreads) : "memory"); });
      __syncthreads();  // g_j of the request are written
      select_segment<kRegKeys, false>(r, b, f.s, g, lambda, idx_off, idx, mask, s_hat, coeff, nullptr,
                                      f.status, nullptr, nullptr, nullptr);
    }
    __syncthreads();  // the next request reuses the shared arrays
  }
}

// ------------------------------------------------ one cluster per request
// Requests too large for one CTA's registers (more than 8 x 1024 tokens) take
// a cluster of kClusterCtas CTAs: CTA c of the cluster owns the c-th
// contiguous chunk of the request's tokens and keeps its keys in registers.
// Each radix pass builds a 256-bin histogram per CTA in shared memory; after a
// cluster barrier every CTA sums the kClusterCtas histograms through
// distributed shared memory and takes the same digit decision. The selected
// indices go out in ascending order: each CTA's count of keys above the k-th
// and of keys equal to it are exchanged the same way, ties go to the lowest
// tokens. Histograms alternate between two buffers, so one cluster barrier per
// pass suffices (a CTA rewrites a buffer only after every CTA has passed the
// barrier that follows the reads of it).
constexpr int kClusterCtas = 8;

__device__ __forceinline__ void cluster_barrier() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// 32-bit word at the same shared-memory offset in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_ld(const void* local, uint32_t rank) {
  const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(local));
  uint32_t ra, v;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(ra) : "memory");
  return v;
}

template <int kRegKeys>
__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kSelThreads)
    select_cluster_kernel(BatchDev b, const float* s, const float* g, float lambda,
                          const int32_t* idx_off, int32_t* idx, uint8_t* mask, float* s_hat,
                          float* coeff, int32_t* status) {
  __shared__ float c_s[kMaxImagesPerRequest];
  __shared__ int img_s[kMaxImagesPerRequest + 1];
  __shared__ unsigned hist[2][256];
  __shared__ unsigned tot[256];
  __shared__ int warp_s[32];
  __shared__ uint32_t prefix_s;
  __shared__ int remaining_s;
  __shared__ float gbar_s;
  __shared__ int counts_s[2];  // this CTA's keys above the k-th, equal to it

  const uint32_t crank = cluster_rank();
  const int r = blockIdx.x / kClusterCtas;
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  const int j0 = b.req_img_off[r], K = b.req_img_off[r + 1] - j0;
  const int k = idx_off[r + 1] - idx_off[r];
  int32_t* out = idx + idx_off[r];
  for (int j = threadIdx.x; j <= K; j += blockDim.x) img_s[j] = b.img_off[j0 + j] - t0;
  if (threadIdx.x == 0) gbar_s = image_mean_f32(g + j0, K);
  __syncthreads();
  for (int j = threadIdx.x; j < K; j += blockDim.x) {
    const float c = image_coefficient(g[j0 + j], gbar_s, lambda, K);
    c_s[j] = c;
    if (coeff && crank == 0) coeff[j0 + j] = c;
  }
  __syncthreads();

  // this CTA's chunk [c_lo, c_hi), then each thread's contiguous tokens
  const int chunk = (N + kClusterCtas - 1) / kClusterCtas;
  const int c_lo = min(N, int(crank) * chunk), c_hi = min(N, c_lo + chunk);
  const int per = (c_hi - c_lo + kSelThreads - 1) / kSelThreads;
  const int lo = min(c_hi, c_lo + int(threadIdx.x) * per), hi = min(c_hi, lo + per);
  uint32_t kr[kRegKeys];
  bool bad = false;
  {
    int a0 = 0, a1 = K - 1;  // image of token lo
    while (a0 < a1) {
      const int mid = (a0 + a1 + 1) >> 1;
      if (img_s[mid] <= lo) a0 = mid; else a1 = mid - 1;
    }
    int img = a0;
#pragma unroll
    for (int j = 0; j < kRegKeys; ++j) {
      kr[j] = 0u;
      const int t = lo + j;
      if (t < hi) {
        while (img + 1 < K && img_s[img + 1] <= t) ++img;
        float key = s[t0 + t] * c_s[img];
        if (!isfinite(key) || key < 0.f) bad = true;
        if (s_hat) s_hat[t0 + t] = key == 0.f ? 0.f : key;
        if (key == 0.f) key = 0.f;  // -0 -> +0
        kr[j] = __float_as_uint(key);
      }
    }
  }
  if (bad) flag_status(status, CONDUIT_FLAG_NONFINITE);
  if (k == 0) {  // the same for every CTA of the cluster: none touches another's memory
    if (mask)
      for (int t = c_lo + int(threadIdx.x); t < c_hi; t += blockDim.x) mask[t0 + t] = 0;
    return;
  }

  if (threadIdx.x == 0) {
    prefix_s = 0u;
    remaining_s = k;
  }
  uint32_t pmask = 0u;
  int pass = 0;
  for (int shift = 24; shift >= 0; shift -= 8, ++pass) {
    unsigned* h = hist[pass & 1];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0u;
    __syncthreads();
    const uint32_t prefix = prefix_s;
#pragma unroll
    for (int j = 0; j < kRegKeys; ++j)
      if (lo + j < hi && (kr[j] & pmask) == prefix) atomicAdd(&h[(kr[j] >> shift) & 255u], 1u);
    cluster_barrier();  // every CTA's histogram of this pass is complete
    for (int i = threadIdx.x; i < 256; i += blockDim.x) {
      unsigned t = 0u;
      for (uint32_t c = 0; c < kClusterCtas; ++c) t += dsmem_ld(&h[i], c);  // fixed order
      tot[i] = t;
    }
    __syncthreads();
    if (threadIdx.x < 32) {  // the digit holding the remaining rank, as in select_kernel
      const int lane = threadIdx.x;
      int cnt[8], lsum = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        cnt[q] = int(tot[255 - 8 * lane - q]);
        lsum += cnt[q];
      }
      int incl = lsum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int rem = remaining_s, excl = incl - lsum;
      const unsigned hit = __ballot_sync(0xffffffffu, excl < rem && rem <= incl);
      if (lane == __ffs(hit) - 1) {
        int r2 = rem - excl, q = 0;
        for (; q < 7; ++q) {
          if (cnt[q] >= r2) break;
          r2 -= cnt[q];
        }
        remaining_s = r2;
        prefix_s = prefix | (uint32_t(255 - 8 * lane - q) << shift);
      }
    }
    pmask |= 255u << shift;
    __syncthreads();
  }
  const uint32_t kth = prefix_s;
  const int need = remaining_s;  // keys equal to kth still to take over the request, >= 1

  int gt = 0, eq = 0;
#pragma unroll
  for (int j = 0; j < kRegKeys; ++j)
    if (lo + j < hi) {
      gt += kr[j] > kth;
      eq += kr[j] == kth;
    }
  int cta_gt = 0, cta_eq = 0;
  const int eq_base_local = block_exclusive_scan(eq, warp_s, &cta_eq);
  block_exclusive_scan(gt, warp_s, &cta_gt);
  if (threadIdx.x == 0) {
    counts_s[0] = cta_gt;
    counts_s[1] = cta_eq;
  }
  cluster_barrier();  // every CTA's counts are published
  // ties and output slots before this CTA's chunk (lower tokens)
  int eq_before = 0, gt_before = 0;
  for (uint32_t c = 0; c < crank; ++c) {
    gt_before += int(dsmem_ld(&counts_s[0], c));
    eq_before += int(dsmem_ld(&counts_s[1], c));
  }
  const int take_cta = max(0, min(cta_eq, need - eq_before));
  const int out0 = gt_before + min(eq_before, need);
  const int take_eq = max(0, min(eq, take_cta - eq_base_local));
  const int pos0 = out0 + block_exclusive_scan(gt + take_eq, warp_s, nullptr);
  int pos = pos0, seen_eq = 0;
#pragma unroll
  for (int j = 0; j < kRegKeys; ++j) {
    const int t = lo + j;
    if (t < hi) {
      const uint32_t key = kr[j];
      bool sel = key > kth;
      if (key == kth) {
        sel = seen_eq < take_eq;
        ++seen_eq;
      }
      if (sel) out[pos++] = t;
      if (mask) mask[t0 + t] = sel ? 1 : 0;
    }
  }
  cluster_barrier();  // no CTA leaves while another may still read its counts
}

// Quotas of one request (App. D.3): c_j as the global rule computes it, then
// k_j proportional to c_j n_j with sum k_j = k_r and k_j <= n_j, by the largest
// remainder in float64 (w_j = c_j n_j, W summed left to right over the open
// images, ideal_j = (kk w_j) / W; images whose ideal exceeds n_j close at n_j
// and the rest is shared again; leftover units go to the largest remainders,
// ties to the lower index; all-zero weights fall back to n_j). Also the offset
// of each image's indices within the request's slice.
// Dynamic shared memory: K_max doubles (remainders), ints (quotas), bytes (open).
__global__ void __launch_bounds__(kQuotaThreads) quota_kernel(BatchDev b, const float* g, float lambda,
                                                              const int32_t* idx_off, float* c_out,
                                                              int32_t* quota_out, int32_t* qoff_out,
                                                              float* coeff, int32_t* quota_user,
                                                              int32_t* status) {
  extern __shared__ __align__(8) unsigned char qsm[];
  __shared__ float gbar_s;
  __shared__ double total_s;
  __shared__ int kk_s, any_s, zero_s, left_s;
  const int r = blockIdx.x;
  const int j0 = b.req_img_off[r], K = b.req_img_off[r + 1] - j0;
  double* rem_s = reinterpret_cast<double*>(qsm);
  int* quota_s = reinterpret_cast<int*>(rem_s + K);
  unsigned char* open_s = reinterpret_cast<unsigned char*>(quota_s + K);
  if (threadIdx.x == 0) {
    gbar_s = image_mean_f32(g + j0, K);
    kk_s = idx_off[r + 1] - idx_off[r];
  }
  __syncthreads();
  for (int j = threadIdx.x; j < K; j += blockDim.x) {
    const float c = image_coefficient(g[j0 + j], gbar_s, lambda, K);
    c_out[j0 + j] = c;
    if (coeff) coeff[j0 + j] = c;
    quota_s[j] = 0;
    open_s[j] = 1;
  }
  __syncthreads();
  auto n_of = [&](int j) { return b.img_off[j0 + j + 1] - b.img_off[j0 + j]; };
  for (int round = 0; round <= K; ++round) {  // each round closes at least one image or ends
    if (threadIdx.x == 0) {  // W in index order; size weights if every open weight is zero
      int zero = 1;
      for (int j = 0; j < K; ++j)
        if (open_s[j] && double(c_out[j0 + j]) * double(n_of(j)) != 0.0) zero = 0;
      for (int j = 0; j < K; ++j)  // a non-finite c_j (from g): flag it, share by size
        if (open_s[j] && !isfinite(c_out[j0 + j])) {
          zero = 1;
          flag_status(status, CONDUIT_FLAG_NONFINITE);
        }
      double total = 0.0;
      for (int j = 0; j < K; ++j)
        if (open_s[j]) total = total + (zero ? double(n_of(j)) : double(c_out[j0 + j]) * double(n_of(j)));
      zero_s = zero;
      total_s = total;
      any_s = 0;
    }
    __syncthreads();
    const double total = total_s, kk = double(kk_s);
    for (int j = threadIdx.x; j < K; j += blockDim.x) {
      if (!open_s[j]) continue;
      const double w = zero_s ? double(n_of(j)) : double(c_out[j0 + j]) * double(n_of(j));
      const double ideal = total > 0.0 ? (kk * w) / total : 0.0;
      rem_s[j] = ideal;
      if (ideal > double(n_of(j))) any_s = 1;
    }
    __syncthreads();
    if (any_s) {  // close the images over their size
      if (threadIdx.x == 0) {
        int kk2 = kk_s;
        for (int j = 0; j < K; ++j)
          if (open_s[j] && rem_s[j] > double(n_of(j))) {
            quota_s[j] = n_of(j);
            kk2 -= n_of(j);
            open_s[j] = 0;
          }
        kk_s = kk2;
      }
      __syncthreads();
      continue;
    }
    // floors, then the leftover units by remainder rank
    for (int j = threadIdx.x; j < K; j += blockDim.x) {
      if (!open_s[j]) continue;
      const double fl = floor(rem_s[j]);
      quota_s[j] = int(fl);
      rem_s[j] = rem_s[j] - fl;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int used = 0;
      for (int j = 0; j < K; ++j)
        if (open_s[j]) used += quota_s[j];
      left_s = kk_s - used;
    }
    __syncthreads();
    const int left = left_s;
    int add[(kMaxImagesPerRequest + kQuotaThreads - 1) / kQuotaThreads];
    int na = 0;
    for (int j = threadIdx.x; j < K; j += blockDim.x, ++na) {
      add[na] = 0;
      if (!open_s[j]) continue;
      int rank = 0;
      for (int i = 0; i < K; ++i)
        if (open_s[i] && (rem_s[i] > rem_s[j] || (rem_s[i] == rem_s[j] && i < j))) ++rank;
      add[na] = rank < left ? 1 : 0;
    }
    __syncthreads();
    na = 0;
    for (int j = threadIdx.x; j < K; j += blockDim.x, ++na) quota_s[j] += add[na];
    break;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int off = 0;
    for (int j = 0; j < K; ++j) {
      quota_out[j0 + j] = quota_s[j];
      qoff_out[j0 + j] = off;
      if (quota_user) quota_user[j0 + j] = quota_s[j];
      off += quota_s[j];
    }
  }
}

// Scratch of conduit_select_topk_noalloc: the sortable keys of up to
// CONDUIT_NOALLOC_MAX_TOKENS tokens (4 MiB), resident on every device that
// loads the library until the process exits. Each call overwrites the keys of
// its own tokens before reading them, so nothing needs clearing between calls.
constexpr int64_t kNoAllocMaxTokens = CONDUIT_NOALLOC_MAX_TOKENS;
static __device__ __align__(256) uint32_t g_noalloc_keys[kNoAllocMaxTokens];

constexpr int kMaxDevices = 64;
uint32_t* g_noalloc_ptr[kMaxDevices] = {};
std::mutex g_noalloc_mu;

}  // namespace

int64_t select_noalloc_max_tokens() { return kNoAllocMaxTokens; }

cudaError_t launch_select_noalloc(const BatchDev& b, int max_tokens, const float* s, const float* g,
                                  float lambda,
                                  const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                  float* s_hat, float* coeff, int32_t* status,
                                  cudaStream_t stream) {
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err) return err;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  uint32_t* keys = nullptr;
  {
    // Set-up once per device, with that device current: the host-side name of
    // the array is not a device address, so ask the runtime for the address.
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void* p = nullptr;
      err = cudaGetSymbolAddress(&p, g_noalloc_keys);
      if (err) return err;
      g_noalloc_ptr[dev] = static_cast<uint32_t*>(p);
    }
    keys = g_noalloc_ptr[dev];
  }
  return launch_select(b, max_tokens, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys,
                       status, stream, /*cluster_ok=*/false);
}

cudaError_t launch_select(const BatchDev& b, int max_tokens, const float* s, const float* g,
                          float lambda, const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                          float* s_hat, float* coeff, uint32_t* keys, int32_t* status,
                          cudaStream_t stream, bool cluster_ok) {
  // the smallest register budget that holds every request's keys
  if (max_tokens <= kSelThreads)
    select_kernel<1, false><<<b.R, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, nullptr, nullptr, nullptr);
  else if (max_tokens <= 8 * kSelThreads)
    select_kernel<8, false><<<b.R, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, nullptr, nullptr, nullptr);
  else if (cluster_ok && max_tokens <= kClusterCtas * 8 * kSelThreads)
    select_cluster_kernel<8><<<b.R * kClusterCtas, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, status);
  else
    select_kernel<0, false><<<b.R, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, nullptr, nullptr, nullptr);
  count_launches(1);
  return cudaGetLastError();
}

// The fused tail pays one fence and one atomic per token block before the
// block may retire; with more token blocks than SMs those waits queue up
// wave after wave (batched serving: 4 096 blocks, 27 waves, 0.32 ms against
// 0.28 ms for the three separate launches), so it is taken only when every
// token block runs in the first wave.
bool finalize_select_supported(int max_tokens, int64_t n_tot) {
  if (max_tokens > 8 * kSelThreads) return false;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return false;
  return (n_tot + kTokBlock - 1) / kTokBlock <= sms;
}

cudaError_t launch_finalize_select(const float* pa, const float* pa2, const float* ss, const float* vnorm,
                                   int vmode, const LayerList& layers, const BatchDev& b, int n_layers,
                                   int Hkv, int Hq, int rg_max, int group_rows, int parts, int64_t n_tot,
                                   int max_tokens, float* s, float* attn_sum, float* g, float lambda,
                                   const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask, float* s_hat,
                                   float* coeff, int32_t* arrivals, int32_t* status, cudaStream_t stream) {
  if (max_tokens > 8 * kSelThreads) return cudaErrorInvalidValue;
  const TokenReduceArgs f{pa, pa2, ss, vnorm, vmode, n_layers, Hkv, Hq, rg_max, group_rows, parts,
                          n_tot, s, attn_sum, status};
  const unsigned blocks = unsigned((n_tot + kTokBlock - 1) / kTokBlock);
  if (max_tokens <= kSelThreads)
    finalize_select_kernel<1><<<blocks, kSelThreads, 0, stream>>>(f, layers, b, lambda, idx_off_dev, idx, mask,
                                                                   s_hat, coeff, g, arrivals);
  else
    finalize_select_kernel<8><<<blocks, kSelThreads, 0, stream>>>(f, layers, b, lambda, idx_off_dev, idx, mask,
                                                                   s_hat, coeff, g, arrivals);
  count_launches(1);
  return cudaGetLastError();
}

size_t quota_scratch_bytes(int total_images) {
  return size_t(total_images) * (sizeof(float) + 2 * sizeof(int32_t));
}

cudaError_t launch_select_quota(const BatchDev& b, int max_images, int max_image_tokens,
                                const float* s, const float* g, float lambda,
                                const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                                float* s_hat, float* coeff, int32_t* quota, uint32_t* keys,
                                void* scratch, int32_t* status, cudaStream_t stream) {
  float* c_seg = static_cast<float*>(scratch);
  int32_t* q_seg = reinterpret_cast<int32_t*>(c_seg + b.K);
  int32_t* qoff = q_seg + b.K;
  const size_t smem = size_t(max_images) * (sizeof(double) + sizeof(int) + 1);
  cudaError_t err;
  if (smem > 48 * 1024 &&
      (err = cudaFuncSetAttribute(quota_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem))))
    return err;
  quota_kernel<<<b.R, kQuotaThreads, smem, stream>>>(b, g, lambda, idx_off_dev, c_seg, q_seg, qoff,
                                                     coeff, quota, status);
  if ((err = cudaGetLastError())) return err;
  if (max_image_tokens <= kSelThreads)
    select_kernel<1, true><<<b.K, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, c_seg, q_seg, qoff);
  else if (max_image_tokens <= 8 * kSelThreads)
    select_kernel<8, true><<<b.K, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, c_seg, q_seg, qoff);
  else
    select_kernel<0, true><<<b.K, kSelThreads, 0, stream>>>(
        b, s, g, lambda, idx_off_dev, idx, mask, s_hat, coeff, keys, status, c_seg, q_seg, qoff);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
