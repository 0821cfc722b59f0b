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
#include <mutex>

#include "internal.cuh"

namespace conduit {
namespace {

constexpr int kSelThreads = 1024;

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

template <int kRegKeys>  // keys a thread keeps in registers (0: keys in the workspace)
__global__ void __launch_bounds__(kSelThreads) select_kernel(BatchDev b, const float* s,
                                                             const float* g, float lambda,
                                                             const int32_t* idx_off, int32_t* idx,
                                                             uint8_t* mask, float* s_hat,
                                                             float* coeff, uint32_t* keys,
                                                             int32_t* status) {
  __shared__ float c_s[kMaxImagesPerRequest];
  __shared__ int img_s[kMaxImagesPerRequest + 1];
  __shared__ unsigned hist[256];
  __shared__ int warp_s[32];
  __shared__ uint32_t prefix_s;
  __shared__ int remaining_s;
  __shared__ float gbar_s;

  const int r = blockIdx.x;
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  const int j0 = b.req_img_off[r], K = b.req_img_off[r + 1] - j0;
  const int k = idx_off[r + 1] - idx_off[r];
  int32_t* out = idx + idx_off[r];

  // c_j (Eq. 9): g_bar in a fixed order by one thread.
  for (int j = threadIdx.x; j <= K; j += blockDim.x) img_s[j] = b.img_off[j0 + j] - t0;
  if (threadIdx.x == 0) {
    float sum = 0.f;
    for (int j = 0; j < K; ++j) sum += g[j0 + j];
    gbar_s = sum / float(K);
  }
  __syncthreads();
  const float gbar = gbar_s;
  for (int j = threadIdx.x; j < K; j += blockDim.x) {
    const float c = (K == 1 || gbar == 0.f) ? 1.f : (1.f - lambda) + lambda * (g[j0 + j] / gbar);
    c_s[j] = c;
    if (coeff) coeff[j0 + j] = c;
  }
  __syncthreads();

  // s_hat (Eq. 10) and its sortable key. Each thread owns the contiguous
  // tokens [lo, hi); up to kRegKeys of them stay in registers for the radix
  // passes (requests of up to 1024 x kRegKeys tokens), otherwise the keys go
  // through the workspace.
  const int per = (N + kSelThreads - 1) / kSelThreads;
  const int lo = min(N, int(threadIdx.x) * per), hi = min(N, lo + per);
  const bool in_regs = kRegKeys > 0 && per <= kRegKeys;
  uint32_t kr[kRegKeys > 0 ? kRegKeys : 1];
  bool bad = false;
  {
    int img = 0;  // image of token lo
    {
      int a0 = 0, a1 = K - 1;
      while (a0 < a1) {
        const int mid = (a0 + a1 + 1) >> 1;
        if (img_s[mid] <= lo) a0 = mid; else a1 = mid - 1;
      }
      img = a0;
    }
    auto key_of = [&](int t) -> uint32_t {
      while (img + 1 < K && img_s[img + 1] <= t) ++img;
      float sh = s[t0 + t] * c_s[img];
      if (!isfinite(sh) || sh < 0.f) bad = true;
      if (sh == 0.f) sh = 0.f;  // -0 -> +0
      if (s_hat) s_hat[t0 + t] = sh;
      return __float_as_uint(sh);
    };
    if (in_regs) {
#pragma unroll
      for (int j = 0; j < kRegKeys; ++j) kr[j] = (lo + j < hi) ? key_of(lo + j) : 0u;
    } else {
      for (int t = lo; t < hi; ++t) keys[t0 + t] = key_of(t);
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
    if (sel) out[pos++] = t;
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

// Scratch of conduit_select_topk_noalloc: the sortable keys of up to
// kNoAllocMaxTokens tokens (4 MiB), resident on every device that loads the
// library until the process exits. Each call overwrites the keys of its own
// tokens before reading them, so nothing needs clearing between calls.
constexpr int64_t kNoAllocMaxTokens = int64_t(1) << 20;
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
                       status, stream);
}

cudaError_t launch_select(const BatchDev& b, int max_tokens, const float* s, const float* g,
                          float lambda, const int32_t* idx_off_dev, int32_t* idx, uint8_t* mask,
                          float* s_hat, float* coeff, uint32_t* keys, int32_t* status,
                          cudaStream_t stream) {
  // the smallest register budget that holds every request's keys
  if (max_tokens <= kSelThreads)
    select_kernel<1><<<b.R, kSelThreads, 0, stream>>>(b, s, g, lambda, idx_off_dev, idx, mask, s_hat,
                                                      coeff, keys, status);
  else if (max_tokens <= 8 * kSelThreads)
    select_kernel<8><<<b.R, kSelThreads, 0, stream>>>(b, s, g, lambda, idx_off_dev, idx, mask, s_hat,
                                                      coeff, keys, status);
  else
    select_kernel<0><<<b.R, kSelThreads, 0, stream>>>(b, s, g, lambda, idx_off_dev, idx, mask, s_hat,
                                                      coeff, keys, status);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
