// Per-token and per-image reductions of the scoring pass (Conduit Eqs. 6-8).
//   a_t^(l)  = sum_g pa[l][g][t] / (|Q| Hq)            Eq. 6 (head/query mean)
//   v_t^(l)  = sqrt(ss[l][t])                           concatenated-head norm
//   s_t      = (1/|L|) sum_l a_t^(l) v_t^(l)            Eq. 7
//   A_t      = sum_l a_t^(l)
//   g_j      = (1/(|L| n_j)) sum_{t in V_j} A_t         Eq. 8
// Sums run in a fixed order (deterministic).
#include "internal.cuh"

namespace conduit {
namespace {

__global__ void __launch_bounds__(256) finalize_tokens_kernel(const float* pa, const float* ss,
                                                              BatchDev b, int n_layers, int Hkv,
                                                              int Hq, int64_t n_tot, float* s,
                                                              float* attn_sum, int32_t* status) {
  const int64_t tg = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (tg >= n_tot) return;
  const int r = request_of(b.tok_off, b.R, tg);
  const float denom = float((b.q_off[r + 1] - b.q_off[r]) * Hq);
  float acc_s = 0.f, acc_a = 0.f;
  for (int li = 0; li < n_layers; ++li) {
    float col = 0.f;
    for (int g = 0; g < Hkv; ++g) col += pa[(int64_t(li) * Hkv + g) * n_tot + tg];
    const float a = col / denom;
    const float vn = sqrtf(ss[int64_t(li) * n_tot + tg]);
    acc_s = fmaf(a, vn, acc_s);
    acc_a += a;
  }
  const float sv = acc_s / float(n_layers);
  if (!isfinite(sv) || !isfinite(acc_a)) flag_status(status, CONDUIT_FLAG_NONFINITE);
  s[tg] = sv;
  attn_sum[tg] = acc_a;
}

// One CTA per image: g_j by a fixed-order tree reduction of A over its span.
__global__ void __launch_bounds__(256) image_means_kernel(const float* attn_sum, BatchDev b,
                                                          int n_layers, float* g) {
  __shared__ float warp_s[8];
  const int j = blockIdx.x;
  const int lo = b.img_off[j], hi = b.img_off[j + 1];
  float acc = 0.f;
  for (int t = lo + threadIdx.x; t < hi; t += blockDim.x) acc += attn_sum[t];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) warp_s[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tot = 0.f;
    for (int w = 0; w < 8; ++w) tot += warp_s[w];
    g[j] = tot / (float(n_layers) * float(hi - lo));
  }
}

}  // namespace

cudaError_t launch_finalize(const float* pa, const float* ss, const BatchDev& b, int n_layers,
                            int Hkv, int Hq, int64_t n_tot, float* s, float* attn_sum, float* g,
                            int32_t* status, cudaStream_t stream) {
  if (n_tot == 0) return cudaSuccess;
  finalize_tokens_kernel<<<unsigned((n_tot + 255) / 256), 256, 0, stream>>>(
      pa, ss, b, n_layers, Hkv, Hq, n_tot, s, attn_sum, status);
  cudaError_t err = cudaGetLastError();
  if (err) return err;
  image_means_kernel<<<b.K, 256, 0, stream>>>(attn_sum, b, n_layers, g);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
