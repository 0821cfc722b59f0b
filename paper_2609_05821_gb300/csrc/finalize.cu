// Launches of the per-token and per-image reductions of the scoring pass
// (Conduit Eqs. 6-8; the block-level code is in token_reduce.cuh):
// finalize_tokens_kernel reduces 32 tokens per block over the layers (one
// warp per layer slot), image_means_kernel takes one CTA per image.
#include "token_reduce.cuh"

namespace conduit {
namespace {

__global__ void __launch_bounds__(1024) finalize_tokens_kernel(TokenReduceArgs f,
                                                               const __grid_constant__ LayerList layers,
                                                               BatchDev b) {
  __shared__ float part_s[kLayerSlots][33];
  __shared__ float part_a[kLayerSlots][33];
  token_reduce_block(f, layers, b, int64_t(blockIdx.x) * kTokBlock, part_s, part_a);
}

// One CTA of 256 threads per image: g_j by a fixed-order tree reduction of A over its span.
__global__ void __launch_bounds__(kMeanThreads) image_means_kernel(const float* attn_sum, BatchDev b,
                                                                   int n_layers, float* g) {
  __shared__ float warp_s[kMeanThreads / 32];
  const int j = blockIdx.x;
  image_mean_group(attn_sum, b.img_off[j], b.img_off[j + 1], n_layers, int(threadIdx.x), warp_s, &g[j],
                   [] { __syncthreads(); });
}

}  // namespace

cudaError_t launch_finalize(const float* pa, const float* pa2, const float* ss, const float* vnorm,
                            int vmode, const LayerList& layers, const BatchDev& b, int n_layers, int Hkv,
                            int Hq, int rg_max, int group_rows, int parts, int64_t n_tot, float* s,
                            float* attn_sum, float* g, int32_t* status, cudaStream_t stream) {
  if (n_tot == 0) return cudaSuccess;
  const TokenReduceArgs f{pa, pa2, ss, vnorm, vmode, n_layers, Hkv, Hq, rg_max, group_rows, parts,
                          n_tot, s, attn_sum, status};
  const int threads = 32 * std::min(kLayerSlots, n_layers);
  finalize_tokens_kernel<<<unsigned((n_tot + kTokBlock - 1) / kTokBlock), threads, 0, stream>>>(f, layers, b);
  cudaError_t err = cudaGetLastError();
  if (err) return err;
  image_means_kernel<<<b.K, kMeanThreads, 0, stream>>>(attn_sum, b, n_layers, g);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
