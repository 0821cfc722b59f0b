// Per-token and per-image reductions of the scoring pass (Conduit Eqs. 6-8).
//   a_t^(l)  = sum_g sum_group,part pa[l][g][group][part][t] / (|Q| Hq)   Eq. 6 (head/query mean)
//   v_t^(l)  = sqrt(sum_g,part ss[l][g][part][t])                     norm of the concatenated heads
//              (or vnorm[layer id][t] when the norms come from the side cache,
//              or 1 when the score is attention alone)
//   s_t      = (1/|L|) sum_l a_t^(l) v_t^(l)                   Eq. 7
//              (with the RMS statistic, abar_t^(l) = sqrt(sum pa2 / (|Q| Hq))
//              of Eq. 4 takes the place of a_t^(l) here)
//   A_t      = sum_l a_t^(l)
//   g_j      = (1/(|L| n_j)) sum_{t in V_j} A_t                Eq. 8
// A block covers 32 tokens with one warp per layer slot (layers l, l+32, ...;
// coalesced loads across the 32 tokens of a warp), then combines the layer
// slots in a fixed order, so the sums are deterministic.
#include "internal.cuh"

namespace conduit {
namespace {

constexpr int kLayerSlots = 32;
constexpr int kBatch = 8;

__global__ void __launch_bounds__(1024) finalize_tokens_kernel(const float* pa, const float* pa2,
                                                               const float* ss, const float* vnorm,
                                                               int vmode,
                                                               const __grid_constant__ LayerList layers,
                                                               BatchDev b, int n_layers, int Hkv,
                                                               int Hq, int rg_max, int group_rows,
                                                               int parts, int64_t n_tot, float* s,
                                                               float* attn_sum, int32_t* status) {
  __shared__ float part_s[kLayerSlots][33];
  __shared__ float part_a[kLayerSlots][33];
  const int lane = threadIdx.x & 31, slot = threadIdx.x >> 5;
  const int64_t tg = int64_t(blockIdx.x) * 32 + lane;
  float acc_s = 0.f, acc_a = 0.f;
  if (tg < n_tot) {
    const int r = request_of(b.tok_off, b.R, tg);
    const int nq = b.q_off[r + 1] - b.q_off[r];
    const float denom = float(nq * Hq);
    const int rows = (Hq / Hkv) * nq;
    const int n_sl = (group_rows ? (rows + group_rows - 1) / group_rows : 1) * parts;
    const int npa = Hkv * n_sl, nss = Hkv * parts;  // partials of one layer
    for (int li = slot; li < n_layers; li += kLayerSlots) {
      // loads go out in batches of eight, so their latencies overlap
      const float* pa_l = pa + int64_t(li) * Hkv * rg_max * parts * n_tot + tg;
      float col = 0.f;
      for (int q0 = 0; q0 < npa; q0 += kBatch) {
        float x[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          const int q = q0 + k;
          x[k] = q < npa ? pa_l[(int64_t(q / n_sl) * rg_max * parts + q % n_sl) * n_tot] : 0.f;
        }
#pragma unroll
        for (int k = 0; k < kBatch; ++k) col += x[k];
      }
      const float a = col / denom;
      float stat = a;
      if (pa2) {  // RMS statistic (Eq. 4) over the same query rows and heads
        const float* p2_l = pa2 + int64_t(li) * Hkv * rg_max * parts * n_tot + tg;
        float col2 = 0.f;
        for (int q0 = 0; q0 < npa; q0 += kBatch) {
          float x[kBatch];
#pragma unroll
          for (int k = 0; k < kBatch; ++k) {
            const int q = q0 + k;
            x[k] = q < npa ? p2_l[(int64_t(q / n_sl) * rg_max * parts + q % n_sl) * n_tot] : 0.f;
          }
#pragma unroll
          for (int k = 0; k < kBatch; ++k) col2 += x[k];
        }
        stat = sqrtf(col2 / denom);
      }
      float vn;
      if (vmode == 2) {
        vn = 1.f;
      } else if (vmode == 1) {
        vn = vnorm[int64_t(layers.ids[li]) * n_tot + tg];
      } else {
        const float* ss_l = ss + int64_t(li) * nss * n_tot + tg;
        float sq = 0.f;
        for (int q0 = 0; q0 < nss; q0 += kBatch) {
          float x[kBatch];
#pragma unroll
          for (int k = 0; k < kBatch; ++k) x[k] = q0 + k < nss ? ss_l[int64_t(q0 + k) * n_tot] : 0.f;
#pragma unroll
          for (int k = 0; k < kBatch; ++k) sq += x[k];
        }
        vn = sqrtf(sq);
      }
      acc_s = fmaf(stat, vn, acc_s);
      acc_a += a;
    }
  }
  part_s[slot][lane] = acc_s;
  part_a[slot][lane] = acc_a;
  __syncthreads();
  if (slot == 0 && tg < n_tot) {
    float ts = 0.f, ta = 0.f;
    const int used = min(kLayerSlots, n_layers);
    for (int w = 0; w < used; ++w) {
      ts += part_s[w][lane];
      ta += part_a[w][lane];
    }
    const float sv = ts / float(n_layers);
    if (!isfinite(sv) || !isfinite(ta)) flag_status(status, CONDUIT_FLAG_NONFINITE);
    s[tg] = sv;
    attn_sum[tg] = ta;
  }
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

cudaError_t launch_finalize(const float* pa, const float* pa2, const float* ss, const float* vnorm,
                            int vmode, const LayerList& layers, const BatchDev& b, int n_layers, int Hkv,
                            int Hq, int rg_max, int group_rows, int parts, int64_t n_tot, float* s,
                            float* attn_sum, float* g, int32_t* status, cudaStream_t stream) {
  if (n_tot == 0) return cudaSuccess;
  const int threads = 32 * std::min(kLayerSlots, n_layers);
  finalize_tokens_kernel<<<unsigned((n_tot + 31) / 32), threads, 0, stream>>>(
      pa, pa2, ss, vnorm, vmode, layers, b, n_layers, Hkv, Hq, rg_max, group_rows, parts, n_tot, s, attn_sum,
      status);
  cudaError_t err = cudaGetLastError();
  if (err) return err;
  image_means_kernel<<<b.K, 256, 0, stream>>>(attn_sum, b, n_layers, g);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
