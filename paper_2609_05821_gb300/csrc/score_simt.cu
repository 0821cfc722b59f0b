// CUDA-core scoring pass (any head_dim multiple of 8 up to 256, fp32 or bf16).
//
// Conduit Eq. 6 needs, per (request, layer, KV head g), the softmax over all
// N_r visual keys of every scoring row (query head h of group g, query q):
//   pass 1  row statistics: m = max_t x_t and Z = sum_t 2^(x_t - m), with
//           x = <q, k_t> log2(e) / sqrt(d) (the log2 domain keeps exp2 exact
//           to the same softmax);
//   pass 2  column sums pa[l][g][t] = sum_rows 2^(x_t - m - log2 Z), i.e. the
//           sum over the group's heads and the span of alpha_{q,t}.
// Value norms (Sec. 3.3, concatenated heads) are a separate streaming
// reduction ss[l][t] = sum_g sum_e V[l][g][t][e]^2.
// All reductions run in a fixed order, so results are deterministic.
#include "internal.cuh"

namespace conduit {
namespace {

constexpr int kRowBlock = 32;   // scoring rows per CTA block
constexpr int kTokTile = 32;    // tokens per tile
constexpr int kThreads = 256;   // 32 rows x 8 token lanes

template <typename T>
__device__ __forceinline__ void load_rows_to_smem(float* dst, int ld, const T* src_base,
                                                  const int64_t* row_off, int nrows, int d) {
  // row_off[i] < 0 marks a missing row (filled with zeros)
  for (int idx = threadIdx.x; idx < nrows * d; idx += blockDim.x) {
    const int i = idx / d, e = idx % d;
    const int64_t off = row_off[i];
    dst[i * ld + e] = off >= 0 ? to_float(src_base[off + e]) : 0.f;
  }
}

// Pass 1: one CTA per (row block, layer*Hkv + g, request); sweeps all tokens.
template <typename T>
__global__ void __launch_bounds__(kThreads) rowstats_kernel(KvDev kv, BatchDev b, const T* q,
                                                            int32_t q_tot, LayerList layers,
                                                            float2* stats) {
  extern __shared__ float smem[];
  const int d = kv.d, ld = d + 1;
  float* q_s = smem;                       // [32][d+1]
  float* k_s = smem + kRowBlock * ld;      // [32][d+1]
  __shared__ int64_t q_off_s[kRowBlock], k_off_s[kTokTile];

  const int r = blockIdx.z;
  const int li = blockIdx.y / kv.Hkv, g = blockIdx.y % kv.Hkv;
  const int l = layers.ids[li];
  const int q0 = b.q_off[r], nq = b.q_off[r + 1] - q0;
  const int R = kv.G * nq;
  const int row0 = blockIdx.x * kRowBlock;
  if (row0 >= R || nq == 0) return;
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;

  if (threadIdx.x < kRowBlock) {
    const int rr = row0 + threadIdx.x;
    int64_t off = -1;
    if (rr < R) {
      const int h = g * kv.G + rr / nq, qi = rr % nq;
      off = ((int64_t(l) * kv.Hq + h) * q_tot + q0 + qi) * d;
    }
    q_off_s[threadIdx.x] = off;
  }
  __syncthreads();
  load_rows_to_smem(q_s, ld, q, q_off_s, kRowBlock, d);

  const int i = threadIdx.x / 8, j = threadIdx.x % 8;
  const float scale = kLog2e * rsqrtf(float(d));
  float m_run = -INFINITY, z_run = 0.f;
  const T* kbase = static_cast<const T*>(kv.k);

  for (int tt = 0; tt < N; tt += kTokTile) {
    __syncthreads();
    if (threadIdx.x < kTokTile) {
      const int t = tt + threadIdx.x;
      k_off_s[threadIdx.x] = t < N ? kv.row(l, g, r, int64_t(t0) + t, t) : -1;
    }
    __syncthreads();
    load_rows_to_smem(k_s, ld, kbase, k_off_s, kTokTile, d);
    __syncthreads();
    float x[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) x[m] = 0.f;
    for (int e = 0; e < d; ++e) {
      const float qe = q_s[i * ld + e];
#pragma unroll
      for (int m = 0; m < 4; ++m) x[m] = fmaf(qe, k_s[(j + 8 * m) * ld + e], x[m]);
    }
    float tmax = -INFINITY;
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      x[m] = (tt + j + 8 * m < N) ? x[m] * scale : -INFINITY;
      tmax = fmaxf(tmax, x[m]);
    }
    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 1));
    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));
    tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 4));
    const float m_new = fmaxf(m_run, tmax);
    float psum = 0.f;
#pragma unroll
    for (int m = 0; m < 4; ++m) psum += exp2f(x[m] - m_new);
    psum += __shfl_xor_sync(0xffffffffu, psum, 1);
    psum += __shfl_xor_sync(0xffffffffu, psum, 2);
    psum += __shfl_xor_sync(0xffffffffu, psum, 4);
    z_run = z_run * exp2f(m_run - m_new) + psum;
    m_run = m_new;
  }
  const int rr = row0 + i;
  if (j == 0 && rr < R) {
    const int64_t base = int64_t(blockIdx.y) * kv.G * q_tot + int64_t(kv.G) * q0;
    stats[base + rr] = make_float2(m_run, z_run);
  }
}

// Pass 2: one CTA per (token tile, layer*Hkv + g, request); loops over all
// row blocks of the slab and writes the complete column sums of its tile.
template <typename T>
__global__ void __launch_bounds__(kThreads) colsum_kernel(KvDev kv, BatchDev b, const T* q,
                                                          int32_t q_tot, LayerList layers,
                                                          const float2* stats, float* pa,
                                                          float* pa2, const float* extra_lse) {
  extern __shared__ float smem[];
  const int d = kv.d, ld = d + 1;
  float* q_s = smem;
  float* k_s = smem + kRowBlock * ld;
  __shared__ int64_t q_off_s[kRowBlock], k_off_s[kTokTile];
  __shared__ float lse_s[kRowBlock];
  __shared__ float red_s[kThreads / 32][kTokTile];
  __shared__ float red2_s[kThreads / 32][kTokTile];

  const int r = blockIdx.z;
  const int li = blockIdx.y / kv.Hkv, g = blockIdx.y % kv.Hkv;
  const int l = layers.ids[li];
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  const int tt = blockIdx.x * kTokTile;
  if (tt >= N) return;
  const int q0 = b.q_off[r], nq = b.q_off[r + 1] - q0;
  const int R = kv.G * nq;
  const int64_t sbase = int64_t(blockIdx.y) * kv.G * q_tot + int64_t(kv.G) * q0;

  if (threadIdx.x < kTokTile) {
    const int t = tt + threadIdx.x;
    k_off_s[threadIdx.x] = t < N ? kv.row(l, g, r, int64_t(t0) + t, t) : -1;
  }
  __syncthreads();
  load_rows_to_smem(k_s, ld, static_cast<const T*>(kv.k), k_off_s, kTokTile, d);

  const int i = threadIdx.x / 8, j = threadIdx.x % 8;
  const float scale = kLog2e * rsqrtf(float(d));
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  float acc2[4] = {0.f, 0.f, 0.f, 0.f};

  for (int row0 = 0; row0 < R; row0 += kRowBlock) {
    __syncthreads();
    if (threadIdx.x < kRowBlock) {
      const int rr = row0 + threadIdx.x;
      int64_t off = -1;
      float lse = 0.f;
      if (rr < R) {
        const int h = g * kv.G + rr / nq, qi = rr % nq;
        off = ((int64_t(l) * kv.Hq + h) * q_tot + q0 + qi) * d;
        const float2 st = stats[sbase + rr];
        lse = st.x + log2f(st.y);
        if (extra_lse)  // full-context softmax: keys outside the visual span join the denominator
          lse = log2_add(lse, extra_lse[(int64_t(l) * kv.Hq + h) * q_tot + q0 + qi] * kLog2e);
      }
      q_off_s[threadIdx.x] = off;
      lse_s[threadIdx.x] = lse;
    }
    __syncthreads();
    load_rows_to_smem(q_s, ld, q, q_off_s, kRowBlock, d);
    __syncthreads();
    float x[4] = {0.f, 0.f, 0.f, 0.f};
    for (int e = 0; e < d; ++e) {
      const float qe = q_s[i * ld + e];
#pragma unroll
      for (int m = 0; m < 4; ++m) x[m] = fmaf(qe, k_s[(j + 8 * m) * ld + e], x[m]);
    }
    const bool row_ok = row0 + i < R;
    const float lse = lse_s[i];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      float p = (row_ok && tt + j + 8 * m < N) ? exp2f(x[m] * scale - lse) : 0.f;
      float p2 = p * p;
      // sum over the 4 rows of this warp that share token lane j
      p += __shfl_xor_sync(0xffffffffu, p, 8);
      p += __shfl_xor_sync(0xffffffffu, p, 16);
      acc[m] += p;
      if (pa2) {
        p2 += __shfl_xor_sync(0xffffffffu, p2, 8);
        p2 += __shfl_xor_sync(0xffffffffu, p2, 16);
        acc2[m] += p2;
      }
    }
  }
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (lane < 8) {
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      red_s[warp][lane + 8 * m] = acc[m];
      red2_s[warp][lane + 8 * m] = acc2[m];
    }
  }
  __syncthreads();
  if (threadIdx.x < kTokTile && tt + threadIdx.x < N) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) sum += red_s[w][threadIdx.x];
    pa[int64_t(blockIdx.y) * kv.n_tot + t0 + tt + threadIdx.x] = sum;
    if (pa2) {
      float sum2 = 0.f;
#pragma unroll
      for (int w = 0; w < kThreads / 32; ++w) sum2 += red2_s[w][threadIdx.x];
      pa2[int64_t(blockIdx.y) * kv.n_tot + t0 + tt + threadIdx.x] = sum2;
    }
  }
}

// ss[li][g][tg] = sum over e of V[l][g][t][e]^2 for every KV head g; one warp per token.
template <typename T>
__global__ void __launch_bounds__(256) value_sumsq_kernel(KvDev kv, BatchDev b, LayerList layers,
                                                          float* ss) {
  const int r = blockIdx.y, li = blockIdx.z, l = layers.ids[li];
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  const int t = blockIdx.x * 8 + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (t >= N) return;
  const T* vb = static_cast<const T*>(kv.v);
  for (int g = 0; g < kv.Hkv; ++g) {
    const float acc = warp_row_sumsq(vb + kv.row(l, g, r, int64_t(t0) + t, t), kv.d, lane);
    if (lane == 0) ss[(int64_t(li) * kv.Hkv + g) * kv.n_tot + t0 + t] = acc;
  }
}

}  // namespace

cudaError_t launch_value_sumsq(const KvDev& kv, const BatchDev& b, const LayerList& layers,
                               int max_tokens, float* ss, cudaStream_t stream) {
  const dim3 grid((max_tokens + 7) / 8, b.R, layers.n);
  if (grid.x == 0 || layers.n == 0) return cudaSuccess;
  if (kv.dtype == CONDUIT_BF16)
    value_sumsq_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(kv, b, layers, ss);
  else
    value_sumsq_kernel<float><<<grid, 256, 0, stream>>>(kv, b, layers, ss);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_score_simt(const KvDev& kv, const BatchDev& b, const void* q, int32_t q_tot,
                              const LayerList& layers, int max_rows, int max_tokens,
                              float2* stats, float* pa, float* pa2, const float* extra_lse,
                              cudaStream_t stream) {
  if (layers.n == 0 || max_rows == 0 || max_tokens == 0) return cudaSuccess;
  const size_t smem = size_t(kRowBlock + kTokTile) * (kv.d + 1) * sizeof(float);
  const dim3 g1((max_rows + kRowBlock - 1) / kRowBlock, layers.n * kv.Hkv, b.R);
  const dim3 g2((max_tokens + kTokTile - 1) / kTokTile, layers.n * kv.Hkv, b.R);
  cudaError_t err;
  if (kv.dtype == CONDUIT_BF16) {
    auto* f1 = rowstats_kernel<__nv_bfloat16>;
    auto* f2 = colsum_kernel<__nv_bfloat16>;
    if ((err = cudaFuncSetAttribute(f1, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    if ((err = cudaFuncSetAttribute(f2, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    const auto* qq = static_cast<const __nv_bfloat16*>(q);
    f1<<<g1, kThreads, smem, stream>>>(kv, b, qq, q_tot, layers, stats);
    if ((err = cudaGetLastError())) return err;
    f2<<<g2, kThreads, smem, stream>>>(kv, b, qq, q_tot, layers, stats, pa, pa2, extra_lse);
  } else {
    auto* f1 = rowstats_kernel<float>;
    auto* f2 = colsum_kernel<float>;
    if ((err = cudaFuncSetAttribute(f1, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    if ((err = cudaFuncSetAttribute(f2, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    const auto* qq = static_cast<const float*>(q);
    f1<<<g1, kThreads, smem, stream>>>(kv, b, qq, q_tot, layers, stats);
    if ((err = cudaGetLastError())) return err;
    f2<<<g2, kThreads, smem, stream>>>(kv, b, qq, q_tot, layers, stats, pa, pa2, extra_lse);
  }
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
