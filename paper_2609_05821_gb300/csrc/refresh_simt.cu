// CUDA-core causal refresh attention over the patched cache (selective
// recompute, Conduit Sec. 3.1 / 4.3):
//   out[l][i][h] = sum_{j <= p_i} softmax_j(<q[l][i][h], K'[l][h/G][j]> / sqrt(d)) V'[l][h/G][j]
// One CTA per (selected row, KV head, layer) handles the G query heads that
// share the KV head; keys stream through shared memory in tiles of 32 with an
// online softmax (running max and sum per head) in the log2 domain.
#include "internal.cuh"

namespace conduit {
namespace {

constexpr int kRThreads = 128;
constexpr int kKeyTile = 32;
constexpr int kMaxOutPerThread = 32;  // G * d / 128 outputs per thread (G*d <= 4096)

template <typename T>
__global__ void __launch_bounds__(kRThreads) refresh_simt_kernel(KvDev kv, BatchDev b,
                                                                 const int32_t* idx,
                                                                 const int32_t* idx_off,
                                                                 int32_t n_sel, const T* q_rows,
                                                                 T* out) {
  extern __shared__ float sm[];
  const int d = kv.d, G = kv.G, ld = d + 1;
  float* q_s = sm;                         // [G][d]
  float* k_s = q_s + G * d;                // [32][d+1]
  float* v_s = k_s + kKeyTile * ld;        // [32][d]
  float* p_s = v_s + kKeyTile * d;         // [G][32]
  float* m_s = p_s + G * kKeyTile;         // [G]
  float* l_s = m_s + G;                    // [G]
  float* f_s = l_s + G;                    // [G] rescale factor of this tile
  __shared__ int64_t off_s[kKeyTile];

  const int i = blockIdx.x, g = blockIdx.y, l = blockIdx.z;
  const int r = request_of(idx_off, b.R, i);
  const int t0 = b.tok_off[r], N = b.tok_off[r + 1] - t0;
  const int p = idx[i];
  if (p < 0 || p >= N) return;
  const float scale = kLog2e * rsqrtf(float(d));

  for (int x = threadIdx.x; x < G * d; x += blockDim.x) {
    const int hh = x / d, e = x % d;
    q_s[x] = to_float(q_rows[((int64_t(l) * n_sel + i) * kv.Hq + g * G + hh) * d + e]) * scale;
  }
  for (int hh = threadIdx.x; hh < G; hh += blockDim.x) {
    m_s[hh] = -INFINITY;
    l_s[hh] = 0.f;
  }
  float acc[kMaxOutPerThread];
  const int n_out = (G * d + kRThreads - 1) / kRThreads;
#pragma unroll
  for (int u = 0; u < kMaxOutPerThread; ++u) acc[u] = 0.f;

  const T* kb = static_cast<const T*>(kv.k);
  const T* vb = static_cast<const T*>(kv.v);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  for (int j0 = 0; j0 <= p; j0 += kKeyTile) {
    __syncthreads();
    if (threadIdx.x < kKeyTile) {
      const int j = j0 + threadIdx.x;
      off_s[threadIdx.x] = j <= p ? kv.row(l, g, r, int64_t(t0) + j, j) : -1;
    }
    __syncthreads();
    for (int x = threadIdx.x; x < kKeyTile * d; x += blockDim.x) {
      const int jj = x / d, e = x % d;
      const int64_t off = off_s[jj];
      k_s[jj * ld + e] = off >= 0 ? to_float(kb[off + e]) : 0.f;
      v_s[jj * d + e] = off >= 0 ? to_float(vb[off + e]) : 0.f;
    }
    __syncthreads();
    for (int x = threadIdx.x; x < G * kKeyTile; x += blockDim.x) {
      const int hh = x / kKeyTile, jj = x % kKeyTile;
      float dot = 0.f;
      for (int e = 0; e < d; ++e) dot = fmaf(q_s[hh * d + e], k_s[jj * ld + e], dot);
      p_s[x] = (j0 + jj <= p) ? dot : -INFINITY;
    }
    __syncthreads();
    for (int hh = warp; hh < G; hh += kRThreads / 32) {
      const float xv = p_s[hh * kKeyTile + lane];
      float tmax = xv;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
      const float m_old = m_s[hh];
      const float m_new = fmaxf(m_old, tmax);
      const float pv = exp2f(xv - m_new);
      float psum = pv;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
      p_s[hh * kKeyTile + lane] = pv;
      __syncwarp();
      if (lane == 0) {
        const float f = exp2f(m_old - m_new);
        f_s[hh] = f;
        l_s[hh] = l_s[hh] * f + psum;
        m_s[hh] = m_new;
      }
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < kMaxOutPerThread; ++u) {
      if (u >= n_out) break;
      const int x = threadIdx.x + u * kRThreads;
      if (x >= G * d) break;
      const int hh = x / d, e = x % d;
      float a = acc[u] * f_s[hh];
      for (int jj = 0; jj < kKeyTile; ++jj) a = fmaf(p_s[hh * kKeyTile + jj], v_s[jj * d + e], a);
      acc[u] = a;
    }
  }
  __syncthreads();
#pragma unroll
  for (int u = 0; u < kMaxOutPerThread; ++u) {
    if (u >= n_out) break;
    const int x = threadIdx.x + u * kRThreads;
    if (x >= G * d) break;
    const int hh = x / d, e = x % d;
    out[((int64_t(l) * n_sel + i) * kv.Hq + g * G + hh) * d + e] = from_float<T>(acc[u] / l_s[hh]);
  }
}

}  // namespace

cudaError_t launch_refresh_simt(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                                const int32_t* idx_off_dev, int32_t n_sel, const void* q_rows,
                                void* out, cudaStream_t stream) {
  if (n_sel == 0) return cudaSuccess;
  const int d = kv.d, G = kv.G;
  const size_t smem = sizeof(float) * (size_t(G) * d + kKeyTile * (d + 1) + kKeyTile * d +
                                       G * kKeyTile + 3 * G);
  const dim3 grid(n_sel, kv.Hkv, kv.L);
  cudaError_t err;
  if (kv.dtype == CONDUIT_BF16) {
    auto* f = refresh_simt_kernel<__nv_bfloat16>;
    if ((err = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    f<<<grid, kRThreads, smem, stream>>>(kv, b, idx, idx_off_dev, n_sel,
                                         static_cast<const __nv_bfloat16*>(q_rows),
                                         static_cast<__nv_bfloat16*>(out));
  } else {
    auto* f = refresh_simt_kernel<float>;
    if ((err = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)))) return err;
    f<<<grid, kRThreads, smem, stream>>>(kv, b, idx, idx_off_dev, n_sel,
                                         static_cast<const float*>(q_rows),
                                         static_cast<float*>(out));
  }
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
