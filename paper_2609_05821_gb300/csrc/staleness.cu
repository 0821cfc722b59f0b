// Isotropic Monte Carlo staleness estimator (Conduit App. D): the error a
// refresh set T leaves under sampled stale value displacements,
//   E_iso(T) = sum_{l, h, q} (1/M) sum_m || sum_{t not in T} alpha_{q,t} xi_t^(m) ||^2,
//   xi_t^(m) = kappa ||V_{l,g,t}|| / sqrt(d) z_{l,g,t}^(m)   (per layer, KV head, token).
// sum_t alpha_{q,t} xi_t is the attention output of query row q over all the
// request's visual keys with the values xi (zero for t in T), so each draw m
// runs the refresh attention kernels with every scoring row at position
// N_r - 1 over (K, xi^(m)); these kernels build xi^(m) in the cache's own
// layout, lay the scoring queries out as refresh rows, and reduce ||O||^2.
#include "internal.cuh"

namespace conduit {
namespace {

// Per (layer, KV head, token) row: the standard deviation of its draws,
// kappa ||V|| / sqrt(d), or 0 when the token is refreshed (the same for every
// draw, so computed once). One warp per row.
template <typename T>
__global__ void __launch_bounds__(256) stale_scale_kernel(KvDev kv, BatchDev b,
                                                          const uint8_t* refreshed, float kappa,
                                                          float* scale) {
  const int64_t row = int64_t(blockIdx.x) * 8 + threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int64_t rows = int64_t(kv.L) * kv.Hkv * kv.n_tot;
  if (row >= rows) return;
  const int64_t tg = row % kv.n_tot;
  const int lg = int(row / kv.n_tot);
  const int r = request_of(b.tok_off, b.R, tg);
  const int t = int(tg - b.tok_off[r]);
  const T* vb = static_cast<const T*>(kv.v);
  const float ss = warp_row_sumsq(vb + kv.row(lg / kv.Hkv, lg % kv.Hkv, r, tg, t), kv.d, lane);
  if (lane == 0) scale[row] = refreshed[tg] ? 0.f : kappa * sqrtf(ss / float(kv.d));
}

// xi^(m) rows in the layout of kv.v (contiguous or paged): one warp per
// (layer, KV head, token) row, xi = scale * z.
template <typename T>
__global__ void __launch_bounds__(256) stale_values_kernel(KvDev kv, BatchDev b, const float* scale,
                                                           const T* z, T* xi) {
  const int64_t row = int64_t(blockIdx.x) * 8 + threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int64_t rows = int64_t(kv.L) * kv.Hkv * kv.n_tot;
  if (row >= rows) return;
  const int64_t tg = row % kv.n_tot;
  const int lg = int(row / kv.n_tot);
  const int r = request_of(b.tok_off, b.R, tg);
  const int t = int(tg - b.tok_off[r]);
  const int64_t off = kv.row(lg / kv.Hkv, lg % kv.Hkv, r, tg, t);
  const float sc = scale[row];
  const T* zr = z + row * kv.d;  // z is [L][Hkv][N_tot][d]
  for (int e = lane; e < kv.d; e += 32) xi[off + e] = from_float<T>(sc * to_float(zr[e]));
}

// q [L][Hq][Q_tot][d] -> rows [L][Q_tot][Hq][d] (the refresh kernels' row layout).
template <typename T>
__global__ void __launch_bounds__(256) stale_queries_kernel(const T* q, int L, int Hq, int q_tot, int d,
                                                            T* rows) {
  const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t n = int64_t(L) * Hq * q_tot * d;
  if (i >= n) return;
  const int e = int(i % d);
  int64_t x = i / d;
  const int h = int(x % Hq);
  x /= Hq;
  const int qi = int(x % q_tot);
  const int l = int(x / q_tot);
  rows[i] = q[((int64_t(l) * Hq + h) * q_tot + qi) * d + e];
}

// Every scoring row of request r sits at position N_r - 1 (all keys visible).
__global__ void stale_positions_kernel(BatchDev b, int32_t* pos) {
  const int r = blockIdx.x;
  const int n = b.tok_off[r + 1] - b.tok_off[r];
  for (int i = b.q_off[r] + threadIdx.x; i < b.q_off[r + 1]; i += blockDim.x) pos[i] = n - 1;
}

// part[r][l] += sum over the request's rows and heads of ||O[l][q][h]||^2, one
// block per (layer, request), fixed-order reduction.
template <typename T>
__global__ void __launch_bounds__(256) stale_reduce_kernel(const T* out, BatchDev b, int L, int Hq,
                                                           int q_tot, int d, double* part) {
  __shared__ double warp_s[8];
  const int l = blockIdx.x, r = blockIdx.y;
  const int q0 = b.q_off[r], nq = b.q_off[r + 1] - q0;
  const int64_t base = (int64_t(l) * q_tot + q0) * Hq * d;
  const int64_t n = int64_t(nq) * Hq * d;
  float acc = 0.f;
  for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
    const float x = to_float(out[base + i]);
    acc = fmaf(x, x, acc);
  }
  double a = acc;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
  if ((threadIdx.x & 31) == 0) warp_s[threadIdx.x >> 5] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    double tot = 0.0;
    for (int w = 0; w < 8; ++w) tot += warp_s[w];
    part[int64_t(r) * L + l] += tot;
  }
}

// err[r] = sum_l part[r][l] / M, and per layer err_rl[r][l] = part[r][l] / M.
__global__ void stale_final_kernel(const double* part, int R, int L, int M, double* err,
                                   double* err_rl) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  double tot = 0.0;
  for (int l = 0; l < L; ++l) {
    const double x = part[int64_t(r) * L + l] / double(M);
    if (err_rl) err_rl[int64_t(r) * L + l] = x;
    tot += x;
  }
  err[r] = tot;
}

}  // namespace

StaleLayout stale_layout(const KvDev& kv, const BatchDev& b, int32_t q_tot, int M) {
  (void)M;
  const size_t esz = kv.dtype == CONDUIT_BF16 ? 2 : 4;
  auto up = [](size_t x) { return (x + 255) / 256 * 256; };
  StaleLayout s{};
  const size_t v_elems = kv.page_size == 0
                             ? size_t(kv.L) * kv.Hkv * size_t(kv.n_tot) * kv.d
                             : size_t(kv.L) * kv.num_pages * kv.Hkv * size_t(kv.page_size) * kv.d;
  s.xi_bytes = v_elems * esz;
  size_t off = 0;
  s.xi = off;
  off += up(s.xi_bytes);
  s.rows = off;
  off += up(size_t(kv.L) * q_tot * kv.Hq * kv.d * esz);
  s.out = off;
  off += up(size_t(kv.L) * q_tot * kv.Hq * kv.d * esz);
  s.pos = off;
  off += up(size_t(q_tot) * 4);
  s.part = off;
  off += up(size_t(b.R) * kv.L * 8);
  s.scale = off;
  off += up(size_t(kv.L) * kv.Hkv * size_t(kv.n_tot) * 4);
  s.counter = off;
  off += 256;
  s.total = off;
  return s;
}

cudaError_t launch_staleness_iso(const KvDev& kv, const BatchDev& b, const int32_t* q_off_host,
                                 int32_t q_tot, const void* q, const uint8_t* refreshed,
                                 const void* z, int M, float kappa, double* err, double* err_rl,
                                 void* workspace, int32_t* status, cudaStream_t stream) {
  const StaleLayout lay = stale_layout(kv, b, q_tot, M);
  char* ws = static_cast<char*>(workspace);
  void* xi = ws + lay.xi;
  void* rows = ws + lay.rows;
  void* out = ws + lay.out;
  int32_t* pos = reinterpret_cast<int32_t*>(ws + lay.pos);
  double* part = reinterpret_cast<double*>(ws + lay.part);
  float* scale = reinterpret_cast<float*>(ws + lay.scale);
  int32_t* counter = reinterpret_cast<int32_t*>(ws + lay.counter);
  const bool bf16 = kv.dtype == CONDUIT_BF16;
  cudaError_t err_c;
  // pool rows that hold no token (a partial last page) stay zero for every draw
  if ((err_c = cudaMemsetAsync(xi, 0, lay.xi_bytes, stream))) return err_c;
  if ((err_c = cudaMemsetAsync(part, 0, size_t(b.R) * kv.L * 8, stream))) return err_c;
  const int64_t nq = int64_t(kv.L) * kv.Hq * q_tot * kv.d;
  if (nq > 0) {
    const unsigned blocks = unsigned((nq + 255) / 256);
    if (bf16)
      stale_queries_kernel<__nv_bfloat16><<<blocks, 256, 0, stream>>>(
          static_cast<const __nv_bfloat16*>(q), kv.L, kv.Hq, q_tot, kv.d, static_cast<__nv_bfloat16*>(rows));
    else
      stale_queries_kernel<float><<<blocks, 256, 0, stream>>>(static_cast<const float*>(q), kv.L, kv.Hq,
                                                              q_tot, kv.d, static_cast<float*>(rows));
    stale_positions_kernel<<<b.R, 128, 0, stream>>>(b, pos);
    count_launches(2);
    if ((err_c = cudaGetLastError())) return err_c;
  }
  KvDev kx = kv;
  kx.v = xi;
  const int64_t vrows = int64_t(kv.L) * kv.Hkv * kv.n_tot;
  const int64_t zdraw = vrows * kv.d;  // elements of one draw
  const unsigned vblocks = unsigned((vrows + 7) / 8);
  if (vrows > 0) {
    if (bf16)
      stale_scale_kernel<__nv_bfloat16><<<vblocks, 256, 0, stream>>>(kv, b, refreshed, kappa, scale);
    else
      stale_scale_kernel<float><<<vblocks, 256, 0, stream>>>(kv, b, refreshed, kappa, scale);
    count_launches(1);
    if ((err_c = cudaGetLastError())) return err_c;
  }
  for (int m = 0; m < M; ++m) {
    if (bf16)
      stale_values_kernel<__nv_bfloat16><<<vblocks, 256, 0, stream>>>(
          kv, b, scale, static_cast<const __nv_bfloat16*>(z) + m * zdraw, static_cast<__nv_bfloat16*>(xi));
    else
      stale_values_kernel<float><<<vblocks, 256, 0, stream>>>(
          kv, b, scale, static_cast<const float*>(z) + m * zdraw, static_cast<float*>(xi));
    count_launches(1);
    if ((err_c = cudaGetLastError())) return err_c;
    if (q_tot > 0) {
      err_c = refresh_tc_supported(kx)
                  ? launch_refresh_tc(kx, b, pos, b.q_off, q_off_host, q_tot, rows, out, counter, status,
                                      stream)
                  : launch_refresh_simt(kx, b, pos, b.q_off, q_tot, rows, out, stream);
      if (err_c) return err_c;
      const dim3 grid(kv.L, b.R);
      if (bf16)
        stale_reduce_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(
            static_cast<const __nv_bfloat16*>(out), b, kv.L, kv.Hq, q_tot, kv.d, part);
      else
        stale_reduce_kernel<float><<<grid, 256, 0, stream>>>(static_cast<const float*>(out), b, kv.L,
                                                             kv.Hq, q_tot, kv.d, part);
      count_launches(1);
      if ((err_c = cudaGetLastError())) return err_c;
    }
  }
  stale_final_kernel<<<(b.R + 127) / 128, 128, 0, stream>>>(part, b.R, kv.L, M, err, err_rl);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
