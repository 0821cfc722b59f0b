// Value-norm side cache (Conduit Sec. 4.3 and App. C.2): ||V_t^(l)|| depends
// only on the cached content, so it can be computed once per token and layer
// when the cache is built, and the scoring pass then reads one fp32 per token
// and layer instead of the value rows.
//   vnorm[l][tg] = sqrt( sum_g sum_part ss_{l,g,part}(t) )
// The partial sums ss and the order they are added in are those of the
// scoring pass for the same cache (two 64-element halves per head for the
// tensor-core kernel, one warp-reduced row per head for the CUDA-core one),
// so the stored norm is bitwise the one the scoring pass computes from V.
//
// Rows are either every token of the batch (mode all) or the selected rows of
// a refresh (mode selection: request r's idx[idx_off[r] ..], after a scatter or
// exchange rewrote them).
#include "internal.cuh"

namespace conduit {
namespace {

struct RowSource {
  const int32_t* idx;      // NULL: row i is global token i
  const int32_t* idx_off;  // device [R+1] (selection mode)
  int64_t n_rows;
};

// Request, request-local token and global token row of row i.
__device__ __forceinline__ void locate(const RowSource& src, const BatchDev& b, int64_t i, int& r,
                                       int& t, int64_t& tg) {
  if (src.idx == nullptr) {
    tg = i;
    r = request_of(b.tok_off, b.R, i);
    t = int(i - b.tok_off[r]);
  } else {
    r = request_of(src.idx_off, b.R, i);
    t = src.idx[i];
    tg = int64_t(b.tok_off[r]) + t;
  }
}

// bf16, head_dim 128 (the tensor-core scoring kernel's order). Each token
// has a group of S lanes (S = 2 Hkv rounded up to a power of two, at most 32);
// lane j of the group sums the squares of the 64-element half rows p = j,
// j + S, ... (p = 2 g + half), and the group's partials are added up in p
// order by shuffles, every lane of the warp taking part.
__global__ void __launch_bounds__(256) vnorm_halves_kernel(KvDev kv, BatchDev b, RowSource src,
                                                           int lanes_per_token, float* vnorm) {
  const int l = blockIdx.y;
  const int S = lanes_per_token, tpw = 32 / S;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = lane / S, j = lane % S;
  const int64_t i = (int64_t(blockIdx.x) * (blockDim.x >> 5) + warp) * tpw + grp;
  const bool live = i < src.n_rows;
  int r = 0, t = 0;
  int64_t tg = 0;
  if (live) locate(src, b, i, r, t, tg);
  const __nv_bfloat16* vb = static_cast<const __nv_bfloat16*>(kv.v);
  const int halves = 2 * kv.Hkv;
  float total = 0.f;
  for (int p0 = 0; p0 < halves; p0 += S) {  // warp-uniform
    const int p = p0 + j;
    float part = 0.f;
    if (live && p < halves) {
      const int64_t off = kv.row(l, p >> 1, r, tg, t) + (p & 1) * 64;  // half p & 1 of head p >> 1
      const uint4* row = reinterpret_cast<const uint4*>(vb + off);
      uint4 x[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) x[c] = __ldg(row + c);
      float sq[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < 8; ++c) sumsq_bf16_chunk(x[c], sq);
      part = sumsq_combine(sq);
    }
    for (int jj = 0; jj < S; ++jj) {
      const float v = __shfl_sync(0xffffffffu, part, grp * S + jj);
      if (p0 + jj < halves) total += v;
    }
  }
  if (live && j == 0) vnorm[int64_t(l) * kv.n_tot + tg] = sqrtf(total);
}

// Any other cache (fp32, or head_dim != 128): one warp per row, one
// warp-reduced sum per head, heads added in order.
template <typename T>
__global__ void __launch_bounds__(256) vnorm_rows_kernel(KvDev kv, BatchDev b, RowSource src,
                                                         float* vnorm) {
  const int l = blockIdx.y;
  const int64_t i = int64_t(blockIdx.x) * 8 + threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  if (i >= src.n_rows) return;
  int r, t;
  int64_t tg;
  locate(src, b, i, r, t, tg);
  const T* vb = static_cast<const T*>(kv.v);
  float total = 0.f;
  for (int g = 0; g < kv.Hkv; ++g) total += warp_row_sumsq(vb + kv.row(l, g, r, tg, t), kv.d, lane);
  if (lane == 0) vnorm[int64_t(l) * kv.n_tot + tg] = sqrtf(total);
}

}  // namespace

cudaError_t launch_value_norms(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                               const int32_t* idx_off_dev, int64_t n_rows, float* vnorm,
                               cudaStream_t stream) {
  if (n_rows == 0) return cudaSuccess;
  const RowSource src{idx, idx_off_dev, n_rows};
  if (score_tc_supported(kv)) {
    int S = 2;
    while (S < 2 * kv.Hkv && S < 32) S *= 2;
    const int64_t per_block = 8 * (32 / S);  // tokens of a 256-thread block
    const dim3 grid(unsigned((n_rows + per_block - 1) / per_block), kv.L);
    vnorm_halves_kernel<<<grid, 256, 0, stream>>>(kv, b, src, S, vnorm);
  } else {
    const dim3 grid(unsigned((n_rows + 7) / 8), kv.L);
    if (kv.dtype == CONDUIT_BF16)
      vnorm_rows_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(kv, b, src, vnorm);
    else
      vnorm_rows_kernel<float><<<grid, 256, 0, stream>>>(kv, b, src, vnorm);
  }
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
