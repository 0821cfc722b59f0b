// Tensor-core causal refresh attention for bf16 caches with head_dim 128
// (selective recompute, Conduit Sec. 3.1 / 4.3):
//   out[l][i][h] = sum_{j <= p_i} softmax_j(<q[l][i][h], K'[l][h/G][j]> / sqrt(d)) V'[l][h/G][j]
//
// One CTA owns a block of 128 query rows of one (layer, KV head, request):
// floor(128/G) consecutive selected rows times the G query heads that share
// the KV head. Keys stream in tiles of 64 through a two-stage TMA ring:
//   S = Q K_tile^T          tcgen05, rows as M, into TMEM columns [0, 64)
//   softmax                 each thread owns one row: causal mask j <= p_i,
//                           running max kept lazily (O and the row sum are
//                           rescaled only when the max grows by 2^8), P in bf16
//                           written into the K half of the tile's stage
//   O += P V_tile           tcgen05 with V as an MN-major operand, TMEM
//                           columns [64, 192)
// then O / rowsum is written in bf16. Rows are sorted by position, so a
// block needs keys up to its last row's position only. Two CTAs fit an SM
// (96 KB shared, 256 TMEM columns each), so one CTA's softmax overlaps the
// other's MMAs. Every wait is bounded (CONDUIT_FLAG_TIMEOUT on expiry).
#include <cuda.h>

#include "internal.cuh"
#include "tc_common.cuh"

namespace conduit {
namespace {

constexpr int kD = 128;
constexpr int kKT = 64;                          // keys per tile
constexpr int kRows = 128;
constexpr int kThreads = 128;
constexpr uint32_t kQHalf = kRows * 128;         // 16 KB: one 64-dim half of the query tile
constexpr uint32_t kKVHalf = kKT * 128;          // 8 KB: one 64-dim half of a K or V tile
constexpr uint32_t kStage = 4 * kKVHalf;         // K (2 halves) then V (2 halves)
constexpr uint32_t kSmem = 1024 + 2 * kQHalf + 2 * kStage + 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kOCol = 64;
constexpr float kRescaleLog2 = 8.f;

struct RefArgs {
  KvDev kv;
  BatchDev b;
  const int32_t* idx;
  const int32_t* idx_off;
  const __nv_bfloat16* q_rows;
  __nv_bfloat16* out;
  int32_t n_sel;
  int32_t rows_per_block;  // selected rows per CTA, floor(128 / G)
  int32_t n_blocks;        // CTA blocks per (layer, KV head)
  float scale_log2;
  int32_t* status;
};

__device__ __forceinline__ void load_kv_tile(const RefArgs& a, const CUtensorMap* kmap,
                                             const CUtensorMap* vmap, uint8_t* st, uint64_t* bar,
                                             int l, int g, int r, int t0, int N, int j0) {
  const KvDev& kv = a.kv;
  tc::mbar_arrive_expect_tx(bar, kStage);
  if (kv.page_size == 0) {
    const int32_t y = int32_t((int64_t(l) * kv.Hkv + g) * kv.n_tot + t0 + j0);
    tc::tma_load_2d(st, kmap, bar, 0, y);
    tc::tma_load_2d(st + kKVHalf, kmap, bar, 64, y);
    tc::tma_load_2d(st + 2 * kKVHalf, vmap, bar, 0, y);
    tc::tma_load_2d(st + 3 * kKVHalf, vmap, bar, 64, y);
  } else {
    const int ps = kv.page_size;
    const int last_page = (N - 1) / ps;
    for (int i = 0; i < kKT / ps; ++i) {
      const int lp = min((j0 + i * ps) / ps, last_page);
      const int page = kv.page_table[int64_t(r) * kv.max_pages + lp];
      const int32_t y = int32_t(((int64_t(l) * kv.num_pages + page) * kv.Hkv + g) * ps);
      tc::tma_load_2d(st + i * ps * 128, kmap, bar, 0, y);
      tc::tma_load_2d(st + kKVHalf + i * ps * 128, kmap, bar, 64, y);
      tc::tma_load_2d(st + 2 * kKVHalf + i * ps * 128, vmap, bar, 0, y);
      tc::tma_load_2d(st + 3 * kKVHalf + i * ps * 128, vmap, bar, 64, y);
    }
  }
}

__global__ void __launch_bounds__(kThreads, 2)
    refresh_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                      const __grid_constant__ RefArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_s = base;                       // [2][128 rows][128 B]
  uint8_t* stages = base + 2 * kQHalf;       // [2][K half0, K half1, V half0, V half1]
  uint64_t* full = reinterpret_cast<uint64_t*>(stages + 2 * kStage);  // [2]
  uint64_t* s_bar = full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(s_bar + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int l = blockIdx.z, g = blockIdx.y;
  const KvDev& kv = a.kv;
  const int G = kv.G, Hq = kv.Hq;

  // block -> (request, first selected row); larger positions first
  int blk = a.n_blocks - 1 - int(blockIdx.x);
  int r = 0, i0 = -1, cnt = 0;
  for (int rr = 0; rr < a.b.R; ++rr) {
    const int k0 = a.idx_off[rr], kr = a.idx_off[rr + 1] - k0;
    const int nb = (kr + a.rows_per_block - 1) / a.rows_per_block;
    if (blk < nb) {
      r = rr;
      i0 = k0 + blk * a.rows_per_block;
      cnt = min(a.rows_per_block, kr - blk * a.rows_per_block);
      break;
    }
    blk -= nb;
  }
  if (i0 < 0) return;
  const int t0 = a.b.tok_off[r], N = a.b.tok_off[r + 1] - t0;
  const int p_max = min(a.idx[i0 + cnt - 1], N - 1);
  if (p_max < 0) return;
  const int ntiles = p_max / kKT + 1;

  // this thread's row: selected row i0 + row / G, query head g*G + row % G
  const int row = warp * 32 + lane;
  const bool row_ok = row < cnt * G;
  const int i_row = i0 + (row_ok ? row / G : 0);
  const int h_row = g * G + (row_ok ? row % G : 0);
  int p_row = row_ok ? a.idx[i_row] : -1;
  if (p_row >= N) p_row = -1;

  if (tid == 0) {
    tc::mbar_init(&full[0], 1);
    tc::mbar_init(&full[1], 1);
    tc::mbar_init(s_bar, 1);
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
    tc::prefetch_tensormap(&vmap);
  }
  if (warp == 0) tc::tmem_alloc(tmem_slot, kTmemCols);
  // query tile: rows as above, zero beyond cnt * G
  for (int x = tid; x < kRows * 16; x += kThreads) {
    const int rr = x >> 4, ch = x & 15;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (rr < cnt * G) {
      const int ii = i0 + rr / G, hh = g * G + rr % G;
      val = *reinterpret_cast<const uint4*>(a.q_rows + ((int64_t(l) * a.n_sel + ii) * Hq + hh) * kD + ch * 8);
    }
    *reinterpret_cast<uint4*>(q_s + (ch >> 3) * kQHalf + tc::sw128_offset(rr, ch & 7)) = val;
  }
  tc::fence_proxy_async_smem();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t lane_base = uint32_t(warp * 32) << 16;

  bool ok = true;
  int32_t site = 0;
  if (tid == 0) {
    load_kv_tile(a, &kmap, &vmap, stages, &full[0], l, g, r, t0, N, 0);
    if (ntiles > 1) load_kv_tile(a, &kmap, &vmap, stages + kStage, &full[1], l, g, r, t0, N, kKT);
  }
  int loads_issued = min(ntiles, 2);

  float m_ref = -INFINITY, lsum = 0.f;
  const uint32_t q_addr = tc::smem_u32(q_s);
  const uint32_t idesc_s = tc::idesc_bf16(kRows, kKT);
  const uint32_t idesc_o = tc::idesc_bf16(kRows, kD, /*b_mn_major=*/true);
  int t = 0;
  for (; t < ntiles; ++t) {
    const int st = t & 1;
    uint8_t* stage = stages + st * kStage;
    const uint32_t k_addr = tc::smem_u32(stage);
    int issued = 1;
    if (tid == 0) {
      if (!tc::mbar_wait(&full[st], (t >> 1) & 1)) {
        issued = 0;
      } else {
        tc::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk & 3) * 32;
          tc::mma_bf16(tmem, tc::desc_sw128(q_addr + (kk >> 2) * kQHalf + off),
                       tc::desc_sw128(k_addr + (kk >> 2) * kKVHalf + off), idesc_s, kk > 0);
        }
        tc::mma_commit(s_bar);
      }
    }
    if (!__syncthreads_and(issued)) { ok = false; site = tc::kSiteLoad; break; }
    // S of tile t ready, and every earlier MMA (the P.V of tile t-1) is complete
    if (!__syncthreads_and(tc::mbar_wait(s_bar, t & 1))) { ok = false; site = tc::kSiteMma; break; }
    tc::tc_fence_after();
    if (tid == 0 && t >= 1 && t + 1 < ntiles) {  // stage of tile t-1 is free again
      load_kv_tile(a, &kmap, &vmap, stages + ((t + 1) & 1) * kStage, &full[(t + 1) & 1], l, g, r, t0,
                   N, (t + 1) * kKT);
    }
    if (t >= 1 && t + 1 < ntiles) ++loads_issued;

    float sv[2][32];
    tc::tmem_ld32(tmem + lane_base + 0, sv[0]);
    tc::tmem_ld32(tmem + lane_base + 32, sv[1]);
    const int j0 = t * kKT;
    float tmax = -INFINITY;
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2)
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float x = (j0 + h2 * 32 + i <= p_row) ? sv[h2][i] * a.scale_log2 : -INFINITY;
        sv[h2][i] = x;
        tmax = fmaxf(tmax, x);
      }
    // Lazy rescale of this row's O and sum when its max grew by more than 2^8.
    // tcgen05.ld / st are warp-collective, so the TMEM pass runs for the whole
    // warp whenever any lane needs it; lanes that do not rescale use alpha = 1.
    const bool need = tmax > m_ref + kRescaleLog2 || (m_ref == -INFINITY && tmax != -INFINITY);
    const float alpha = need ? exp2f(m_ref - tmax) : 1.f;  // 0 when m_ref is -inf
    if (__any_sync(0xffffffffu, need) && t > 0) {
      for (int c = 0; c < kD; c += 32) {
        float o[32];
        tc::tmem_ld32(tmem + lane_base + kOCol + c, o);
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] *= alpha;
        tc::tmem_st32(tmem + lane_base + kOCol + c, o);
      }
    }
    if (need) {
      lsum *= alpha;
      m_ref = tmax;
    }
    // P = 2^(x - m_ref) in bf16 into the K half of this stage (K is consumed)
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
      for (int c8 = 0; c8 < 4; ++c8) {
        uint32_t w4[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float p0 = (m_ref == -INFINITY) ? 0.f : exp2f(sv[h2][c8 * 8 + 2 * u] - m_ref);
          const float p1 = (m_ref == -INFINITY) ? 0.f : exp2f(sv[h2][c8 * 8 + 2 * u + 1] - m_ref);
          lsum += p0 + p1;
          __nv_bfloat162 pr = __floats2bfloat162_rn(p0, p1);
          w4[u] = *reinterpret_cast<uint32_t*>(&pr);
        }
        const int chunk = h2 * 4 + c8;  // 16-byte chunk of the 128-byte P row
        *reinterpret_cast<uint4*>(stage + tc::sw128_offset(row, chunk)) =
            make_uint4(w4[0], w4[1], w4[2], w4[3]);
      }
    }
    tc::fence_proxy_async_smem();
    tc::tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc::tc_fence_after();
      const uint32_t p_addr = k_addr;                       // P: [128 rows][64 keys] K-major
      const uint32_t v_addr = k_addr + 2 * kKVHalf;          // V: [64 keys][128 dims] MN-major
#pragma unroll
      for (int kk = 0; kk < kKT / 16; ++kk) {
        tc::mma_bf16(tmem + kOCol, tc::desc_sw128(p_addr + kk * 32),
                     tc::desc_sw128_mn(v_addr + kk * 2048, kKVHalf), idesc_o, t > 0 || kk > 0);
      }
    }
  }
  // final P.V -> O ready
  if (ok) {
    if (tid == 0) tc::mma_commit(s_bar);
    if (!__syncthreads_and(tc::mbar_wait(s_bar, ntiles & 1))) { ok = false; site = tc::kSiteFinal; }
  }
  if (ok) {
    tc::tc_fence_after();
    const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
    __nv_bfloat16* dst = a.out + ((int64_t(l) * a.n_sel + i_row) * Hq + h_row) * kD;
    for (int c = 0; c < kD; c += 32) {
      float o[32];
      tc::tmem_ld32(tmem + lane_base + kOCol + c, o);
      if (row_ok && p_row >= 0) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          uint32_t w4[4];
#pragma unroll
          for (int k2 = 0; k2 < 4; ++k2) {
            __nv_bfloat162 pr = __floats2bfloat162_rn(o[u * 8 + 2 * k2] * inv, o[u * 8 + 2 * k2 + 1] * inv);
            w4[k2] = *reinterpret_cast<uint32_t*>(&pr);
          }
          *reinterpret_cast<uint4*>(dst + c + u * 8) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
      }
    }
  } else {
    flag_status(a.status, CONDUIT_FLAG_TIMEOUT | site);
    if (tid == 0) {  // drain loads still in flight into this CTA's shared memory
      for (int tt = t; tt < loads_issued; ++tt) tc::mbar_wait(&full[tt & 1], (tt >> 1) & 1);
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, kTmemCols);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool make_map(CUtensorMap* m, const KvDev& kv, void* base) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {cuuint64_t(kD), 0};
  cuuint64_t strides[1] = {cuuint64_t(kD) * 2};
  cuuint32_t box[2] = {64, 0};
  cuuint32_t estr[2] = {1, 1};
  if (kv.page_size == 0) {
    dims[1] = cuuint64_t(kv.L) * kv.Hkv * kv.n_tot;
    box[1] = kKT;
  } else {
    dims[1] = cuuint64_t(kv.L) * kv.num_pages * kv.Hkv * kv.page_size;
    box[1] = kv.page_size;
  }
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool refresh_tc_supported(const KvDev& kv) {
  if (kv.dtype != CONDUIT_BF16 || kv.d != kD || kv.G > kRows) return false;
  if (kv.page_size != 0 && (kv.page_size % 8 != 0 || kKT % kv.page_size != 0)) return false;
  return true;
}

cudaError_t launch_refresh_tc(const KvDev& kv, const BatchDev& b, const int32_t* idx,
                              const int32_t* idx_off_dev, const int32_t* idx_off_host, int32_t n_sel,
                              const void* q_rows, void* out, int32_t* status, cudaStream_t stream) {
  if (n_sel == 0) return cudaSuccess;
  CUtensorMap kmap, vmap;
  if (!make_map(&kmap, kv, kv.k) || !make_map(&vmap, kv, kv.v)) return cudaErrorInvalidValue;
  RefArgs a{};
  a.kv = kv;
  a.b = b;
  a.idx = idx;
  a.idx_off = idx_off_dev;
  a.q_rows = static_cast<const __nv_bfloat16*>(q_rows);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.n_sel = n_sel;
  a.rows_per_block = kRows / kv.G;
  int blocks = 0;
  for (int r = 0; r < b.R; ++r) {
    const int kr = idx_off_host[r + 1] - idx_off_host[r];
    blocks += (kr + a.rows_per_block - 1) / a.rows_per_block;
  }
  a.n_blocks = blocks;
  a.scale_log2 = kLog2e / sqrtf(float(kD));
  a.status = status;
  if (blocks == 0) return cudaSuccess;
  cudaError_t err = cudaFuncSetAttribute(refresh_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         int(kSmem));
  if (err) return err;
  const dim3 grid(blocks, kv.Hkv, kv.L);
  refresh_tc_kernel<<<grid, kThreads, kSmem, stream>>>(kmap, vmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
