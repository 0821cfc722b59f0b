// Tensor-core scoring pass for bf16 caches with head_dim 128 (Conduit Eq. 6).
//
// Per slab (request r, scored layer l, KV head g) the logits are
// S = Q_g K_g^T over R = G*|Q| scoring rows and the request's N_r keys. Two
// persistent kernels share one work list of units (slab, token chunk):
//
//   rowstats_tc  D[rows x 128 tokens] = Q_rows . K_tile^T on tcgen05 (rows are
//                the MMA M dimension, so each thread owns one row): running
//                row max and sum of 2^((S - m) log2(e)/sqrt(d)) over the
//                chunk -> partial (m, Z) per row and chunk.
//   colsum_tc    D[128 tokens x rows] = K_tile . Q_rows^T (tokens are M, so
//                each thread owns one token): merges the chunk statistics
//                into log2-sum-exp per row, then sums 2^(x - lse) over the
//                rows -> pa[l][g][t], the group's share of Eq. 6.
//
// K tiles (128 tokens x 128 dims) arrive by TMA with 128-byte swizzle into a
// two-stage ring; scoring rows are staged once per unit by the threads in
// the same swizzled layout. One thread issues the TMA loads and the MMAs;
// accumulators live in TMEM (512 columns, double-buffered when a tile needs
// at most 256) and are read back with tcgen05.ld. Every wait is bounded; on
// timeout the kernel sets CONDUIT_FLAG_TIMEOUT, drains its copies and frees
// its TMEM.
#include <cuda.h>

#include "internal.cuh"
#include "tc_common.cuh"

namespace conduit {
namespace {

constexpr int kD = 128;
constexpr int kTile = 128;
constexpr int kStages = 2;
constexpr int kRowGroup = 512;
constexpr int kThreads = 128;
constexpr uint32_t kHalfQ = kRowGroup * 128;        // bytes of one 64-dim half of the row tile
constexpr uint32_t kQBytes = 2 * kHalfQ;            // 128 KB
constexpr uint32_t kHalfK = kTile * 128;            // 16 KB
constexpr uint32_t kStageBytes = 2 * kHalfK;        // 32 KB per K tile
constexpr uint32_t kSmemBytes = 1024 + kQBytes + kStages * kStageBytes + 256 + kRowGroup * 4;

struct TcArgs {
  KvDev kv;
  BatchDev b;
  const __nv_bfloat16* q;
  int32_t q_tot;
  int32_t chunk;        // tokens per unit (multiple of 128)
  int32_t nchunks_max;  // chunks per slab for the longest request
  int32_t n_units;
  int64_t total_rows;   // n_layers * Hq * Q_tot
  float scale_log2;     // log2(e) / sqrt(d)
  float2* part;         // [nchunks_max][total_rows] partial (max S, sum) per row
  float* pa;            // [n_layers][Hkv][n_tot]
  int32_t* status;
  LayerList layers;
};

struct Unit {
  int r, li, l, g, c, t0, N, q0, nq, R, tok0, tiles;
};

__device__ __forceinline__ bool decode_unit(const TcArgs& a, int u, Unit& w) {
  const int per_slab = a.nchunks_max;
  int slab = u / per_slab;
  w.c = u % per_slab;
  const int Hkv = a.kv.Hkv, nl = a.layers.n;
  w.g = slab % Hkv;
  slab /= Hkv;
  w.li = slab % nl;
  w.r = slab / nl;
  w.l = a.layers.ids[w.li];
  w.t0 = a.b.tok_off[w.r];
  w.N = a.b.tok_off[w.r + 1] - w.t0;
  w.q0 = a.b.q_off[w.r];
  w.nq = a.b.q_off[w.r + 1] - w.q0;
  w.R = a.kv.G * w.nq;
  w.tok0 = w.c * a.chunk;
  if (w.tok0 >= w.N || w.R == 0) return false;
  w.tiles = (min(a.chunk, w.N - w.tok0) + kTile - 1) / kTile;
  return true;
}

struct Smem {
  uint8_t* q;        // [2 halves][kRowGroup rows][128 B], 128-byte swizzle
  uint8_t* k;        // [kStages][2 halves][128 rows][128 B]
  uint64_t* full;    // [kStages]
  uint64_t* mma;     // [2]
  uint32_t* tmem_slot;
  float* lse;        // [kRowGroup]
  int32_t* pages;    // page ids of the current tile (paged caches)
};

__device__ __forceinline__ Smem carve(uint8_t* raw) {
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  Smem s;
  s.q = base;
  s.k = base + kQBytes;
  uint8_t* tail = s.k + kStages * kStageBytes;
  s.full = reinterpret_cast<uint64_t*>(tail);
  s.mma = s.full + kStages;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.mma + 2);
  s.pages = reinterpret_cast<int32_t*>(tail + 64);
  s.lse = reinterpret_cast<float*>(tail + 256);
  return s;
}

// Stage scoring rows [row0, row0 + nrows) of the unit's slab into the swizzled
// row tile; rows at or beyond R are zero.
__device__ __forceinline__ void stage_rows(const TcArgs& a, const Unit& w, uint8_t* q_s, int row0,
                                           int nrows) {
  const int Hq = a.kv.Hq, G = a.kv.G;
  for (int idx = threadIdx.x; idx < nrows * 16; idx += blockDim.x) {
    const int row = idx >> 4, ch = idx & 15;
    const int j = row0 + row;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (j < w.R) {
      const int h = w.g * G + j / w.nq, qi = j % w.nq;
      const __nv_bfloat16* src = a.q + ((int64_t(w.l) * Hq + h) * a.q_tot + w.q0 + qi) * kD + ch * 8;
      val = *reinterpret_cast<const uint4*>(src);
    }
    uint8_t* dst = q_s + (ch >> 3) * kHalfQ + tc::sw128_offset(row, ch & 7);
    *reinterpret_cast<uint4*>(dst) = val;
  }
}

// Issue the TMA loads of K tile `tile` of the unit into ring stage `stage`.
__device__ __forceinline__ void load_k_tile(const TcArgs& a, const CUtensorMap* kmap, const Unit& w,
                                            const Smem& s, int tile, int stage) {
  uint8_t* dst = s.k + stage * kStageBytes;
  uint64_t* bar = &s.full[stage];
  tc::mbar_arrive_expect_tx(bar, kStageBytes);
  const int tok = w.tok0 + tile * kTile;
  const KvDev& kv = a.kv;
  if (kv.page_size == 0) {
    const int32_t y = int32_t((int64_t(w.l) * kv.Hkv + w.g) * kv.n_tot + w.t0 + tok);
    tc::tma_load_2d(dst, kmap, bar, 0, y);
    tc::tma_load_2d(dst + kHalfK, kmap, bar, 64, y);
  } else {
    const int ps = kv.page_size;
    const int last_page = (w.N - 1) / ps;
    for (int i = 0; i < kTile / ps; ++i) {
      const int lp = min((tok + i * ps) / ps, last_page);  // tail pages repeat the last one (masked)
      const int page = kv.page_table[int64_t(w.r) * kv.max_pages + lp];
      const int32_t y = int32_t(((int64_t(w.l) * kv.num_pages + page) * kv.Hkv + w.g) * ps);
      tc::tma_load_2d(dst + i * ps * 128, kmap, bar, 0, y);
      tc::tma_load_2d(dst + kHalfK + i * ps * 128, kmap, bar, 64, y);
    }
  }
}

// Row statistics: one unit = (slab, chunk); rows as M.
__global__ void __launch_bounds__(kThreads, 1)
    rowstats_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const Smem s = carve(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) tc::mbar_init(&s.full[i], 1);
    tc::mbar_init(&s.mma[0], 1);
    tc::mbar_init(&s.mma[1], 1);
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
  }
  if (warp == 0) tc::tmem_alloc(s.tmem_slot, 512);
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *s.tmem_slot;
  const uint32_t lane_base = uint32_t(warp * 32) << 16;

  uint32_t ld_seq = 0;          // K tiles issued so far (thread 0's view == everyone's)
  uint32_t mma_phase[2] = {0u, 0u};
  bool ok = true;
  uint32_t pending_lo = 0, pending_hi = 0;  // tiles issued but not yet consumed (for draining)

  for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
    Unit w;
    if (!decode_unit(a, u, w)) continue;
    for (int rg0 = 0; rg0 < w.R && ok; rg0 += kRowGroup) {
      const int rows = min(kRowGroup, w.R - rg0);
      const int nrb = (rows + 127) / 128;
      const int nbuf = nrb <= 2 ? 2 : 1;
      __syncthreads();
      stage_rows(a, w, s.q, rg0, nrb * 128);
      tc::fence_proxy_async_smem();
      __syncthreads();
      const uint32_t base = ld_seq;
      const int T = w.tiles;
      if (tid == 0) {
        for (int t = 0; t < min(kStages, T); ++t) load_k_tile(a, &kmap, w, s, t, (base + t) % kStages);
      }
      ld_seq += min(kStages, T);
      pending_lo = base;
      pending_hi = ld_seq;

      auto issue_mma = [&](int t, int buf) {
        const uint32_t seq = base + t;
        const int st = seq % kStages;
        if (!tc::mbar_wait(&s.full[st], (seq / kStages) & 1)) return false;
        tc::tc_fence_after();
        const uint32_t kb = tc::smem_u32(s.k + st * kStageBytes);
        const uint32_t qb = tc::smem_u32(s.q);
        const uint32_t idesc = tc::idesc_bf16(128, kTile);
        for (int rb = 0; rb < nrb; ++rb) {
          const uint32_t d = tmem + uint32_t(buf * nrb * 128 + rb * 128);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (kk >> 2) * 0 + (kk & 3) * 32;
            const uint64_t adesc = tc::desc_sw128(qb + (kk >> 2) * kHalfQ + rb * 128 * 128 + off);
            const uint64_t bdesc = tc::desc_sw128(kb + (kk >> 2) * kHalfK + off);
            tc::mma_bf16(d, adesc, bdesc, idesc, kk > 0);
          }
        }
        tc::mma_commit(&s.mma[buf]);
        return true;
      };

      int mma_ok = 1;
      if (tid == 0) mma_ok = issue_mma(0, 0);
      float m[4], z[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        m[i] = -INFINITY;
        z[i] = 0.f;
      }
      for (int t = 0; t < T; ++t) {
        const int buf = nbuf == 2 ? (t & 1) : 0;
        if (!__syncthreads_and(mma_ok)) { ok = false; break; }
        if (!tc::mbar_wait(&s.mma[buf], mma_phase[buf])) ok = false;
        mma_phase[buf] ^= 1u;
        if (!__syncthreads_and(ok)) { ok = false; break; }
        tc::tc_fence_after();
        if (tid == 0) {
          if (t + kStages < T) {
            load_k_tile(a, &kmap, w, s, t + kStages, (base + t + kStages) % kStages);
          }
          if (nbuf == 2 && t + 1 < T) mma_ok = issue_mma(t + 1, buf ^ 1);
        }
        if (t + kStages < T) ++ld_seq;
        pending_lo = base + t + 1;
        pending_hi = ld_seq;
        // epilogue: this thread's rows are rb*128 + warp*32 + lane
        const int tok_base = w.tok0 + t * kTile;
        for (int rb = 0; rb < nrb; ++rb) {
          for (int cc = 0; cc < 4; ++cc) {
            float v[32];
            tc::tmem_ld32(tmem + lane_base + uint32_t(buf * nrb * 128 + rb * 128 + cc * 32), v);
            const int tok = tok_base + cc * 32;
            float cmax = -INFINITY;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              if (tok + i >= w.N) v[i] = -INFINITY;
              cmax = fmaxf(cmax, v[i]);
            }
            float mr = m[0], zr = z[0];
            if (rb == 1) { mr = m[1]; zr = z[1]; }
            if (rb == 2) { mr = m[2]; zr = z[2]; }
            if (rb == 3) { mr = m[3]; zr = z[3]; }
            const float mn = fmaxf(mr, cmax);
            if (mn != -INFINITY) {
              const float nb = -mn * a.scale_log2;
              float acc = 0.f;
#pragma unroll
              for (int i = 0; i < 32; ++i) acc += exp2f(fmaf(v[i], a.scale_log2, nb));
              zr = zr * exp2f((mr - mn) * a.scale_log2) + acc;
              mr = mn;
            }
            if (rb == 0) { m[0] = mr; z[0] = zr; }
            if (rb == 1) { m[1] = mr; z[1] = zr; }
            if (rb == 2) { m[2] = mr; z[2] = zr; }
            if (rb == 3) { m[3] = mr; z[3] = zr; }
          }
        }
        tc::tc_fence_before();
        __syncthreads();
        if (tid == 0 && nbuf == 1 && t + 1 < T) mma_ok = issue_mma(t + 1, 0);
      }
      if (!ok) break;
      const int64_t srow0 = (int64_t(w.li) * a.kv.Hkv + w.g) * a.kv.G * a.q_tot + int64_t(a.kv.G) * w.q0;
      for (int rb = 0; rb < nrb; ++rb) {
        const int j = rg0 + rb * 128 + warp * 32 + lane;
        if (j < w.R) {
          float mr = rb == 0 ? m[0] : rb == 1 ? m[1] : rb == 2 ? m[2] : m[3];
          float zr = rb == 0 ? z[0] : rb == 1 ? z[1] : rb == 2 ? z[2] : z[3];
          a.part[int64_t(w.c) * a.total_rows + srow0 + j] = make_float2(mr, zr);
        }
      }
    }
  }
  if (!ok) {
    flag_status(a.status, CONDUIT_FLAG_TIMEOUT);
    if (tid == 0) {  // drain TMA copies still in flight into this CTA's shared memory
      for (uint32_t seq = pending_lo; seq < pending_hi; ++seq)
        tc::mbar_wait(&s.full[seq % kStages], (seq / kStages) & 1);
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// Column sums: one unit = (slab, chunk); tokens as M.
__global__ void __launch_bounds__(kThreads, 1)
    colsum_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const Smem s = carve(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) tc::mbar_init(&s.full[i], 1);
    tc::mbar_init(&s.mma[0], 1);
    tc::mbar_init(&s.mma[1], 1);
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
  }
  if (warp == 0) tc::tmem_alloc(s.tmem_slot, 512);
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *s.tmem_slot;
  const uint32_t lane_base = uint32_t(warp * 32) << 16;

  uint32_t ld_seq = 0;
  uint32_t mma_phase[2] = {0u, 0u};
  bool ok = true;
  uint32_t pending_lo = 0, pending_hi = 0;

  for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
    Unit w;
    if (!decode_unit(a, u, w)) continue;
    const int nch = (w.N + a.chunk - 1) / a.chunk;
    const int64_t srow0 = (int64_t(w.li) * a.kv.Hkv + w.g) * a.kv.G * a.q_tot + int64_t(a.kv.G) * w.q0;
    float* pa_out = a.pa + (int64_t(w.li) * a.kv.Hkv + w.g) * a.kv.n_tot + w.t0;
    for (int rg0 = 0; rg0 < w.R && ok; rg0 += kRowGroup) {
      const int rows = min(kRowGroup, w.R - rg0);
      const int ncols = (rows + 15) & ~15;
      const int nbuf = ncols <= 256 ? 2 : 1;
      __syncthreads();
      // log2-sum-exp of each row from the chunk statistics of rowstats_tc
      for (int j = tid; j < rows; j += blockDim.x) {
        float M = -INFINITY;
        for (int c = 0; c < nch; ++c) M = fmaxf(M, a.part[int64_t(c) * a.total_rows + srow0 + rg0 + j].x);
        float Z = 0.f;
        for (int c = 0; c < nch; ++c) {
          const float2 st = a.part[int64_t(c) * a.total_rows + srow0 + rg0 + j];
          Z += st.y * exp2f((st.x - M) * a.scale_log2);
        }
        s.lse[j] = M * a.scale_log2 + log2f(Z);
      }
      stage_rows(a, w, s.q, rg0, ncols);
      tc::fence_proxy_async_smem();
      __syncthreads();
      const uint32_t base = ld_seq;
      const int T = w.tiles;
      if (tid == 0) {
        for (int t = 0; t < min(kStages, T); ++t) load_k_tile(a, &kmap, w, s, t, (base + t) % kStages);
      }
      ld_seq += min(kStages, T);
      pending_lo = base;
      pending_hi = ld_seq;

      auto issue_mma = [&](int t, int buf) {
        const uint32_t seq = base + t;
        const int st = seq % kStages;
        if (!tc::mbar_wait(&s.full[st], (seq / kStages) & 1)) return false;
        tc::tc_fence_after();
        const uint32_t kb = tc::smem_u32(s.k + st * kStageBytes);
        const uint32_t qb = tc::smem_u32(s.q);
        for (int n0 = 0; n0 < ncols; n0 += 256) {
          const int nn = min(256, ncols - n0);
          const uint32_t idesc = tc::idesc_bf16(128, nn);
          const uint32_t d = tmem + uint32_t(buf * 256 + n0);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            const uint64_t adesc = tc::desc_sw128(kb + (kk >> 2) * kHalfK + off);
            const uint64_t bdesc = tc::desc_sw128(qb + (kk >> 2) * kHalfQ + n0 * 128 + off);
            tc::mma_bf16(d, adesc, bdesc, idesc, kk > 0);
          }
        }
        tc::mma_commit(&s.mma[buf]);
        return true;
      };

      int mma_ok = 1;
      if (tid == 0) mma_ok = issue_mma(0, 0);
      for (int t = 0; t < T; ++t) {
        const int buf = nbuf == 2 ? (t & 1) : 0;
        if (!__syncthreads_and(mma_ok)) { ok = false; break; }
        if (!tc::mbar_wait(&s.mma[buf], mma_phase[buf])) ok = false;
        mma_phase[buf] ^= 1u;
        if (!__syncthreads_and(ok)) { ok = false; break; }
        tc::tc_fence_after();
        if (tid == 0) {
          if (t + kStages < T) load_k_tile(a, &kmap, w, s, t + kStages, (base + t + kStages) % kStages);
          if (nbuf == 2 && t + 1 < T) mma_ok = issue_mma(t + 1, buf ^ 1);
        }
        if (t + kStages < T) ++ld_seq;
        pending_lo = base + t + 1;
        pending_hi = ld_seq;
        // epilogue: this thread's token is warp*32 + lane of the tile
        float acc = 0.f;
        const int nchunk32 = (rows + 31) / 32;
        for (int cc = 0; cc < nchunk32; ++cc) {
          float v[32];
          tc::tmem_ld32(tmem + lane_base + uint32_t(buf * 256 + cc * 32), v);
          const int jb = cc * 32;
          if (jb + 32 <= rows) {
#pragma unroll
            for (int i = 0; i < 32; ++i) acc += exp2f(fmaf(v[i], a.scale_log2, -s.lse[jb + i]));
          } else {
            for (int i = 0; i < rows - jb; ++i) acc += exp2f(fmaf(v[i], a.scale_log2, -s.lse[jb + i]));
          }
        }
        const int tok = w.tok0 + t * kTile + warp * 32 + lane;
        if (tok < w.N) pa_out[tok] = rg0 == 0 ? acc : pa_out[tok] + acc;
        tc::tc_fence_before();
        __syncthreads();
        if (tid == 0 && nbuf == 1 && t + 1 < T) mma_ok = issue_mma(t + 1, 0);
      }
    }
  }
  if (!ok) {
    flag_status(a.status, CONDUIT_FLAG_TIMEOUT);
    if (tid == 0) {
      for (uint32_t seq = pending_lo; seq < pending_hi; ++seq)
        tc::mbar_wait(&s.full[seq % kStages], (seq / kStages) & 1);
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
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

}  // namespace

bool score_tc_supported(const KvDev& kv) {
  if (kv.dtype != CONDUIT_BF16 || kv.d != kD) return false;
  if (kv.page_size != 0 && (kv.page_size % 8 != 0 || kTile % kv.page_size != 0)) return false;
  return true;
}

int score_tc_chunk(int R, const int32_t* tok_off_host, int n_layers, int Hkv) {
  // largest chunk that still gives at least two units per SM of a 152-SM part
  for (int chunk = 1024; chunk > kTile; chunk >>= 1) {
    int64_t units = 0;
    for (int r = 0; r < R; ++r)
      units += int64_t(n_layers) * Hkv * ((tok_off_host[r + 1] - tok_off_host[r] + chunk - 1) / chunk);
    if (units >= 304) return chunk;
  }
  return kTile;
}

size_t score_tc_part_bytes(int chunk, int max_tokens, int64_t total_rows) {
  const int nch = (max_tokens + chunk - 1) / chunk;
  return size_t(nch) * size_t(total_rows) * sizeof(float2);
}

cudaError_t launch_score_tc(const KvDev& kv, const BatchDev& b, const void* q, int32_t q_tot,
                            const LayerList& layers, int max_tokens, int chunk, float2* part,
                            float* pa, int32_t* status, cudaStream_t stream) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap kmap;
  cuuint64_t dims[2];
  cuuint64_t strides[1] = {cuuint64_t(kD) * 2};
  cuuint32_t box[2];
  cuuint32_t estr[2] = {1, 1};
  if (kv.page_size == 0) {
    dims[0] = kD;
    dims[1] = cuuint64_t(kv.L) * kv.Hkv * kv.n_tot;
    box[0] = 64;
    box[1] = kTile;
  } else {
    dims[0] = kD;
    dims[1] = cuuint64_t(kv.L) * kv.num_pages * kv.Hkv * kv.page_size;
    box[0] = 64;
    box[1] = kv.page_size;
  }
  CUresult cr = enc(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, kv.k, dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return cudaErrorInvalidValue;

  TcArgs a{};
  a.kv = kv;
  a.b = b;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.q_tot = q_tot;
  a.chunk = chunk;
  a.nchunks_max = (max_tokens + chunk - 1) / chunk;
  a.n_units = b.R * layers.n * kv.Hkv * a.nchunks_max;
  a.total_rows = int64_t(layers.n) * kv.Hq * q_tot;
  a.scale_log2 = kLog2e / sqrtf(float(kD));
  a.part = part;
  a.pa = pa;
  a.status = status;
  a.layers = layers;

  int dev = 0, sms = 0;
  cudaError_t err;
  if ((err = cudaGetDevice(&dev))) return err;
  if ((err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))) return err;
  const int grid = std::max(1, std::min(a.n_units, sms));
  if ((err = cudaFuncSetAttribute(rowstats_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  int(kSmemBytes))))
    return err;
  if ((err = cudaFuncSetAttribute(colsum_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  int(kSmemBytes))))
    return err;
  rowstats_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(kmap, a);
  if ((err = cudaGetLastError())) return err;
  colsum_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(kmap, a);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace conduit
