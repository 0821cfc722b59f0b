// Tensor-core causal refresh attention for bf16 caches with head_dim 128
// (selective recompute, Conduit Sec. 3.1 / 4.3):
//   out[l][i][h] = sum_{j <= p_i} softmax_j(<q[l][i][h], K'[l][h/G][j]> / sqrt(d)) V'[l][h/G][j]
//
// One CTA owns up to two query tiles of 128 rows of one (layer, KV head,
// request); a tile holds floor(128/G) consecutive selected rows times the G
// query heads that share the KV head, and both tiles share every K/V tile.
// Keys stream in tiles of 64. Roles (320 threads):
//   warp 0     one thread issues TMA loads of K and V tiles into two
//              three-stage rings (K frees after both S, V after both P.V)
//   warp 1     one thread issues tcgen05 MMAs: per query tile, S(t) = Q K(t)^T
//              into one of two TMEM S buffers and O += P(t) V(t); S(t+2) is
//              issued right after P.V(t), so softmax overlaps tensor work
//   warps 2-5, 6-9   softmax of tile 0 and tile 1: stage the query rows, then
//              per key tile read S(t) (one row per thread), apply the causal
//              mask j <= p_i, keep a lazy running max (O and the row sum are
//              rescaled only when the max grows by 2^8; warp-uniform, since
//              tcgen05.ld/st are warp-collective), write P(t) in bf16 to one
//              of two shared buffers, and finally write O / rowsum in bf16
// TMEM: tile q uses columns [256q, 256q + 128) for its two S buffers and
// [256q + 128, 256q + 256) for O. Rows are sorted by position, so a CTA needs
// keys up to its last row's position only. Every wait is bounded by one
// second; a role that gives up raises an abort flag the others watch, the
// kernel sets CONDUIT_FLAG_TIMEOUT, drains its copies and MMAs, frees TMEM.
#include <cuda.h>

#include "internal.cuh"
#include "tc_common.cuh"

namespace conduit {
namespace {

constexpr int kD = 128;
constexpr int kKT = 64;                          // keys per tile
constexpr int kRows = 128;                       // rows per query tile
constexpr int kTiles = 2;                        // query tiles per CTA
constexpr int kSoftThreads = 128;
constexpr int kThreads = 64 + kTiles * kSoftThreads;
constexpr int kStages = 3;
constexpr uint32_t kQHalf = kRows * 128;         // 16 KB: one 64-dim half of a query tile
constexpr uint32_t kQBytes = 2 * kQHalf;         // 32 KB
constexpr uint32_t kTileHalf = kKT * 128;        // 8 KB: one 64-dim half of a K or V tile
constexpr uint32_t kTileBytes = 2 * kTileHalf;   // 16 KB
constexpr uint32_t kPBytes = kRows * 128;        // 16 KB: 128 rows x 64 keys
constexpr uint32_t kSmem =
    1024 + kTiles * kQBytes + 2 * kStages * kTileBytes + kTiles * 2 * kPBytes + 512;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTileCols = 256;              // TMEM columns per query tile
constexpr uint32_t kOCol = 128;                  // O offset inside a tile's columns
constexpr float kRescaleLog2 = 8.f;

struct RefArgs {
  KvDev kv;
  BatchDev b;
  const int32_t* idx;
  const int32_t* idx_off;
  const __nv_bfloat16* q_rows;
  __nv_bfloat16* out;
  int32_t n_sel;
  int32_t rows_per_tile;   // selected rows per query tile, floor(128 / G)
  int32_t n_blocks;        // CTAs per (layer, KV head)
  float scale_log2;
  int32_t* status;
};

struct Smem {
  uint8_t* q;        // [kTiles][2 halves][128 rows][128 B]
  uint8_t* k;        // [kStages][2 halves][64 keys][128 B]
  uint8_t* v;        // [kStages][2 halves][64 keys][128 B]
  uint8_t* p;        // [kTiles][2][128 rows][128 B]
  uint64_t *kfull, *kempty, *vfull, *vempty;  // [kStages] each
  uint64_t *sfull, *pfull, *pempty;           // [kTiles][2] each
  uint64_t *obar;                             // [kTiles]
  uint64_t *qready, *mdone;
  uint32_t* tmem_slot;
  volatile int* abort;
  uint32_t* counters;  // [0] K loads, [1] V loads, [2] K consumed, [3] V consumed
};

__device__ __forceinline__ Smem carve(uint8_t* raw) {
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  Smem s;
  s.q = base;
  s.k = s.q + kTiles * kQBytes;
  s.v = s.k + kStages * kTileBytes;
  s.p = s.v + kStages * kTileBytes;
  uint64_t* bar = reinterpret_cast<uint64_t*>(s.p + kTiles * 2 * kPBytes);
  s.kfull = bar;
  s.kempty = bar + kStages;
  s.vfull = bar + 2 * kStages;
  s.vempty = bar + 3 * kStages;
  s.sfull = bar + 4 * kStages;
  s.pfull = s.sfull + 2 * kTiles;
  s.pempty = s.pfull + 2 * kTiles;
  s.obar = s.pempty + 2 * kTiles;
  s.qready = s.obar + kTiles;
  s.mdone = s.qready + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.mdone + 1);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  s.counters = reinterpret_cast<uint32_t*>(s.tmem_slot + 2);
  return s;
}

__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (tc::mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = tc::globaltimer_ns();
  for (uint32_t i = 1; i < tc::kSpinLimit; ++i) {
    if (tc::mbar_try_wait(bar, parity)) return true;
    if ((i & 7u) == 0 && (*abort || tc::globaltimer_ns() - t0 > tc::kWaitNs)) return false;
  }
  return false;
}

__device__ __forceinline__ void raise_abort(const RefArgs& a, const Smem& s, int32_t site) {
  if (!*s.abort) flag_status(a.status, CONDUIT_FLAG_TIMEOUT | site);
  *s.abort = 1;
}

// TMA of the 64-key tile starting at request-local key j0 (one 64-dim half per box).
__device__ __forceinline__ void load_tile(const RefArgs& a, const CUtensorMap* map, uint8_t* dst,
                                          uint64_t* bar, int l, int g, int r, int t0, int N, int j0) {
  const KvDev& kv = a.kv;
  tc::mbar_arrive_expect_tx(bar, kTileBytes);
  if (kv.page_size == 0) {
    const int32_t y = int32_t((int64_t(l) * kv.Hkv + g) * kv.n_tot + t0 + j0);
    tc::tma_load_2d(dst, map, bar, 0, y);
    tc::tma_load_2d(dst + kTileHalf, map, bar, 64, y);
  } else {
    const int ps = kv.page_size;
    const int last_page = (N - 1) / ps;
    for (int i = 0; i < kKT / ps; ++i) {
      const int lp = min((j0 + i * ps) / ps, last_page);
      const int page = kv.page_table[int64_t(r) * kv.max_pages + lp];
      const int32_t y = int32_t(((int64_t(l) * kv.num_pages + page) * kv.Hkv + g) * ps);
      tc::tma_load_2d(dst + i * ps * 128, map, bar, 0, y);
      tc::tma_load_2d(dst + kTileHalf + i * ps * 128, map, bar, 64, y);
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    refresh_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                      const __grid_constant__ RefArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const Smem s = carve(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int l = blockIdx.z, g = blockIdx.y;
  const KvDev& kv = a.kv;
  const int G = kv.G, Hq = kv.Hq;

  // CTA -> (request, first selected row, row count); larger positions first
  const int span = kTiles * a.rows_per_tile;
  int blk = a.n_blocks - 1 - int(blockIdx.x);
  int r = 0, i0 = -1, cnt = 0;
  for (int rr = 0; rr < a.b.R; ++rr) {
    const int k0 = a.idx_off[rr], kr = a.idx_off[rr + 1] - k0;
    const int nb = (kr + span - 1) / span;
    if (blk < nb) {
      r = rr;
      i0 = k0 + blk * span;
      cnt = min(span, kr - blk * span);
      break;
    }
    blk -= nb;
  }
  if (i0 < 0) return;
  const int t0 = a.b.tok_off[r], N = a.b.tok_off[r + 1] - t0;
  const int p_max = min(a.idx[i0 + cnt - 1], N - 1);
  if (p_max < 0) return;
  const int ntiles = p_max / kKT + 1;
  const int nq = cnt > a.rows_per_tile ? 2 : 1;   // query tiles in use (CTA-uniform)

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      tc::mbar_init(&s.kfull[i], 1);
      tc::mbar_init(&s.kempty[i], 1);
      tc::mbar_init(&s.vfull[i], 1);
      tc::mbar_init(&s.vempty[i], 1);
    }
    for (int i = 0; i < 2 * kTiles; ++i) {
      tc::mbar_init(&s.sfull[i], 1);
      tc::mbar_init(&s.pfull[i], kSoftThreads);
      tc::mbar_init(&s.pempty[i], 1);
    }
    for (int i = 0; i < kTiles; ++i) tc::mbar_init(&s.obar[i], 1);
    tc::mbar_init(s.qready, kTiles);
    tc::mbar_init(s.mdone, 1);
    *s.abort = 0;
    for (int i = 0; i < 4; ++i) s.counters[i] = 0;
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
    tc::prefetch_tensormap(&vmap);
  }
  if (warp == 1) tc::tmem_alloc(s.tmem_slot, kTmemCols);
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *s.tmem_slot;

  if (warp == 0 && lane == 0) {
    // ---------------------------------------------------------------- loads
    uint32_t nk = 0, nv = 0;
    for (int t = 0; t < ntiles; ++t) {
      const int st = t % kStages;
      const uint32_t ph = ((t / kStages) & 1) ^ 1;
      if (!wait_or_abort(&s.kempty[st], ph, s.abort)) { raise_abort(a, s, tc::kSiteLoad); break; }
      load_tile(a, &kmap, s.k + st * kTileBytes, &s.kfull[st], l, g, r, t0, N, t * kKT);
      ++nk;
      if (!wait_or_abort(&s.vempty[st], ph, s.abort)) { raise_abort(a, s, tc::kSiteLoad); break; }
      load_tile(a, &vmap, s.v + st * kTileBytes, &s.vfull[st], l, g, r, t0, N, t * kKT);
      ++nv;
    }
    s.counters[0] = nk;
    s.counters[1] = nv;
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------------ MMA
    uint32_t ck = 0, cv = 0;
    const uint32_t idesc_s = tc::idesc_bf16(kRows, kKT);
    const uint32_t idesc_o = tc::idesc_bf16(kRows, kD, /*b_mn_major=*/true);
    auto issue_s = [&](int t) -> bool {  // S(t) of every query tile into its S buffer t & 1
      const int st = t % kStages;
      if (!wait_or_abort(&s.kfull[st], (t / kStages) & 1, s.abort)) return false;
      ++ck;
      tc::tc_fence_after();
      const uint32_t k_addr = tc::smem_u32(s.k + st * kTileBytes);
      for (int qi = 0; qi < nq; ++qi) {
        const uint32_t q_addr = tc::smem_u32(s.q + qi * kQBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk & 3) * 32;
          tc::mma_bf16(tmem + qi * kTileCols + uint32_t(t & 1) * kKT,
                       tc::desc_sw128(q_addr + (kk >> 2) * kQHalf + off),
                       tc::desc_sw128(k_addr + (kk >> 2) * kTileHalf + off), idesc_s, kk > 0);
        }
        tc::mma_commit(&s.sfull[qi * 2 + (t & 1)]);
      }
      tc::mma_commit(&s.kempty[st]);
      return true;
    };
    bool ok = wait_or_abort(s.qready, 0, s.abort);
    if (ok) ok = issue_s(0);
    if (ok && ntiles > 1) ok = issue_s(1);
    for (int t = 0; t < ntiles && ok; ++t) {
      const int b = t & 1, st = t % kStages;
      if (!wait_or_abort(&s.vfull[st], (t / kStages) & 1, s.abort)) { ok = false; break; }
      ++cv;
      const uint32_t v_addr = tc::smem_u32(s.v + st * kTileBytes);
      for (int qi = 0; qi < nq && ok; ++qi) {
        if (!wait_or_abort(&s.pfull[qi * 2 + b], (t >> 1) & 1, s.abort)) { ok = false; break; }
        tc::tc_fence_after();
        const uint32_t p_addr = tc::smem_u32(s.p + (qi * 2 + b) * kPBytes);
#pragma unroll
        for (int kk = 0; kk < kKT / 16; ++kk) {
          tc::mma_bf16(tmem + qi * kTileCols + kOCol, tc::desc_sw128(p_addr + kk * 32),
                       tc::desc_sw128_mn(v_addr + kk * 2048, kTileHalf), idesc_o, t > 0 || kk > 0);
        }
        tc::mma_commit(&s.pempty[qi * 2 + b]);
        tc::mma_commit(&s.obar[qi]);
      }
      if (!ok) break;
      tc::mma_commit(&s.vempty[st]);
      if (t + 2 < ntiles && !issue_s(t + 2)) { ok = false; break; }
    }
    if (!ok) raise_abort(a, s, tc::kSiteMma);
    s.counters[2] = ck;
    s.counters[3] = cv;
    tc::mma_commit(s.mdone);  // every MMA issued above has completed once this arrives
    tc::mbar_wait(s.mdone, 0);
  } else if (warp >= 2) {
    // -------------------------------------------------------------- softmax
    const int qi = (warp - 2) >> 2;                      // query tile of this warp
    const int et = tid - 64 - qi * kSoftThreads;         // 0..127 within the tile
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;                 // TMEM lane = query row of the tile
    const uint32_t lane_base = uint32_t(quarter * 32) << 16;
    const uint32_t tcol = qi * kTileCols;
    const int ti0 = i0 + qi * a.rows_per_tile;           // first selected row of the tile
    const int tcnt = max(0, min(a.rows_per_tile, cnt - qi * a.rows_per_tile));
    const bool active = qi < nq;
    const bool row_ok = row < tcnt * G;
    const int i_row = ti0 + (row_ok ? row / G : 0);
    const int h_row = g * G + (row_ok ? row % G : 0);
    int p_row = row_ok ? a.idx[i_row] : -1;
    if (p_row >= N) p_row = -1;
    uint8_t* q_s = s.q + qi * kQBytes;
    if (active) {  // query tile: row = (ti0 + row / G, head g*G + row % G), zero beyond tcnt * G
      for (int base = 0; base < kRows * 16; base += kSoftThreads * 8) {
        uint4 val[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int x = base + u * kSoftThreads + et;
          const int rr = x >> 4, ch = x & 15;
          val[u] = make_uint4(0u, 0u, 0u, 0u);
          if (rr < tcnt * G) {
            const int ii = ti0 + rr / G, hh = g * G + rr % G;
            val[u] = *reinterpret_cast<const uint4*>(a.q_rows + ((int64_t(l) * a.n_sel + ii) * Hq + hh) * kD + ch * 8);
          }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int x = base + u * kSoftThreads + et;
          const int rr = x >> 4, ch = x & 15;
          *reinterpret_cast<uint4*>(q_s + (ch >> 3) * kQHalf + tc::sw128_offset(rr, ch & 7)) = val[u];
        }
      }
      tc::fence_proxy_async_smem();
    }
    asm volatile("bar.sync %0, %1;" ::"r"(1 + qi), "n"(kSoftThreads) : "memory");
    if (et == 0) tc::mbar_arrive(s.qready);

    bool ok = active;
    float m_ref = -INFINITY, lsum = 0.f;
    for (int t = 0; t < ntiles && active; ++t) {
      const int b = t & 1;
      // the tcgen05.ld below is warp-collective: the whole warp goes on or stops
      const bool got = __all_sync(0xffffffffu, ok && wait_or_abort(&s.sfull[qi * 2 + b], (t >> 1) & 1, s.abort));
      if (!got) {
        if (ok) raise_abort(a, s, tc::kSiteMma);
        ok = false;
        continue;
      }
      tc::tc_fence_after();
      float sv[2][32];
      tc::tmem_ld32(tmem + lane_base + tcol + uint32_t(b) * kKT, sv[0]);
      tc::tmem_ld32(tmem + lane_base + tcol + uint32_t(b) * kKT + 32, sv[1]);
      const int j0 = t * kKT;
      float tm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      if (j0 + kKT - 1 <= p_row) {  // the whole tile is visible to this row
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2)
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            sv[h2][i] *= a.scale_log2;
            tm[i & 3] = fmaxf(tm[i & 3], sv[h2][i]);
          }
      } else {
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2)
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float x = (j0 + h2 * 32 + i <= p_row) ? sv[h2][i] * a.scale_log2 : -INFINITY;
            sv[h2][i] = x;
            tm[i & 3] = fmaxf(tm[i & 3], x);
          }
      }
      const float tmax = fmaxf(fmaxf(tm[0], tm[1]), fmaxf(tm[2], tm[3]));
      const bool need = tmax > m_ref + kRescaleLog2 || (m_ref == -INFINITY && tmax != -INFINITY);
      const float alpha = need ? exp2f(m_ref - tmax) : 1.f;  // 0 when m_ref is -inf
      if (__any_sync(0xffffffffu, need) && t > 0) {
        // P.V(t-1) must be complete before this warp rescales its rows of O.
        // S(t) was issued after P.V(t-2), so obar is at most one phase behind
        // here and its parity cannot alias.
        if (!__all_sync(0xffffffffu, wait_or_abort(&s.obar[qi], (t - 1) & 1, s.abort))) {
          raise_abort(a, s, tc::kSiteMma);
          ok = false;
          continue;
        }
        tc::tc_fence_after();
        for (int c = 0; c < kD; c += 32) {
          float o[32];
          tc::tmem_ld32(tmem + lane_base + tcol + kOCol + c, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tc::tmem_st32(tmem + lane_base + tcol + kOCol + c, o);
        }
      }
      if (need) {
        lsum *= alpha;
        m_ref = tmax;
      }
      // the P buffer of tile t was last read by P.V(t-2)
      if (!wait_or_abort(&s.pempty[qi * 2 + b], ((t >> 1) & 1) ^ 1, s.abort)) {
        raise_abort(a, s, tc::kSiteMma);
        ok = false;
        continue;
      }
      uint8_t* pb = s.p + (qi * 2 + b) * kPBytes;
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          uint32_t w4[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float p0 = (m_ref == -INFINITY) ? 0.f : tc::ex2(sv[h2][c8 * 8 + 2 * u] - m_ref);
            const float p1 = (m_ref == -INFINITY) ? 0.f : tc::ex2(sv[h2][c8 * 8 + 2 * u + 1] - m_ref);
            ls[u] += p0 + p1;
            __nv_bfloat162 pr = __floats2bfloat162_rn(p0, p1);
            w4[u] = *reinterpret_cast<uint32_t*>(&pr);
          }
          *reinterpret_cast<uint4*>(pb + tc::sw128_offset(row, h2 * 4 + c8)) =
              make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
      }
      lsum += (ls[0] + ls[1]) + (ls[2] + ls[3]);
      tc::fence_proxy_async_smem();
      tc::tc_fence_before();
      tc::mbar_arrive(&s.pfull[qi * 2 + b]);
    }
    if (active) {
      // O is complete once the MMA thread's final commit arrives. (The obar
      // phase of the last P.V could alias: after this warp's last tile only
      // P.V up to ntiles-3 is known to be done, two phases behind.)
      if (ok && !wait_or_abort(s.mdone, 0, s.abort)) {
        raise_abort(a, s, tc::kSiteFinal);
        ok = false;
      }
      const bool all_ok = !__any_sync(0xffffffffu, !ok);
      if (all_ok) {
        tc::tc_fence_after();
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
        __nv_bfloat16* dst = a.out + ((int64_t(l) * a.n_sel + i_row) * Hq + h_row) * kD;
        for (int c = 0; c < kD; c += 32) {
          float o[32];
          tc::tmem_ld32(tmem + lane_base + tcol + kOCol + c, o);
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
      }
    }
  }
  __syncthreads();
  if (tid == 0) {  // drain loads issued but never consumed (only after an abort)
    for (uint32_t n = s.counters[2]; n < s.counters[0]; ++n)
      tc::mbar_wait(&s.kfull[n % kStages], (n / kStages) & 1);
    for (uint32_t n = s.counters[3]; n < s.counters[1]; ++n)
      tc::mbar_wait(&s.vfull[n % kStages], (n / kStages) & 1);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) tc::tmem_dealloc(tmem, kTmemCols);
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
  a.rows_per_tile = kRows / kv.G;
  int blocks = 0;
  for (int r = 0; r < b.R; ++r) {
    const int kr = idx_off_host[r + 1] - idx_off_host[r];
    blocks += (kr + kTiles * a.rows_per_tile - 1) / (kTiles * a.rows_per_tile);
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
