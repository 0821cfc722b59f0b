// Tensor-core scoring pass for bf16 caches with head_dim 128 (Conduit Eq. 6).
//
// One persistent, warp-specialised kernel. A work unit is one slab (request
// r, scored layer l, KV head g) restricted to a group of at most 256 scoring
// rows (rows = the G query heads of group g times the |Q| span queries).
// Each unit makes two passes over the request's N_r keys:
//
//   pass A   D[rows x 128 tokens] = Q_rows . K_tile^T     (rows are the MMA M)
//            each epilogue thread owns one row and a share of the columns:
//            running max m and sum z = sum 2^((S - m) log2(e)/sqrt(d)), merged
//            into lse = m log2(e)/sqrt(d) + log2 z; the same threads read the
//            tile's V rows (loaded by TMA) for the value norms (ss)
//   pass B   D[128 tokens x rows] = K_tile . Q_rows^T     (tokens are the MMA M)
//            each epilogue thread owns one token and half of the rows: sum of
//            2^(x - lse) -> pa[l][g][group][half][t], this share of
//            sum_q sum_h alpha
//
// Pass B walks the tiles in reverse so the most recent K tiles of pass A are
// still in L2. Roles (352 threads):
//   warp 0       TMA loads of K tiles (128 tokens x 128 dims, 128-byte
//                swizzle) into a three-stage ring, the lanes issuing a tile's
//                copies together (one per page half when paged)
//   warp 10      the same for the matching V tiles of pass A (two buffers);
//                idle when the value norms come from the side cache
//   warp 1       one thread issues tcgen05 MMAs into two 256-column TMEM
//                accumulator slots (it also owns the TMEM allocation)
//   warps 2-9    epilogue, two warps per TMEM lane quarter (warp group h
//                = 0, 1 splits each tile's columns, or takes row block h):
//                stage the unit's scoring rows in shared memory (same
//                swizzle), then read accumulators with tcgen05.ld
// The roles meet on mbarriers (ring full / empty, accumulator full / empty,
// rows ready). Every wait is bounded by one second; a role that gives up
// raises an abort flag the others also watch, the kernel sets
// CONDUIT_FLAG_TIMEOUT, drains its copies and MMAs, and frees TMEM.
#include <cuda.h>

#include "internal.cuh"
#include "tc_common.cuh"

namespace conduit {
namespace {

constexpr int kD = 128;
constexpr int kTile = 128;
constexpr int kStages = 3;                     // K ring
constexpr int kVBufs = 2;                      // V tiles (value norms, pass A)
constexpr int kGroupRows = 256;
constexpr int kThreads = 352;
constexpr int kEpiThreads = 256;
constexpr int kVWarp = 10;                     // warps 2-9 are the epilogue
constexpr uint32_t kHalfQ = kGroupRows * 128;  // 32 KB: one 64-dim half of the row tile
constexpr uint32_t kHalfK = kTile * 128;       // 16 KB
constexpr uint32_t kStageBytes = 2 * kHalfK;   // 32 KB per K tile
constexpr uint32_t kSlotCols = 256;
constexpr uint32_t kSmemBytes = 1024 + 2 * kHalfQ + (kStages + kVBufs) * kStageBytes + 256 + kGroupRows * 4;

struct TcArgs {
  KvDev kv;
  BatchDev b;
  const __nv_bfloat16* q;
  int32_t q_tot;
  int32_t n_units;
  int32_t rg_max;      // row groups per slab, maximum over requests (pa stride)
  float scale_log2;    // log2(e) / sqrt(d)
  float* pa;           // [n_layers][Hkv][rg_max][2][n_tot]
  float* ss;           // [n_layers][Hkv][2][n_tot] sum of squares of V, per half of the head;
                       // NULL when the norms come from the side cache (V is not read)
  float* pa2;          // like pa, sums of alpha^2 (RMS statistic, Eq. 4), or NULL
  const float* extra_lse;  // [L][Hq][q_tot] natural-log LSE of keys outside the visual span, or NULL
  int32_t* status;
  LayerList layers;
#ifdef CONDUIT_TEST_HOOKS
  int32_t withhold_v;  // test builds: the V producer skips this V tile of each CTA (-1: none)
#endif
};

struct Unit {
  int r, li, l, g, rg, t0, N, q0, nq, row0, rows, tiles;
};

// Row groups of a slab with R scoring rows: ceil(R / 256) groups of equal
// size rounded up to 16 (the last one takes the rest).
__host__ __device__ __forceinline__ int n_groups(int R) { return (R + kGroupRows - 1) / kGroupRows; }
__host__ __device__ __forceinline__ int group_rows(int R) {
  const int ng = n_groups(R);
  return ng == 0 ? 0 : (((R + ng - 1) / ng) + 15) & ~15;
}

__device__ __forceinline__ bool decode_unit(const TcArgs& a, int u, Unit& w) {
  const int Hkv = a.kv.Hkv, nl = a.layers.n, G = a.kv.G;
  int base = 0;
  for (int r = 0; r < a.b.R; ++r) {
    const int nq = a.b.q_off[r + 1] - a.b.q_off[r];
    const int R = G * nq;
    const int ng = n_groups(R);
    const int cnt = nl * Hkv * ng;
    if (u < base + cnt) {
      int local = u - base;
      w.r = r;
      w.rg = local % ng;
      local /= ng;
      w.g = local % Hkv;
      w.li = local / Hkv;
      w.l = a.layers.ids[w.li];
      w.t0 = a.b.tok_off[r];
      w.N = a.b.tok_off[r + 1] - w.t0;
      w.q0 = a.b.q_off[r];
      w.nq = nq;
      const int gr = group_rows(R);
      w.row0 = w.rg * gr;
      w.rows = min(gr, R - w.row0);
      w.tiles = (w.N + kTile - 1) / kTile;
      return w.rows > 0;
    }
    base += cnt;
  }
  return false;
}

// Tile index of the i-th K tile of the unit's two passes (pass B in reverse).
__device__ __forceinline__ int tile_of(const Unit& w, int i) {
  return i < w.tiles ? i : 2 * w.tiles - 1 - i;
}

struct Smem {
  uint8_t* q;          // [2 halves][256 rows][128 B]
  uint8_t* k;          // [kStages][2 halves][128 rows][128 B]
  uint64_t* kfull;     // [kStages]
  uint64_t* kempty;    // [kStages]
  uint8_t* v;          // [kVBufs][2 halves][128 rows][128 B]
  uint64_t* vfull;     // [kVBufs]
  uint64_t* vempty;    // [kVBufs]
  uint64_t* tfull;     // [2]
  uint64_t* tempty;    // [2]
  uint64_t* qready;    // [1]
  uint64_t* mdone;     // [1]
  uint32_t* tmem_slot;
  volatile int* abort;
  uint32_t* counters;  // [0] K loads issued, [1] K loads consumed, [2] V issued, [3] V consumed,
                       // [4] (test builds) 1 + the V tile withheld, else 0
  float* lse;          // [256]
};

__device__ __forceinline__ Smem carve(uint8_t* raw) {
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  Smem s;
  s.q = base;
  s.k = base + 2 * kHalfQ;
  s.v = s.k + kStages * kStageBytes;
  uint8_t* tail = s.v + kVBufs * kStageBytes;
  s.kfull = reinterpret_cast<uint64_t*>(tail);
  s.kempty = s.kfull + kStages;
  s.vfull = s.kempty + kStages;
  s.vempty = s.vfull + kVBufs;
  s.tfull = s.vempty + kVBufs;
  s.tempty = s.tfull + 2;
  s.qready = s.tempty + 2;
  s.mdone = s.qready + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.mdone + 1);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  s.counters = reinterpret_cast<uint32_t*>(s.tmem_slot + 2);
  s.lse = reinterpret_cast<float*>(tail + 256);
  return s;
}

// Bounded wait that also gives up when another role has aborted.
// Non-blocking test of the phase with the given parity (no suspension): for
// the epilogue's waits on an accumulator slot, which the MMA thread has
// usually filled already.
__device__ __forceinline__ bool mbar_probe(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\nselp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(done)
      : "r"(tc::smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
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

__device__ __forceinline__ void raise_abort(const TcArgs& a, const Smem& s, int32_t site) {
  *s.abort = 1;
  flag_status(a.status, CONDUIT_FLAG_TIMEOUT | site);
}

__device__ __forceinline__ void epi_barrier() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
}

// Warp-cooperative TMA of K (or V) tile `tile` of unit w into `dst`: lane 0
// posts the byte count, then copy c is issued by lane c. A copy is one 64-dim
// half of the whole tile (contiguous cache: 2 copies) or of one page (paged
// cache: 2 x 128/page copies, up to 32), so a paged tile costs one round of
// parallel page-index loads and copy issues.
__device__ __forceinline__ void load_k_tile(const TcArgs& a, const CUtensorMap* kmap, const Unit& w,
                                            uint8_t* dst, uint64_t* bar, int tile, int lane) {
  if (lane == 0) tc::mbar_arrive_expect_tx(bar, kStageBytes);
  __syncwarp();
  const int tok = tile * kTile;
  const KvDev& kv = a.kv;
  const int hf = lane & 1;
  if (kv.page_size == 0) {
    if (lane < 2) {
      const int32_t y = int32_t((int64_t(w.l) * kv.Hkv + w.g) * kv.n_tot + w.t0 + tok);
      tc::tma_load_2d(dst + hf * kHalfK, kmap, bar, hf * 64, y);
    }
  } else {
    const int ps = kv.page_size;
    const int i = lane >> 1;  // page of the tile
    if (i < kTile / ps) {
      const int lp = min((tok + i * ps) / ps, (w.N - 1) / ps);  // tail pages repeat the last one (masked)
      const int page = kv.page_table[int64_t(w.r) * kv.max_pages + lp];
      const int32_t y = int32_t(((int64_t(w.l) * kv.num_pages + page) * kv.Hkv + w.g) * ps);
      tc::tma_load_2d(dst + hf * kHalfK + i * ps * 128, kmap, bar, hf * 64, y);
    }
  }
}

// Epilogue threads stage scoring rows [row0, row0 + nrows) of the unit into
// the swizzled row tile (rows at or beyond the group are zero); eight
// 16-byte loads per thread are in flight at a time.
__device__ __forceinline__ void stage_rows(const TcArgs& a, const Unit& w, uint8_t* q_s, int nrows,
                                           int et) {
  const int G = a.kv.G, Hq = a.kv.Hq;
  const int total = nrows * 16;
  for (int base = 0; base < total; base += kEpiThreads * 8) {
    uint4 val[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int idx = base + u * kEpiThreads + et;
      val[u] = make_uint4(0u, 0u, 0u, 0u);
      if (idx < total) {
        const int row = idx >> 4, ch = idx & 15;
        if (row < w.rows) {
          const int j = w.row0 + row;
          const int h = w.g * G + j / w.nq, qi = j % w.nq;
          val[u] = *reinterpret_cast<const uint4*>(
              a.q + ((int64_t(w.l) * Hq + h) * a.q_tot + w.q0 + qi) * kD + ch * 8);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int idx = base + u * kEpiThreads + et;
      if (idx < total) {
        const int row = idx >> 4, ch = idx & 15;
        *reinterpret_cast<uint4*>(q_s + (ch >> 3) * kHalfQ + tc::sw128_offset(row, ch & 7)) = val[u];
      }
    }
  }
}

// 2^(s scale + b) for a pair of accumulator values (one packed FMA, two MUFU ops).
__device__ __forceinline__ float2 exp2_pair(float s0, float s1, float2 sc2, float2 b2, int) {
  const float2 y = tc::ffma2(make_float2(s0, s1), sc2, b2);
  return make_float2(tc::ex2(y.x), tc::ex2(y.y));
}

// Online row statistics over NC accumulator columns of which the first
// `valid` are tokens of the slab: running max m (raw logit) and
// z = sum 2^((S - m) scale). Only a ragged last tile takes the masked path.
template <int NC>
__device__ __forceinline__ void row_stats(float (&v)[NC], int valid, float scale, float& m,
                                          float& z) {
  if (valid < NC) {
#pragma unroll
    for (int x = 0; x < NC; ++x)
      if (x >= valid) v[x] = -INFINITY;
  }
  float cm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int x = 0; x < NC / 2; ++x) cm[x & 3] = tc::fmax3(cm[x & 3], v[2 * x], v[2 * x + 1]);
  const float mn = fmaxf(m, fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3])));
  if (mn == -INFINITY) return;
  const float2 sc2 = make_float2(scale, scale), nb2 = make_float2(-mn * scale, -mn * scale);
  float2 ac[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int x = 0; x < NC / 2; ++x) ac[x & 1] = tc::fadd2(ac[x & 1], exp2_pair(v[2 * x], v[2 * x + 1], sc2, nb2, x));
  z = z * tc::ex2((m - mn) * scale) + ((ac[0].x + ac[0].y) + (ac[1].x + ac[1].y));
  m = mn;
}

// Sum over NC accumulator columns (scoring rows c0 ...) of 2^(S scale - lse_row),
// given nlse = -lse. Columns past the row group carry nlse = -inf and add
// exactly zero (the accumulator columns there hold finite values: TMEM is
// zeroed at start).
template <int NC>
__device__ __forceinline__ float col_sum(const float (&v)[NC], const float* nlse, float scale) {
  const float2 sc2 = make_float2(scale, scale);
  float2 ac[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int x4 = 0; x4 < NC / 4; ++x4) {
    const float4 lv = reinterpret_cast<const float4*>(nlse)[x4];
    ac[0] = tc::fadd2(ac[0], exp2_pair(v[4 * x4 + 0], v[4 * x4 + 1], sc2, make_float2(lv.x, lv.y), 2 * x4));
    ac[1] = tc::fadd2(ac[1], exp2_pair(v[4 * x4 + 2], v[4 * x4 + 3], sc2, make_float2(lv.z, lv.w), 2 * x4 + 1));
  }
  return (ac[0].x + ac[0].y) + (ac[1].x + ac[1].y);
}

// col_sum that also returns the sum of the squared terms (alpha^2, for the
// RMS statistic); the plain sum is computed exactly as col_sum computes it.
template <int NC>
__device__ __forceinline__ float col_sum_sq(const float (&v)[NC], const float* nlse, float scale,
                                            float& sq) {
  const float2 sc2 = make_float2(scale, scale);
  float2 ac[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  float2 aq[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int x4 = 0; x4 < NC / 4; ++x4) {
    const float4 lv = reinterpret_cast<const float4*>(nlse)[x4];
    const float2 p0 = exp2_pair(v[4 * x4 + 0], v[4 * x4 + 1], sc2, make_float2(lv.x, lv.y), 2 * x4);
    const float2 p1 = exp2_pair(v[4 * x4 + 2], v[4 * x4 + 3], sc2, make_float2(lv.z, lv.w), 2 * x4 + 1);
    ac[0] = tc::fadd2(ac[0], p0);
    ac[1] = tc::fadd2(ac[1], p1);
    aq[0] = tc::ffma2(p0, p0, aq[0]);
    aq[1] = tc::ffma2(p1, p1, aq[1]);
  }
  sq = (aq[0].x + aq[0].y) + (aq[1].x + aq[1].y);
  return (ac[0].x + ac[0].y) + (ac[1].x + ac[1].y);
}

__global__ void __launch_bounds__(kThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                    const __grid_constant__ TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const Smem s = carve(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      tc::mbar_init(&s.kfull[i], 1);
      tc::mbar_init(&s.kempty[i], 1);
    }
    for (int i = 0; i < kVBufs; ++i) {
      tc::mbar_init(&s.vfull[i], 1);
      tc::mbar_init(&s.vempty[i], kEpiThreads);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.tfull[i], 1);
      tc::mbar_init(&s.tempty[i], kEpiThreads);
    }
    tc::mbar_init(s.qready, 1);
    tc::mbar_init(s.mdone, 1);
    *s.abort = 0;
    for (int i = 0; i < 5; ++i) s.counters[i] = 0;
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
    tc::prefetch_tensormap(&vmap);
  }
  if (warp == 1) tc::tmem_alloc(s.tmem_slot, 2 * kSlotCols);
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *s.tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------- producer: K (warp 0)
    uint32_t seq = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
      Unit w;
      if (!decode_unit(a, u, w)) continue;
      for (int i = 0; i < 2 * w.tiles; ++i, ++seq) {
        const int st = seq % kStages;
        if (!__all_sync(0xffffffffu, wait_or_abort(&s.kempty[st], ((seq / kStages) & 1) ^ 1, s.abort))) {
          if (lane == 0 && !*s.abort) raise_abort(a, s, tc::kSiteLoad);
          ok = false;
          break;
        }
        load_k_tile(a, &kmap, w, s.k + st * kStageBytes, &s.kfull[st], tile_of(w, i), lane);
      }
    }
    if (lane == 0) s.counters[0] = seq;
  } else if (warp == kVWarp) {
    // ------------------------------------------------ producer: V (warp 10)
    // V tiles of pass 1 for the value norms, on a warp of their own so that a
    // V tile waiting for its buffer never holds back the K ring
    uint32_t vseq = 0;
    bool ok = a.ss != nullptr;  // no V traffic when the norms come from the side cache
    for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
      Unit w;
      if (!decode_unit(a, u, w) || w.rg != 0) continue;
      for (int i = 0; i < w.tiles; ++i, ++vseq) {
        const int vb = vseq % kVBufs;
        if (!__all_sync(0xffffffffu, wait_or_abort(&s.vempty[vb], ((vseq / kVBufs) & 1) ^ 1, s.abort))) {
          if (lane == 0 && !*s.abort) raise_abort(a, s, tc::kSiteLoad);
          ok = false;
          break;
        }
#ifdef CONDUIT_TEST_HOOKS
        if (int(vseq) == a.withhold_v) {  // neither copy nor arrive: the consumer's wait runs out
          if (lane == 0) s.counters[4] = vseq + 1;
          continue;
        }
#endif
        load_k_tile(a, &vmap, w, s.v + vb * kStageBytes, &s.vfull[vb], i, lane);
      }
    }
    if (lane == 0) s.counters[2] = vseq;
  } else if (warp == 1 && lane == 0) {
    // ----------------------------------------------------------------- MMA
    uint32_t kseq = 0, tseq = 0, useq = 0;
    bool ok = true;
    const uint32_t qb = tc::smem_u32(s.q);
    for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
      Unit w;
      if (!decode_unit(a, u, w)) continue;
      if (!wait_or_abort(s.qready, useq & 1, s.abort)) {
        if (!*s.abort) raise_abort(a, s, tc::kSiteMma);
        break;
      }
      ++useq;
      tc::tc_fence_after();
      const int nrb = (w.rows + 127) / 128;
      const int ncols = (w.rows + 15) & ~15;
      for (int i = 0; i < 2 * w.tiles; ++i) {
        const int st = kseq % kStages;
        if (!wait_or_abort(&s.kfull[st], (kseq / kStages) & 1, s.abort)) {
          if (!*s.abort) raise_abort(a, s, tc::kSiteLoad);
          ok = false;
          break;
        }
        ++kseq;
        const int slot = tseq & 1;
        if (!wait_or_abort(&s.tempty[slot], ((tseq >> 1) & 1) ^ 1, s.abort)) {
          if (!*s.abort) raise_abort(a, s, tc::kSiteMma);
          ok = false;
          break;
        }
        ++tseq;
        tc::tc_fence_after();
        const uint32_t kb = tc::smem_u32(s.k + st * kStageBytes);
        const uint32_t d = tmem + uint32_t(slot) * kSlotCols;
        if (i < w.tiles) {  // pass A: rows x tokens
          const uint32_t idesc = tc::idesc_bf16(128, kTile);
          for (int rb = 0; rb < nrb; ++rb) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint32_t off = (kk >> 2) * 0 + (kk & 3) * 32;
              tc::mma_bf16(d + rb * 128, tc::desc_sw128(qb + (kk >> 2) * kHalfQ + rb * 128 * 128 + off),
                           tc::desc_sw128(kb + (kk >> 2) * kHalfK + off), idesc, kk > 0);
            }
          }
        } else {            // pass B: tokens x rows
          const uint32_t idesc = tc::idesc_bf16(128, ncols);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            tc::mma_bf16(d, tc::desc_sw128(kb + (kk >> 2) * kHalfK + off),
                         tc::desc_sw128(qb + (kk >> 2) * kHalfQ + off), idesc, kk > 0);
          }
        }
        tc::mma_commit(&s.kempty[st]);
        tc::mma_commit(&s.tfull[slot]);
      }
    }
    s.counters[1] = kseq;
    tc::mma_commit(s.mdone);  // every MMA issued above has completed once this arrives
    tc::mbar_wait(s.mdone, 0);
  } else if (warp >= 2 && warp < kVWarp) {
    // ------------------------------------------------------------ epilogue
    // After an abort the epilogue keeps walking its units (skipping the work)
    // so that every thread reaches every named barrier.
    const int et = tid - 64;                       // 0..255
    const int h = et >> 7;                         // warp group: column half or row block
    const int quarter = warp & 3;                  // TMEM lanes 32*quarter .. +31
    const int lrow = quarter * 32 + lane;          // row (pass A) / token (pass B) in the tile
    const uint32_t lane_base = uint32_t(quarter * 32) << 16;
    const int64_t n_tot = a.kv.n_tot;
    uint32_t tseq = 0, vcons = 0;
    bool ok = true;
    {  // zero this warp's TMEM lanes once, so unwritten accumulator columns hold finite values
      uint32_t zero[64];
#pragma unroll
      for (int i = 0; i < 64; ++i) zero[i] = 0u;
      for (int c = h * 256; c < h * 256 + 256; c += 64) tc::tmem_st64(tmem + lane_base + c, zero);
      tc::tc_fence_before();
    }
    for (int u = blockIdx.x; u < a.n_units; u += gridDim.x) {
      Unit w;
      if (!decode_unit(a, u, w)) continue;
      const int nrb = (w.rows + 127) / 128;
      if (ok && !*s.abort) stage_rows(a, w, s.q, nrb * 128, et);
      tc::fence_proxy_async_smem();
      epi_barrier();
      if (et == 0) tc::mbar_arrive(s.qready);
      // pass A share: row block rb (with one row block the second warp group
      // only does value norms) and this thread's half of each V row
      const bool do_rows = nrb == 2 || h == 0;
      const int rb = nrb == 2 ? h : 0;
      const bool do_norm = w.rg == 0 && a.ss != nullptr;  // one row group of each slab also streams V
      const int64_t lg = int64_t(w.li) * a.kv.Hkv + w.g;
      float* ss_out = do_norm ? a.ss + (lg * 2 + h) * n_tot + w.t0 : nullptr;
      float m = -INFINITY, z = 0.f;
      for (int i = 0; i < w.tiles; ++i) {            // pass A
        const int slot = tseq & 1;
        // tcgen05.ld is warp-collective: the whole warp goes on or stops
        const bool got = __all_sync(0xffffffffu, ok && (mbar_probe(&s.tfull[slot], (tseq >> 1) & 1) ||
                                                        wait_or_abort(&s.tfull[slot], (tseq >> 1) & 1, s.abort)));
        ++tseq;
        if (!got) {
          if (ok && !*s.abort) raise_abort(a, s, tc::kSiteMma);
          ok = false;
          continue;
        }
        tc::tc_fence_after();
        const uint32_t col0 = uint32_t(slot) * kSlotCols + rb * 128;
        const int valid = w.N - i * kTile;
        if (do_rows) {  // 128 columns in two loads; the slot is free again after the second
          float v[64];
          tc::tmem_ld64(tmem + lane_base + col0, v);
          row_stats<64>(v, valid, a.scale_log2, m, z);
          tc::tmem_ld64(tmem + lane_base + col0 + 64, v);
          tc::tc_fence_before();
          tc::mbar_arrive(&s.tempty[slot]);
          row_stats<64>(v, valid - 64, a.scale_log2, m, z);
        } else {
          tc::tc_fence_before();
          tc::mbar_arrive(&s.tempty[slot]);
        }
        if (do_norm) {  // half (64 dims) of V row lrow of the tile, from shared memory
          const int vb = vcons % kVBufs;
          if (!wait_or_abort(&s.vfull[vb], (vcons / kVBufs) & 1, s.abort)) {
            if (!*s.abort) raise_abort(a, s, tc::kSiteLoad);
            ok = false;
            continue;
          }
          ++vcons;
          const uint8_t* vh = s.v + vb * kStageBytes + h * kHalfK;
          float sq[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int c = 0; c < 8; ++c)
            sumsq_bf16_chunk(*reinterpret_cast<const uint4*>(vh + tc::sw128_offset(lrow, c)), sq);
          tc::mbar_arrive(&s.vempty[vb]);
          const int tok = i * kTile + lrow;
          if (tok < w.N) ss_out[tok] = sumsq_combine(sq);
        }
      }
      // minus the log2-sum-exp of each row, shared with the token-owning
      // threads of pass B (-inf past the row group: those columns add nothing)
      {
        const int row = (do_rows ? rb : 1) * 128 + lrow;
        float lse = (do_rows && row < w.rows) ? m * a.scale_log2 + log2f(z) : INFINITY;
        if (a.extra_lse != nullptr && do_rows && row < w.rows) {
          // full-context softmax: the keys outside the visual span join the denominator
          const int j = w.row0 + row, hq = w.g * a.kv.G + j / w.nq, qi = j % w.nq;
          const float e = a.extra_lse[(int64_t(w.l) * a.kv.Hq + hq) * a.q_tot + w.q0 + qi];
          lse = log2_add(lse, e * kLog2e);
        }
        s.lse[row] = -lse;
      }
      epi_barrier();
      // pass B share: 32-row chunks [cb0, cb1)
      const int nchunk = (w.rows + 31) / 32;
      const int hc = (nchunk + 1) / 2;
      const int cb0 = h * hc, cb1 = min(nchunk, cb0 + hc);
      float* pa_out = a.pa + ((lg * a.rg_max + w.rg) * 2 + h) * n_tot + w.t0;
      float* pa2_out = a.pa2 ? a.pa2 + ((lg * a.rg_max + w.rg) * 2 + h) * n_tot + w.t0 : nullptr;
      for (int i = w.tiles; i < 2 * w.tiles; ++i) {  // pass B
        const int slot = tseq & 1;
        const int tok = tile_of(w, i) * kTile + lrow;
        // tcgen05.ld is warp-collective: the whole warp goes on or stops
        const bool got = __all_sync(0xffffffffu, ok && (mbar_probe(&s.tfull[slot], (tseq >> 1) & 1) ||
                                                        wait_or_abort(&s.tfull[slot], (tseq >> 1) & 1, s.abort)));
        ++tseq;
        if (!got) {
          if (ok && !*s.abort) raise_abort(a, s, tc::kSiteMma);
          ok = false;
          continue;
        }
        tc::tc_fence_after();
        // this thread's columns [32 cb0, 32 cb1) in loads of 64 (and one of 32);
        // the slot is free again after the last load
        const uint32_t col0 = uint32_t(slot) * kSlotCols + cb0 * 32;
        const int ncol = (cb1 - cb0) * 32;
        const float* lse = s.lse + cb0 * 32;
        float acc = 0.f, acc2 = 0.f;
        int c = 0;
        for (; c + 64 <= ncol; c += 64) {
          float v[64];
          tc::tmem_ld64(tmem + lane_base + col0 + c, v);
          if (c + 64 == ncol) {
            tc::tc_fence_before();
            tc::mbar_arrive(&s.tempty[slot]);
          }
          if (pa2_out) {
            float q2;
            acc += col_sum_sq<64>(v, lse + c, a.scale_log2, q2);
            acc2 += q2;
          } else {
            acc += col_sum<64>(v, lse + c, a.scale_log2);
          }
        }
        if (c < ncol) {
          float v[32];
          tc::tmem_ld32(tmem + lane_base + col0 + c, v);
          tc::tc_fence_before();
          tc::mbar_arrive(&s.tempty[slot]);
          if (pa2_out) {
            float q2;
            acc += col_sum_sq<32>(v, lse + c, a.scale_log2, q2);
            acc2 += q2;
          } else {
            acc += col_sum<32>(v, lse + c, a.scale_log2);
          }
        } else if (ncol == 0) {
          tc::tc_fence_before();
          tc::mbar_arrive(&s.tempty[slot]);
        }
        if (tok < w.N) {
          pa_out[tok] = acc;
          if (pa2_out) pa2_out[tok] = acc2;
        }
      }
      epi_barrier();  // every thread is done with this unit's rows and lse
    }
    if (et == 0) s.counters[3] = vcons;
  }
  __syncthreads();
  if (tid == 0) {  // drain TMA copies issued but never consumed (only after an abort)
    for (uint32_t n = s.counters[1]; n < s.counters[0]; ++n)
      tc::mbar_wait(&s.kfull[n % kStages], (n / kStages) & 1);
    for (uint32_t n = s.counters[3]; n < s.counters[2]; ++n)
      if (n + 1 != s.counters[4])  // (test builds) a withheld V tile has nothing in flight
        tc::mbar_wait(&s.vfull[n % kVBufs], (n / kVBufs) & 1);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) tc::tmem_dealloc(tmem, 2 * kSlotCols);
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

#ifdef CONDUIT_TEST_HOOKS
// Test builds only (never in libconduit.so): the next scoring launches
// withhold V tile n of each CTA (n < 0: none), so that the epilogue's bounded
// wait for it runs out and the kernel takes its timeout path.
int32_t g_test_withhold_v = -1;
extern "C" void conduit_test_withhold_v_tile(int32_t n) { g_test_withhold_v = n; }
#endif

bool score_tc_supported(const KvDev& kv) {
  if (kv.dtype != CONDUIT_BF16 || kv.d != kD) return false;
  if (kv.page_size != 0 && (kv.page_size % 8 != 0 || kTile % kv.page_size != 0)) return false;
  return true;
}

int score_tc_groups(int rows) { return n_groups(rows); }

cudaError_t launch_score_tc(const KvDev& kv, const BatchDev& b, const int32_t* q_off_host,
                            const void* q, int32_t q_tot, const LayerList& layers, int rg_max,
                            float* pa, float* ss, float* pa2, const float* extra_lse,
                            int32_t* status, cudaStream_t stream) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap kmap, vmap;
  cuuint64_t dims[2] = {cuuint64_t(kD), 0};
  cuuint64_t strides[1] = {cuuint64_t(kD) * 2};
  cuuint32_t box[2] = {64, 0};
  cuuint32_t estr[2] = {1, 1};
  if (kv.page_size == 0) {
    dims[1] = cuuint64_t(kv.L) * kv.Hkv * kv.n_tot;
    box[1] = kTile;
  } else {
    dims[1] = cuuint64_t(kv.L) * kv.num_pages * kv.Hkv * kv.page_size;
    box[1] = kv.page_size;
  }
  if (enc(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, kv.k, dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  if (enc(&vmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ss ? kv.v : kv.k, dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;

  TcArgs a{};
  a.kv = kv;
  a.b = b;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.q_tot = q_tot;
  int units = 0;
  for (int r = 0; r < b.R; ++r)
    units += layers.n * kv.Hkv * n_groups(kv.G * (q_off_host[r + 1] - q_off_host[r]));
  a.n_units = units;
  a.rg_max = rg_max;
  a.scale_log2 = kLog2e / sqrtf(float(kD));
  a.pa = pa;
  a.ss = ss;
  a.pa2 = pa2;
  a.extra_lse = extra_lse;
  a.status = status;
  a.layers = layers;
#ifdef CONDUIT_TEST_HOOKS
  a.withhold_v = g_test_withhold_v;
#endif
  if (units == 0) return cudaSuccess;

  int dev = 0, sms = 0;
  cudaError_t err;
  if ((err = cudaGetDevice(&dev))) return err;
  if ((err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))) return err;
  if ((err = cudaFuncSetAttribute(score_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  int(kSmemBytes))))
    return err;
  score_tc_kernel<<<std::min(units, sms), kThreads, kSmemBytes, stream>>>(kmap, vmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
