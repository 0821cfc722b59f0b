// Tensor-core causal refresh attention for bf16 caches with head_dim 128
// (selective recompute, Conduit Sec. 3.1 / 4.3):
//   out[l][i][h] = sum_{j <= p_i} softmax_j(<q[l][i][h], K'[l][h/G][j]> / sqrt(d)) V'[l][h/G][j]
//
// Work item: one query tile of 128 rows of one (layer, KV head, request),
// floor(128/G) consecutive selected rows times the G query heads that share
// the KV head. Keys stream in tiles of 128 (an MMA-issuing thread, which
// shares its sub-partition with two softmax warps, is paced per instruction,
// so wide tiles halve its work). The kernel is persistent: one CTA per SM
// takes items from an atomic counter, and the query tile of the next item
// loads into a second buffer while the current item computes. Roles (384
// threads):
//   warp 0     TMA loads: the query tile of each item (a 3-D box of 64 dims x
//              G heads x floor(128/G) rows lands in the tile's row order) into
//              one of two buffers, then its K tiles (two stages); the lanes
//              issue the copies of a tile together (one per page half when
//              paged)
//   warp 10    the same for the V tiles (two stages), so that a V stage
//              waiting for its P.V never holds back K and the next query tile
//   warp 1     one thread issues S(t) = Q K(t)^T into TMEM buffer t % 3
//   warp 11    one thread issues O += P(t) V(t) with P read from TMEM; two
//              issuing threads, because one thread issuing both (with a wait
//              for each P.V before the S that reuses its buffer) took longer
//              per key tile than the softmax
//   warps 2-9  softmax, two warps per TMEM lane quarter: each thread owns one
//              row and one half (64 keys) of every key tile. Per tile it reads
//              its half of S(t), applies the causal mask j <= p_i, exchanges
//              the half-row max with its partner through shared memory, keeps
//              a lazy running max (O and the row sum are rescaled only when
//              the max grows by 2^8; warp-uniform, since tcgen05.ld/st are
//              warp-collective), writes its half of P as bf16 pairs over the
//              upper half of S(t), and at the item's end writes its half of
//              O / rowsum
// TMEM: three S buffers at columns [0, 384) (P in the upper 64 of each), O at
// [384, 512). S(t) reuses the buffer of P(t-3), so it is issued once
// P(t-3) V(t-3) has completed (per-buffer completion barriers): the S thread
// runs up to two tiles ahead of the softmax, which finds S(t+1) ready when it
// finishes P(t) and probes for it without suspending; the next item's first
// S tiles are computed while the softmax writes the previous item's O. Rows
// are sorted by position, so an item needs
// keys up to its last row's position only. Every barrier phase follows from
// per-CTA sequence numbers (items n, key tiles T) that all roles advance
// alike. Every wait is bounded by one second; a role that gives up raises an
// abort flag the others watch, the kernel sets CONDUIT_FLAG_TIMEOUT, drains
// its copies and MMAs, and frees TMEM.
#include <cuda.h>

#include "internal.cuh"
#include "tc_common.cuh"

namespace conduit {
namespace {

constexpr int kD = 128;
constexpr int kKT = 128;                         // keys per tile
constexpr int kRows = 128;                       // rows per query tile
constexpr int kSoftThreads = 256;
constexpr int kVWarp = 10;                       // after the loader, MMA and eight softmax warps
constexpr int kPvWarp = 11;                      // the thread issuing O += P V
constexpr int kThreads = 64 + kSoftThreads + 64;
constexpr int kKStages = 2;
constexpr int kVStages = 2;
constexpr int kQBufs = 2;
constexpr uint32_t kQHalf = kRows * 128;         // 16 KB: one 64-dim half of the query tile
constexpr uint32_t kQBytes = 2 * kQHalf;         // 32 KB
constexpr uint32_t kTileHalf = kKT * 128;        // 16 KB: one 64-dim half of a K or V tile
constexpr uint32_t kTileBytes = 2 * kTileHalf;   // 32 KB
constexpr int kRecInts = 9;                      // decoded item record (see Smem::rec)
constexpr uint32_t kSmem = 1024 + kQBufs * kQBytes + (kKStages + kVStages) * kTileBytes + 256 +
                           2 * 2 * 128 * 4 + 2 * 128 * 4 + kQBufs * (kRecInts + kRows) * 4;
constexpr uint32_t kTmemCols = 512;              // three S / P buffers and O
constexpr uint32_t kSCols = 128;                 // one S buffer
constexpr int kSBufs = 3;                        // S runs up to two key tiles ahead of the softmax
constexpr uint32_t kPCol = 64;                   // P (bf16 pairs) over the upper half of S
constexpr uint32_t kOCol = kSBufs * kSCols;      // O
constexpr float kRescaleLog2 = 8.f;

struct RefArgs {
  KvDev kv;
  BatchDev b;
  const int32_t* idx;
  const int32_t* idx_off;
  const __nv_bfloat16* q_rows;
  __nv_bfloat16* out;
  int32_t out32;           // out is 32-byte aligned: rows are written in 32-byte stores
  int32_t n_sel;
  int32_t rows_per_tile;   // selected rows per query tile, floor(128 / G)
  int32_t n_blocks;        // query tiles per (layer, KV head)
  int32_t n_items;         // n_blocks * Hkv * L
  int32_t blocks_major;    // item order: query tile (largest first) outer, or (layer, head) outer
  int32_t* next_item;      // work counter, zero at launch
  float scale_log2;
  int32_t* status;
};

// A work item: query tile `blk` of (layer l, KV head g), counted from the
// largest positions, and the request, first selected row and row count.
// Every layer and head of a request has the same selected positions, so the
// blocks-major order (all (layer, head) pairs of the largest tile first) is
// longest-first scheduling; the (layer, head)-major order keeps the CTAs in
// flight on few K/V prefixes, which L2 then shares when the cache exceeds it.
struct Item {
  int l, g, r, i0, cnt;
};

__device__ __forceinline__ Item decode_item(const RefArgs& a, int u) {
  Item it;
  const int n_lg = a.kv.Hkv * a.kv.L;
  const int x = a.blocks_major ? u / n_lg : u % a.n_blocks;
  const int lg = a.blocks_major ? u % n_lg : u / a.n_blocks;
  it.g = lg % a.kv.Hkv;
  it.l = lg / a.kv.Hkv;
  int blk = a.n_blocks - 1 - x;
  it.r = 0;
  it.i0 = -1;
  it.cnt = 0;
  const int span = a.rows_per_tile;
  for (int rr = 0; rr < a.b.R; ++rr) {
    const int k0 = a.idx_off[rr], kr = a.idx_off[rr + 1] - k0;
    const int nb = (kr + span - 1) / span;
    if (blk < nb) {
      it.r = rr;
      it.i0 = k0 + blk * span;
      it.cnt = min(span, kr - blk * span);
      break;
    }
    blk -= nb;
  }
  return it;
}

// Key tiles of an item: up to its last row's position.
__device__ __forceinline__ int item_tiles(const RefArgs& a, const Item& it) {
  if (it.i0 < 0) return 0;
  const int N = a.b.tok_off[it.r + 1] - a.b.tok_off[it.r];
  const int p_max = min(a.idx[it.i0 + it.cnt - 1], N - 1);
  return p_max < 0 ? 0 : p_max / kKT + 1;
}

struct Smem {
  uint8_t* q;        // [kQBufs][2 halves][128 rows][128 B]
  uint8_t* k;        // [kKStages][2 halves][128 keys][128 B]
  uint8_t* v;        // [kVStages][2 halves][128 keys][128 B]
  uint64_t *kfull, *kempty;   // [kKStages]
  uint64_t *vfull, *vempty;   // [kVStages]
  uint64_t *sfull, *pfull;    // [kSBufs] per S buffer
  uint64_t *pvdone;           // [kSBufs] per S buffer: the P.V that read its P has completed
  uint64_t *qfull, *qempty;   // [kQBufs] query tile (and item index) of one item
  uint64_t *ofull, *oempty;   // once per item: O complete / O read out
  uint64_t *mdone;            // [2] per MMA thread: all its MMAs completed
  uint32_t* tmem_slot;
  volatile int* abort;
  uint32_t* counters;  // [0] K loads, [1] V loads, [2] K consumed, [3] V consumed
  float* xmax;         // [2 tile parities][2 halves][128 rows] half-row maxima
  float* xsum;         // [2 halves][128 rows] half-row sums at the end
  // per query buffer, written by the loader with the query tile: the decoded
  // item {u (-1: no more work), l, g, r, i0, cnt, key tiles, N_r, t0} and the
  // positions of its selected rows, so the other roles read no global memory
  // between items
  volatile int* rec;   // [kQBufs][kRecInts]
  volatile int* pos;   // [kQBufs][kRows]
};

__device__ __forceinline__ Smem carve(uint8_t* raw) {
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
  Smem s;
  s.q = base;
  s.k = s.q + kQBufs * kQBytes;
  s.v = s.k + kKStages * kTileBytes;
  uint64_t* bar = reinterpret_cast<uint64_t*>(s.v + kVStages * kTileBytes);
  s.kfull = bar;
  s.kempty = s.kfull + kKStages;
  s.vfull = s.kempty + kKStages;
  s.vempty = s.vfull + kVStages;
  s.sfull = s.vempty + kVStages;
  s.pfull = s.sfull + kSBufs;
  s.pvdone = s.pfull + kSBufs;
  s.qfull = s.pvdone + kSBufs;
  s.qempty = s.qfull + kQBufs;
  s.ofull = s.qempty + kQBufs;
  s.oempty = s.ofull + 1;
  s.mdone = s.oempty + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.mdone + 2);
  s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
  s.counters = reinterpret_cast<uint32_t*>(s.tmem_slot + 2);
  s.xmax = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bar) + 256);
  s.xsum = s.xmax + 2 * 2 * 128;
  s.rec = reinterpret_cast<volatile int*>(s.xsum + 2 * 128);
  s.pos = s.rec + kQBufs * kRecInts;
  return s;
}

// Non-blocking test of the phase with the given parity (no suspension): for
// the softmax's wait on S, which the S thread has usually completed already.
// Waits that are often not yet complete (the MMA threads') use wait_or_abort
// alone: a probe in front of them cost more than it saved.
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

__device__ __forceinline__ void raise_abort(const RefArgs& a, const Smem& s, int32_t site) {
  if (!*s.abort) flag_status(a.status, CONDUIT_FLAG_TIMEOUT | site);
  *s.abort = 1;
}

// Warp-cooperative TMA of the 128-key tile starting at request-local key j0:
// lane 0 posts the byte count, then copy c is issued by lane c. A copy is one
// 64-dim half of the whole tile (contiguous cache: 2 copies) or of one page
// (paged cache: 2 x 128/page copies, up to 32), so a paged tile costs one
// round of parallel page-index loads and copy issues instead of a serial loop.
__device__ __forceinline__ void load_tile(const RefArgs& a, const CUtensorMap* map, uint8_t* dst,
                                          uint64_t* bar, int l, int g, int r, int t0, int N, int j0,
                                          int lane) {
  const KvDev& kv = a.kv;
  if (lane == 0) tc::mbar_arrive_expect_tx(bar, kTileBytes);
  __syncwarp();
  const int hf = lane & 1;
  if (kv.page_size == 0) {
    if (lane < 2) {
      const int32_t y = int32_t((int64_t(l) * kv.Hkv + g) * kv.n_tot + t0 + j0);
      tc::tma_load_2d(dst + hf * kTileHalf, map, bar, hf * 64, y);
    }
  } else {
    const int ps = kv.page_size;
    const int i = lane >> 1;  // page of the tile
    if (i < kKT / ps) {
      const int lp = min((j0 + i * ps) / ps, (N - 1) / ps);  // tail pages repeat the last one (masked)
      const int page = kv.page_table[int64_t(r) * kv.max_pages + lp];
      const int32_t y = int32_t(((int64_t(l) * kv.num_pages + page) * kv.Hkv + g) * ps);
      tc::tma_load_2d(dst + hf * kTileHalf + i * ps * 128, map, bar, hf * 64, y);
    }
  }
}

// Agreement of the 256 softmax threads (named barrier 1 with an AND
// reduction): every thread arrives, so all of them take the same branch.
__device__ __forceinline__ bool softmax_all(bool pred) {
  uint32_t out;
  asm volatile(
      "{\n.reg .pred pi, po;\nsetp.ne.u32 pi, %1, 0;\nbar.red.and.pred po, 1, %2, pi;\nselp.u32 %0, 1, 0, po;\n}\n"
      : "=r"(out)
      : "r"(uint32_t(pred)), "n"(kSoftThreads)
      : "memory");
  return out != 0;
}

__global__ void __launch_bounds__(kThreads, 1)
    refresh_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                      const __grid_constant__ CUtensorMap qmap, const __grid_constant__ RefArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const Smem s = carve(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const KvDev& kv = a.kv;
  const int G = kv.G, Hq = kv.Hq;
  const int qrows = a.rows_per_tile * G;          // rows the query box fills

  if (tid == 0) {
    for (int i = 0; i < kKStages; ++i) {
      tc::mbar_init(&s.kfull[i], 1);
      tc::mbar_init(&s.kempty[i], 1);
    }
    for (int i = 0; i < kVStages; ++i) {
      tc::mbar_init(&s.vfull[i], 1);
      tc::mbar_init(&s.vempty[i], 1);
    }
    for (int i = 0; i < kSBufs; ++i) {
      tc::mbar_init(&s.sfull[i], 1);
      // per buffer, so the softmax can never be two phases ahead of the MMA's
      // wait: P(t+3) needs S(t+3), issued only after P(t) V(t) has completed
      tc::mbar_init(&s.pfull[i], kSoftThreads);
      tc::mbar_init(&s.pvdone[i], 1);
    }
    for (int i = 0; i < kQBufs; ++i) {
      tc::mbar_init(&s.qfull[i], 1);   // the loader's expect-tx (or plain arrive at the end)
      // the S thread's commit + the P.V thread's, softmax's and V warp's reads of the item
      tc::mbar_init(&s.qempty[i], 4);
    }
    tc::mbar_init(s.ofull, 1);
    tc::mbar_init(s.oempty, kSoftThreads);
    tc::mbar_init(&s.mdone[0], 1);
    tc::mbar_init(&s.mdone[1], 1);
    *s.abort = 0;
    for (int i = 0; i < 4; ++i) s.counters[i] = 0;
    tc::fence_barrier_init();
    tc::prefetch_tensormap(&kmap);
    tc::prefetch_tensormap(&vmap);
    tc::prefetch_tensormap(&qmap);
  }
  if (warp == 1) tc::tmem_alloc(s.tmem_slot, kTmemCols);
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *s.tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------- loads (warp 0)
    uint32_t nk = 0, T = 0;
    bool ok = true;
    for (uint32_t n = 0; ok; ++n) {
      int u = 0;
      if (lane == 0) {
        u = n == 0 ? int(blockIdx.x) : int(gridDim.x) + atomicAdd(a.next_item, 1);
        if (u >= a.n_items) u = -1;
      }
      u = __shfl_sync(0xffffffffu, u, 0);
      const Item it = decode_item(a, u < 0 ? 0 : u);
      const int nt = u < 0 ? 0 : item_tiles(a, it);
      const int t0 = a.b.tok_off[it.r], N = a.b.tok_off[it.r + 1] - t0;
      int my_pos[kRows / 32];  // positions of the item's rows, loaded before the buffer is free
#pragma unroll
      for (int k = 0; k < kRows / 32; ++k) {
        const int i = lane + 32 * k;
        my_pos[k] = (u >= 0 && i < it.cnt) ? a.idx[it.i0 + i] : -1;
      }
      const int qs = n & 1;
      if (!__all_sync(0xffffffffu, wait_or_abort(&s.qempty[qs], ((n >> 1) & 1) ^ 1, s.abort))) {
        if (lane == 0) raise_abort(a, s, tc::kSiteLoad);
        break;
      }
#pragma unroll
      for (int k = 0; k < kRows / 32; ++k) s.pos[qs * kRows + lane + 32 * k] = my_pos[k];
      if (lane == 0) {
        volatile int* rec = s.rec + qs * kRecInts;
        rec[0] = u;
        rec[1] = it.l;
        rec[2] = it.g;
        rec[3] = it.r;
        rec[4] = it.i0;
        rec[5] = it.cnt;
        rec[6] = nt;
        rec[7] = N;
        rec[8] = t0;
      }
      __threadfence_block();
      __syncwarp();  // the lanes' positions are ordered before lane 0's release below
      if (lane == 0) {
        if (u < 0) {
          tc::mbar_arrive(&s.qfull[qs]);  // no more work: the others stop at this buffer
        } else {
          tc::mbar_arrive_expect_tx(&s.qfull[qs], 2u * 128u * uint32_t(qrows));
          for (int hf = 0; hf < 2; ++hf)
            tc::tma_load_3d(s.q + qs * kQBytes + hf * kQHalf, &qmap, &s.qfull[qs], hf * 64,
                            it.g * G, it.l * a.n_sel + max(it.i0, 0));
        }
      }
      if (u < 0) break;
      for (int t = 0; t < nt; ++t, ++T) {
        const int sk = T % kKStages;
        if (!__all_sync(0xffffffffu, wait_or_abort(&s.kempty[sk], ((T / kKStages) & 1) ^ 1, s.abort))) {
          if (lane == 0) raise_abort(a, s, tc::kSiteLoad);
          ok = false;
          break;
        }
        load_tile(a, &kmap, s.k + sk * kTileBytes, &s.kfull[sk], it.l, it.g, it.r, t0, N, t * kKT, lane);
        ++nk;
      }
    }
    if (lane == 0) s.counters[0] = nk;
  } else if (warp == kVWarp) {
    // --------------------------------------------------- V loads (warp 10)
    // on a warp of their own: a V stage frees only once its P.V has
    // completed, and waiting for it must not hold back the K tiles and the
    // next item's query tile
    uint32_t nv = 0, T = 0;
    for (uint32_t n = 0;; ++n) {
      const int qs = n & 1;
      if (!__all_sync(0xffffffffu, wait_or_abort(&s.qfull[qs], (n >> 1) & 1, s.abort))) {
        if (lane == 0) raise_abort(a, s, tc::kSiteLoad);
        break;
      }
      const volatile int* rec = s.rec + qs * kRecInts;
      const int u = rec[0], l = rec[1], g = rec[2], r = rec[3], nt = rec[6], N = rec[7], t0 = rec[8];
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&s.qempty[qs]);  // this warp is done with the record
      if (u < 0) break;
      bool ok = true;
      for (int t = 0; t < nt; ++t, ++T) {
        const int sv = T % kVStages;
        if (!__all_sync(0xffffffffu, wait_or_abort(&s.vempty[sv], ((T / kVStages) & 1) ^ 1, s.abort))) {
          if (lane == 0) raise_abort(a, s, tc::kSiteLoad);
          ok = false;
          break;
        }
        load_tile(a, &vmap, s.v + sv * kTileBytes, &s.vfull[sv], l, g, r, t0, N, t * kKT, lane);
        ++nv;
      }
      if (!ok) break;
    }
    if (lane == 0) s.counters[1] = nv;
  } else if (warp == 1 && lane == 0) {
    // ---------------------------------------------------------- MMA: S = Q K^T
    // S(t) goes to buffer t % kSBufs once P(t-3) V(t-3), which read that
    // buffer's P, has completed (possibly of an earlier item); so this thread
    // runs up to two tiles ahead of the P.V thread
    uint32_t ck = 0, T = 0;
    bool ok = true;
    const uint32_t idesc_s = tc::idesc_bf16(kRows, kKT);
    for (uint32_t n = 0; ok; ++n) {
      const int qs = n & 1;
      if (!wait_or_abort(&s.qfull[qs], (n >> 1) & 1, s.abort)) { ok = false; break; }
      if (s.rec[qs * kRecInts] < 0) break;
      const int nt = s.rec[qs * kRecInts + 6];
      const uint32_t q_addr = tc::smem_u32(s.q + qs * kQBytes);
      tc::tc_fence_after();
      for (int t = 0; t < nt; ++t) {
        const uint32_t Ts = T + t;
        const int b = Ts % kSBufs, sk = Ts % kKStages;
        if (Ts >= uint32_t(kSBufs) && !wait_or_abort(&s.pvdone[b], ((Ts / kSBufs) - 1) & 1, s.abort)) {
          ok = false;
          break;
        }
        if (!wait_or_abort(&s.kfull[sk], (Ts / kKStages) & 1, s.abort)) { ok = false; break; }
        ++ck;
        tc::tc_fence_after();
        const uint32_t k_addr = tc::smem_u32(s.k + sk * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk & 3) * 32;
          tc::mma_bf16(tmem + b * kSCols, tc::desc_sw128(q_addr + (kk >> 2) * kQHalf + off),
                       tc::desc_sw128(k_addr + (kk >> 2) * kTileHalf + off), idesc_s, kk > 0);
        }
        tc::mma_commit(&s.sfull[b]);
        tc::mma_commit(&s.kempty[sk]);
      }
      if (!ok) break;
      tc::mma_commit(&s.qempty[qs]);  // every S of this item is issued
      T += nt;
    }
    if (!ok) raise_abort(a, s, tc::kSiteMma);
    s.counters[2] = ck;
    tc::mma_commit(&s.mdone[0]);  // every MMA issued above has completed once this arrives
    tc::mbar_wait(&s.mdone[0], 0);
  } else if (warp == kPvWarp && lane == 0) {
    // -------------------------------------------------------- MMA: O += P V
    uint32_t cv = 0, T = 0;
    bool ok = true;
    const uint32_t idesc_o = tc::idesc_bf16(kRows, kD, /*b_mn_major=*/true);
    for (uint32_t n = 0; ok; ++n) {
      const int qs = n & 1;
      if (!wait_or_abort(&s.qfull[qs], (n >> 1) & 1, s.abort)) { ok = false; break; }
      const int u = s.rec[qs * kRecInts], nt = s.rec[qs * kRecInts + 6];
      tc::mbar_arrive(&s.qempty[qs]);  // this thread is done with the record
      if (u < 0) break;
      for (int t = 0; t < nt; ++t) {
        const uint32_t Tc = T + t;
        const int b = Tc % kSBufs, sv = Tc % kVStages;
        if (!wait_or_abort(&s.vfull[sv], (Tc / kVStages) & 1, s.abort)) { ok = false; break; }
        ++cv;
        if (!wait_or_abort(&s.pfull[b], (Tc / kSBufs) & 1, s.abort)) { ok = false; break; }
        // O of the previous item must have been read out before P(0) V(0) overwrites it
        if (t == 0 && n > 0 && !wait_or_abort(s.oempty, (n - 1) & 1, s.abort)) { ok = false; break; }
        tc::tc_fence_after();
        const uint32_t v_addr = tc::smem_u32(s.v + sv * kTileBytes);
        const uint32_t pb = tmem + b * kSCols + kPCol;
#pragma unroll
        for (int kk = 0; kk < kKT / 16; ++kk)  // O += P(t) V(t)
          tc::mma_bf16_ts(tmem + kOCol, pb + kk * 8, tc::desc_sw128_mn(v_addr + kk * 2048, kTileHalf),
                          idesc_o, t > 0 || kk > 0);
        tc::mma_commit(&s.pvdone[b]);
        tc::mma_commit(&s.vempty[sv]);
      }
      if (!ok) break;
      T += nt;
      tc::mma_commit(s.ofull);  // O of this item is complete once this arrives
    }
    if (!ok) raise_abort(a, s, tc::kSiteMma);
    s.counters[3] = cv;
    tc::mma_commit(&s.mdone[1]);
    tc::mbar_wait(&s.mdone[1], 0);
  } else if (warp >= 2 && warp < kVWarp) {
    // -------------------------------------------------------------- softmax
    const int et = tid - 64;                             // 0..255
    const int hh = et >> 7;                              // half of the key tile / of O
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;                 // TMEM lane = query row of the tile
    const uint32_t lane_base = uint32_t(quarter * 32) << 16;
    const uint32_t tl = tmem + lane_base;
    bool ok = true;
    uint32_t T = 0;
    for (uint32_t n = 0;; ++n) {
      const int qs = n & 1;
      // all 256 threads agree to go on, so the named barriers below stay uniform
      const bool got = wait_or_abort(&s.qfull[qs], (n >> 1) & 1, s.abort);
      if (!softmax_all(ok && got)) {
        if (ok) raise_abort(a, s, tc::kSiteLoad);
        break;
      }
      const volatile int* rec = s.rec + qs * kRecInts;
      const int u = rec[0];
      Item it;
      it.l = rec[1];
      it.g = rec[2];
      it.r = rec[3];
      it.i0 = rec[4];
      it.cnt = rec[5];
      const int nt = rec[6], N = rec[7];
      const bool row_ok = u >= 0 && row < it.cnt * G;
      const int i_row = it.i0 + (row_ok ? row / G : 0);
      const int h_row = it.g * G + (row_ok ? row % G : 0);
      int p_row = row_ok ? s.pos[qs * kRows + row / G] : -1;  // rows past the item (or the box) are fully masked
      if (p_row >= N) p_row = -1;
      asm volatile("bar.sync 1, %0;" ::"n"(kSoftThreads) : "memory");  // everyone has read the record
      if (et == 0) tc::mbar_arrive(&s.qempty[qs]);
      if (u < 0) break;

      float m_ref = -INFINITY, lsum = 0.f;  // running max (scaled, log2 units, same in both halves) and half-row sum
      for (int t = 0; t < nt; ++t) {
        const uint32_t Tc = T + t;
        const uint32_t sbuf = Tc % kSBufs;
        const uint32_t sb = tl + sbuf * kSCols;
        // the tcgen05.ld below is warp-collective: the whole warp goes on or stops
        const bool gs = __all_sync(0xffffffffu, ok && (mbar_probe(&s.sfull[sbuf], (Tc / kSBufs) & 1) ||
                                                       wait_or_abort(&s.sfull[sbuf], (Tc / kSBufs) & 1, s.abort)));
        if (!gs) {
          if (ok) raise_abort(a, s, tc::kSiteMma);
          ok = false;
        }
        float sv[64];
        float hmax = -INFINITY;
        const int j0 = t * kKT + hh * 64;
        if (gs) {
          tc::tc_fence_after();
          tc::tmem_ld64(sb + hh * 64, sv);
          if (j0 + 63 > p_row) {  // part of this half is past this row's position
#pragma unroll
            for (int i = 0; i < 64; ++i)
              if (j0 + i > p_row) sv[i] = -INFINITY;
          }
          float tm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
          for (int i = 0; i < 32; ++i) tm[i & 3] = tc::fmax3(tm[i & 3], sv[2 * i], sv[2 * i + 1]);
          hmax = fmaxf(fmaxf(tm[0], tm[1]), fmaxf(tm[2], tm[3]));
        }
        // exchange the half-row maxima (buffers alternate with the tile, so a
        // half that runs ahead never overwrites a value its partner still reads)
        float* xm = s.xmax + (Tc & 1) * 256;
        xm[hh * 128 + row] = hmax;
        asm volatile("bar.sync 1, %0;" ::"n"(kSoftThreads) : "memory");
        if (!ok) continue;
        const float tmax = fmaxf(hmax, xm[(hh ^ 1) * 128 + row]) * a.scale_log2;
        const bool need = tmax > m_ref + kRescaleLog2 || (m_ref == -INFINITY && tmax != -INFINITY);
        const float alpha = need ? tc::ex2(m_ref - tmax) : 1.f;  // 0 when m_ref is -inf
        if (need) {
          lsum *= alpha;
          m_ref = tmax;
        }
        // this half of P = 2^(S scale - m) in bf16 pairs over the upper half of S
        // (one packed FMA per pair for scale and bias, packed adds for the sum).
        // A row with no visible key yet (m = -inf) uses bias 0: its logits are
        // all -inf and its P is 0.
        const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
        const float2 nb2 = m_ref == -INFINITY ? make_float2(0.f, 0.f) : make_float2(-m_ref, -m_ref);
        float2 ls2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        {
          uint32_t pw[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float2 y = tc::ffma2(make_float2(sv[2 * i], sv[2 * i + 1]), sc2, nb2);
            const float2 pp = make_float2(tc::ex2(y.x), tc::ex2(y.y));
            ls2[i & 1] = tc::fadd2(ls2[i & 1], pp);
            __nv_bfloat162 pr = __floats2bfloat162_rn(pp.x, pp.y);
            pw[i] = *reinterpret_cast<uint32_t*>(&pr);
          }
          tc::tmem_st32u(sb + kPCol + hh * 32, pw);
        }
        const float ls[4] = {ls2[0].x, ls2[0].y, ls2[1].x, ls2[1].y};
        lsum += (ls[0] + ls[1]) + (ls[2] + ls[3]);
        if (__any_sync(0xffffffffu, need) && t > 0) {
          // P(t-1) V(t-1) must have completed before this warp rescales its half
          // of O. That buffer's next P.V needs a P this softmax has not written
          // yet, so the barrier's parity cannot alias; P(t) V(t) waits for this
          // warp's pfull arrival below.
          if (!__all_sync(0xffffffffu,
                          wait_or_abort(&s.pvdone[(Tc - 1) % kSBufs], ((Tc - 1) / kSBufs) & 1, s.abort))) {
            raise_abort(a, s, tc::kSiteMma);
            ok = false;
            continue;
          }
          tc::tc_fence_after();
          for (int c = hh * 64; c < hh * 64 + 64; c += 32) {
            float o[32];
            tc::tmem_ld32(tl + kOCol + c, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tc::tmem_st32(tl + kOCol + c, o);
          }
        }
        tc::tc_fence_before();
        tc::mbar_arrive(&s.pfull[sbuf]);
      }
      T += nt;
      // row sum = the two halves' sums (same running max in both)
      s.xsum[hh * 128 + row] = lsum;
      asm volatile("bar.sync 1, %0;" ::"n"(kSoftThreads) : "memory");
      const float total = s.xsum[row] + s.xsum[128 + row];
      // O of this item is complete once the MMA thread's per-item commit has
      // arrived (it cannot run a phase ahead: the next one needs this warp's P)
      const bool fin = __all_sync(0xffffffffu, ok && wait_or_abort(s.ofull, n & 1, s.abort));
      if (!fin && ok) {
        raise_abort(a, s, tc::kSiteFinal);
        ok = false;
      }
      if (fin) {
        tc::tc_fence_after();
        const float inv = total > 0.f ? 1.f / total : 0.f;
        __nv_bfloat16* dst = a.out + ((int64_t(it.l) * a.n_sel + i_row) * Hq + h_row) * kD;
        // This thread's 64 columns of O in one load, then its half row as
        // bf16. Each lane writes its own row, so a warp's store covers 32
        // rows: 32-byte stores (whole sectors) when the buffer allows them.
        float o[64];
        tc::tmem_ld64(tl + kOCol + hh * 64, o);
        if (row_ok && p_row >= 0) {
          uint32_t w[32];
#pragma unroll
          for (int k2 = 0; k2 < 32; ++k2) {
            __nv_bfloat162 pr = __floats2bfloat162_rn(o[2 * k2] * inv, o[2 * k2 + 1] * inv);
            w[k2] = *reinterpret_cast<uint32_t*>(&pr);
          }
          __nv_bfloat16* drow = dst + hh * 64;
          if (a.out32) {
#pragma unroll
            for (int u8 = 0; u8 < 4; ++u8)
              asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(drow + u8 * 16),
                           "r"(w[8 * u8]), "r"(w[8 * u8 + 1]), "r"(w[8 * u8 + 2]), "r"(w[8 * u8 + 3]),
                           "r"(w[8 * u8 + 4]), "r"(w[8 * u8 + 5]), "r"(w[8 * u8 + 6]), "r"(w[8 * u8 + 7])
                           : "memory");
          } else {
#pragma unroll
            for (int u4 = 0; u4 < 8; ++u4)
              *reinterpret_cast<uint4*>(drow + u4 * 8) = make_uint4(w[4 * u4], w[4 * u4 + 1], w[4 * u4 + 2], w[4 * u4 + 3]);
          }
        }
      }
      tc::tc_fence_before();
      tc::mbar_arrive(s.oempty);  // O may be overwritten by the next item
    }
  }
  __syncthreads();
  if (tid == 0) {  // drain loads issued but never consumed (only after an abort)
    for (uint32_t n = s.counters[2]; n < s.counters[0]; ++n)
      tc::mbar_wait(&s.kfull[n % kKStages], (n / kKStages) & 1);
    for (uint32_t n = s.counters[3]; n < s.counters[1]; ++n)
      tc::mbar_wait(&s.vfull[n % kVStages], (n / kVStages) & 1);
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

// Query rows [L * n_sel][Hq][d] as a 3-D map with box (64 dims, G heads,
// rows_per_tile rows): one box fills one 64-dim half of a query tile in the
// tile's row order (selected row major, head minor).
bool make_qmap(CUtensorMap* m, const KvDev& kv, const void* q_rows, int32_t n_sel, int rows_per_tile) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {cuuint64_t(kD), cuuint64_t(kv.Hq), cuuint64_t(kv.L) * cuuint64_t(n_sel)};
  cuuint64_t strides[2] = {cuuint64_t(kD) * 2, cuuint64_t(kv.Hq) * kD * 2};
  cuuint32_t box[3] = {64, cuuint32_t(kv.G), cuuint32_t(rows_per_tile)};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q_rows), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
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
                              const void* q_rows, void* out, int32_t* work_counter, int32_t* status,
                              cudaStream_t stream) {
  if (n_sel == 0) return cudaSuccess;
  CUtensorMap kmap, vmap, qmap;
  if (!make_map(&kmap, kv, kv.k) || !make_map(&vmap, kv, kv.v) ||
      !make_qmap(&qmap, kv, q_rows, n_sel, kRows / kv.G))
    return cudaErrorInvalidValue;
  RefArgs a{};
  a.kv = kv;
  a.b = b;
  a.idx = idx;
  a.idx_off = idx_off_dev;
  a.q_rows = static_cast<const __nv_bfloat16*>(q_rows);
  a.out = static_cast<__nv_bfloat16*>(out);
  a.out32 = (reinterpret_cast<uintptr_t>(out) & 31) == 0;
  a.n_sel = n_sel;
  a.rows_per_tile = kRows / kv.G;
  int blocks = 0;
  for (int r = 0; r < b.R; ++r) {
    const int kr = idx_off_host[r + 1] - idx_off_host[r];
    blocks += (kr + a.rows_per_tile - 1) / a.rows_per_tile;
  }
  a.n_blocks = blocks;
  a.n_items = blocks * kv.Hkv * kv.L;
  a.next_item = work_counter;
  a.scale_log2 = kLog2e / sqrtf(float(kD));
  a.status = status;
  if (blocks == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t err;
  if ((err = cudaGetDevice(&dev))) return err;
  if ((err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))) return err;
  int l2 = 0;
  if ((err = cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev))) return err;
  // longest-first when the whole K/V of the batch fits in half of L2 (the rest
  // holds queries and outputs), else (layer, head)-major
  const double kv_bytes = 2.0 * double(kv.L) * kv.Hkv * double(kv.n_tot) * kD * 2;
  a.blocks_major = kv_bytes <= 0.5 * double(l2) ? 1 : 0;
  if ((err = cudaFuncSetAttribute(refresh_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  int(kSmem))))
    return err;
  if ((err = cudaMemsetAsync(work_counter, 0, sizeof(int32_t), stream))) return err;
  refresh_tc_kernel<<<std::min(a.n_items, sms), kThreads, kSmem, stream>>>(kmap, vmap, qmap, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace conduit
