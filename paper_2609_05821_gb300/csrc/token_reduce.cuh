// Per-token and per-image reductions of the scoring pass (Conduit Eqs. 6-8),
// as block-level device code shared by finalize.cu (their own launches) and
// select.cu (the fused scoring tail of conduit_score_select_topk), so that
// both produce bitwise the same s, A and g.
//   a_t^(l)  = sum_g sum_group,part pa[l][g][group][part][t] / (|Q| Hq)   Eq. 6 (head/query mean)
//   v_t^(l)  = sqrt(sum_g,part ss[l][g][part][t])                     norm of the concatenated heads
//              (or vnorm[layer id][t] when the norms come from the side cache,
//              or 1 when the score is attention alone)
//   s_t      = (1/|L|) sum_l a_t^(l) v_t^(l)                   Eq. 7
//              (with the RMS statistic, abar_t^(l) = sqrt(sum pa2 / (|Q| Hq))
//              of Eq. 4 takes the place of a_t^(l) here)
//   A_t      = sum_l a_t^(l)
//   g_j      = (1/(|L| n_j)) sum_{t in V_j} A_t                Eq. 8
#pragma once

#include "internal.cuh"

namespace conduit {

constexpr int kLayerSlots = 32;   // warps of a token block: layers l, l + 32, ...
constexpr int kTokBlock = 32;     // tokens of a block (one per lane)
constexpr int kMeanThreads = 256; // threads reducing one image mean

// Where the partials are and what the reduction computes (launch_finalize's
// arguments).
struct TokenReduceArgs {
  const float* pa;
  const float* pa2;
  const float* ss;
  const float* vnorm;
  int vmode;
  int n_layers, Hkv, Hq, rg_max, group_rows, parts;
  int64_t n_tot;
  float* s;
  float* attn_sum;
  int32_t* status;
};

// Tokens [tok0, tok0 + 32) of the batch, one per lane; warp `slot` takes
// layers slot, slot + 32, ... (coalesced loads across the 32 tokens), then
// lane t of warp 0 combines the layer slots in a fixed order, so the sums are
// deterministic and do not depend on how many warps the block has beyond
// min(32, n_layers). Ends with s[t] and attn_sum[t] written by warp 0; the
// caller synchronises the block if it reads them.
__device__ __forceinline__ void token_reduce_block(const TokenReduceArgs& f, const LayerList& layers,
                                                   const BatchDev& b, int64_t tok0,
                                                   float (*part_s)[33], float (*part_a)[33]) {
  constexpr int kBatch = 8;  // loads in flight per warp, so their latencies overlap
  const int lane = threadIdx.x & 31, slot = threadIdx.x >> 5;
  const int64_t tg = tok0 + lane;
  const int64_t n_tot = f.n_tot;
  float acc_s = 0.f, acc_a = 0.f;
  if (tg < n_tot && slot < kLayerSlots) {
    const int nss = f.Hkv * f.parts;  // value partials of one layer
    // The first layer's value partials (or side-cache norm) do not depend on
    // the request, so they go out before the request's query count is known;
    // later layers issue theirs with the attention partials. The sums below
    // run in index order either way.
    float xs0[kBatch], vn0 = 0.f;
    auto load_values = [&](int li) {
      if (f.vmode == 0) {
        const float* ss_l = f.ss + int64_t(li) * nss * n_tot + tg;
#pragma unroll
        for (int k = 0; k < kBatch; ++k) xs0[k] = k < nss ? ss_l[int64_t(k) * n_tot] : 0.f;
      } else if (f.vmode == 1) {
        vn0 = f.vnorm[int64_t(layers.ids[li]) * n_tot + tg];
      }
    };
    if (slot < f.n_layers) load_values(slot);
    // With few partials per layer (every row-group slot of every KV head, at
    // most 16), the first layer's attention partials go out before the
    // request's query count is known too: all slots are loaded, and only the
    // request's row groups are summed below.
    constexpr int kSpec = 16;
    const int per_g = f.rg_max * f.parts, nall = f.Hkv * per_g;
    const bool spec = nall <= kSpec;
    float xp[kSpec];
    if (spec && slot < f.n_layers) {
      const float* pa_l = f.pa + int64_t(slot) * nall * n_tot + tg;
#pragma unroll
      for (int i = 0; i < kSpec; ++i) xp[i] = i < nall ? pa_l[int64_t(i) * n_tot] : 0.f;
    }
    const int r = request_of(b.tok_off, b.R, tg);
    const int nq = b.q_off[r + 1] - b.q_off[r];
    const float denom = float(nq * f.Hq);
    const int rows = (f.Hq / f.Hkv) * nq;
    const int n_sl = (f.group_rows ? (rows + f.group_rows - 1) / f.group_rows : 1) * f.parts;
    const int npa = f.Hkv * n_sl;  // attention partials of one layer
    for (int li = slot; li < f.n_layers; li += kLayerSlots) {
      if (li != slot) load_values(li);
      const float* pa_l = f.pa + int64_t(li) * f.Hkv * f.rg_max * f.parts * n_tot + tg;
      auto pa_at = [&](const float* base, int q) {
        return base[(int64_t(q / n_sl) * f.rg_max * f.parts + q % n_sl) * n_tot];
      };
      float col = 0.f;
      if (spec && li == slot) {  // the same values in the same order as the loop below
        int sl = 0;
#pragma unroll
        for (int i = 0; i < kSpec; ++i) {
          if (i < nall && sl < n_sl) col += xp[i];
          if (++sl == per_g) sl = 0;
        }
      } else {
        for (int q0 = 0; q0 < npa; q0 += kBatch) {
          float x[kBatch];
#pragma unroll
          for (int k = 0; k < kBatch; ++k) x[k] = q0 + k < npa ? pa_at(pa_l, q0 + k) : 0.f;
#pragma unroll
          for (int k = 0; k < kBatch; ++k) col += x[k];
        }
      }
      const float a = col / denom;
      float stat = a;
      if (f.pa2) {  // RMS statistic (Eq. 4) over the same query rows and heads
        const float* p2_l = f.pa2 + int64_t(li) * f.Hkv * f.rg_max * f.parts * n_tot + tg;
        float col2 = 0.f;
        for (int q0 = 0; q0 < npa; q0 += kBatch) {
          float x[kBatch];
#pragma unroll
          for (int k = 0; k < kBatch; ++k) x[k] = q0 + k < npa ? pa_at(p2_l, q0 + k) : 0.f;
#pragma unroll
          for (int k = 0; k < kBatch; ++k) col2 += x[k];
        }
        stat = sqrtf(col2 / denom);
      }
      float vn;
      if (f.vmode == 2) {
        vn = 1.f;
      } else if (f.vmode == 1) {
        vn = vn0;
      } else {
        const float* ss_l = f.ss + int64_t(li) * nss * n_tot + tg;
        float sq = 0.f;
#pragma unroll
        for (int k = 0; k < kBatch; ++k) sq += xs0[k];
        for (int q0 = kBatch; q0 < nss; q0 += kBatch) {
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
  if (slot < kLayerSlots) {
    part_s[slot][lane] = acc_s;
    part_a[slot][lane] = acc_a;
  }
  __syncthreads();
  if (slot == 0 && tg < n_tot) {
    // the slots' partials are loaded eight at a time, then added in slot order
    const int used = min(kLayerSlots, f.n_layers);
    float ts = 0.f, ta = 0.f;
#pragma unroll
    for (int w0 = 0; w0 < kLayerSlots; w0 += 8) {
      float ps[8], pv[8];
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        ps[w] = w0 + w < used ? part_s[w0 + w][lane] : 0.f;
        pv[w] = w0 + w < used ? part_a[w0 + w][lane] : 0.f;
      }
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        if (w0 + w < used) {
          ts += ps[w];
          ta += pv[w];
        }
      }
    }
    const float sv = ts / float(f.n_layers);
    if (!isfinite(sv) || !isfinite(ta)) flag_status(f.status, CONDUIT_FLAG_NONFINITE);
    f.s[tg] = sv;
    f.attn_sum[tg] = ta;
  }
}

// g_j of image [lo, hi) (Eq. 8) by the 256 threads of a group (thread index
// `gt` in [0, 256) within it): strided sums, a butterfly within each warp,
// then the group's first thread adds the eight warp sums in order and writes
// *gj. warp_s holds the group's eight warp sums; `sync` synchronises exactly
// the group's threads (and orders their shared-memory accesses). attn_sum is
// read through L2, so values written earlier in the same launch by other
// blocks are seen once the writer's fence and the reader's have ordered them.
template <typename Sync>
__device__ __forceinline__ void image_mean_group(const float* attn_sum, int lo, int hi, int n_layers,
                                                 int gt, float* warp_s, float* gj, Sync sync) {
  float acc = 0.f;
  for (int t = lo + gt; t < hi; t += kMeanThreads) acc += __ldcg(attn_sum + t);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((gt & 31) == 0) warp_s[gt >> 5] = acc;
  sync();
  if (gt == 0) {
    float tot = 0.f;
    for (int w = 0; w < kMeanThreads / 32; ++w) tot += warp_s[w];
    *gj = tot / (float(n_layers) * float(hi - lo));
  }
  sync();  // warp_s may be rewritten for the next image
}

}  // namespace conduit
