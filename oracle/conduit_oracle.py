"""CPU oracle for the Conduit refresh policy (test infrastructure, not product code).

This module is the slow, plain statement of what the GPU path computes. It is
test infrastructure: only the test suite, the smoke check in
``__graft_entry__`` and the CPU-baseline leg of ``bench.py`` may import it.
The product path (the CUDA library and its Python binding) never imports or
calls it, and it imports nothing from the product package.

Everything is computed in float64 with numpy; inputs are widened from the
exact values the GPU sees. Library primitives used as single steps: matrix
product (``@``), ``np.exp``, ``np.sqrt``, ``sorted``. There is no blocking,
fusion or reordering beyond what each definition states.

Notation follows the paper (Conduit, Sec. 3 and Algorithm 1):
  L   scored layers (the set \\mathcal{L}),      Hq query heads, Hkv KV heads,
  G = Hq / Hkv query heads per KV head,         d head dimension,
  Q   scoring query span (n_q rows),            N = N_vis visual tokens,
  V_j image j's token span, n_j = |V_j|,        pi(t) image of token t,
  r   refresh ratio, k budget, lambda reweighting strength.

Readings taken where the paper is silent (each is listed in the design notes):
  * the softmax of alpha_{q,t} runs over the N cached visual keys of the
    request, all images jointly (Sec. 1 says attention is normalised over a
    mixed visual prefix);
  * logits are scaled by 1/sqrt(d);
  * under grouped-query attention, H in Eq. 6 counts query heads and head h
    reads KV head floor(h / G);
  * ||V_t^{c,(l)}|| is taken over the concatenation of the Hkv cached heads
    (App. A.2 "concatenated multi-head cached value vector");
  * the budget is floor(r*N + 1e-9) so that decimal ratios land on integers;
  * TopK breaks ties in favour of the lowest token index;
  * if g_bar == 0 every c_j is 1, and K == 1 gives c_1 = 1 exactly (Sec. 3.5);
  * the refresh step writes the fresh K/V rows first, then each refreshed row
    attends causally (positions j <= p_i, itself included) to the patched
    cache.

Pins (tests/test_oracle_pins.py) tie every function here to something other
than itself: a hand-derived closed-form example (tests/golden/), brute-force
enumeration of Lemma 1, library softmax / attention routines, and the
invariants of Sec. 3.5 and App. B.2.
"""

from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np

__all__ = [
    "budget",
    "cached_key_logits",
    "softmax_over_visual_keys",
    "head_query_mean_attention",
    "softmax_with_outside_keys",
    "head_query_rms_attention",
    "value_norms",
    "throughput_score",
    "image_mean_attention",
    "image_coefficients",
    "composite_score",
    "topk_select",
    "image_quotas",
    "quota_select",
    "refresh_mask",
    "score_request",
    "staleness_iso",
    "kv_gather",
    "kv_scatter",
    "refresh_attention",
]


# --------------------------------------------------------------------------
# Sec. 3.1, Eq. 2 and Algorithm 1 (first step): the visual refresh budget.
# --------------------------------------------------------------------------
def budget(r: float, n_vis: int) -> int:
    """k = floor(r * N_vis), Eq. 2. The 1e-9 guard makes decimal r exact."""
    if not (0.0 <= r <= 1.0) or math.isnan(r):
        raise ValueError("refresh ratio r must lie in [0, 1]")
    if n_vis < 0:
        raise ValueError("N_vis must be non-negative")
    k = int(math.floor(r * n_vis + 1e-9))
    return min(k, n_vis)


# --------------------------------------------------------------------------
# Sec. 3.3, Eq. 6: cached-key query attention, averaged over heads and the
# scoring span.
# --------------------------------------------------------------------------
def cached_key_logits(q_h: np.ndarray, k_g: np.ndarray) -> np.ndarray:
    """x[q, t] = <q_q, k_t> / sqrt(d) for one query head and its KV head.

    q_h: [n_q, d] query rows of head h; k_g: [N, d] cached keys of KV head g.
    """
    d = q_h.shape[-1]
    return (q_h @ k_g.T) / math.sqrt(d)


def softmax_over_visual_keys(x: np.ndarray) -> np.ndarray:
    """alpha[q, t] = exp(x[q,t] - m_q) / sum_u exp(x[q,u] - m_q), m_q = max_u x[q,u].

    Each row is normalised over all N visual keys of the request.
    """
    m = x.max(axis=1, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=1, keepdims=True)


def softmax_with_outside_keys(x: np.ndarray, extra_lse: np.ndarray) -> np.ndarray:
    """alpha[q, t] = exp(x[q,t]) / (sum_u exp(x[q,u]) + exp(extra_lse[q])).

    The full-context reading of the softmax: the keys outside the visual span
    (text, query span) stay in the denominator, entering through the natural
    log of their summed exponentials, extra_lse[q] (-inf: no such keys, which
    gives softmax_over_visual_keys). Shifted by c_q = max(max_u x[q,u], extra_lse[q]).
    """
    c = np.maximum(x.max(axis=1), extra_lse)[:, None]
    e = np.exp(x - c)
    return e / (e.sum(axis=1, keepdims=True) + np.exp(extra_lse[:, None] - c))


def _attention_rows(q_l, k_l, extra_lse_l=None):
    """alpha of every query head of one layer, [Hq, n_q, N] (head h reads KV head h // G)."""
    hq = q_l.shape[0]
    hkv = k_l.shape[0]
    if hq % hkv != 0:
        raise ValueError("Hq must be a multiple of Hkv")
    group = hq // hkv
    out = []
    for h in range(hq):
        x = cached_key_logits(q_l[h], k_l[h // group])
        if extra_lse_l is None:
            out.append(softmax_over_visual_keys(x))
        else:
            out.append(softmax_with_outside_keys(x, np.asarray(extra_lse_l[h], dtype=np.float64)))
    return np.stack(out)


def head_query_mean_attention(q_l: np.ndarray, k_l: np.ndarray,
                              extra_lse_l: Optional[np.ndarray] = None) -> np.ndarray:
    """a_t^{(l)} = (1 / (|Q| H)) sum_q sum_h alpha_{q,t,l,h}, Eq. 6.

    q_l: [Hq, n_q, d] scoring queries of one layer; k_l: [Hkv, N, d] cached keys.
    Query head h reads KV head h // G. extra_lse_l: optional [Hq, n_q]
    outside-key log-sum-exps (full-context softmax).
    """
    hq, n_q, _ = q_l.shape
    alpha = _attention_rows(q_l, k_l, extra_lse_l)
    return alpha.sum(axis=(0, 1)) / (n_q * hq)


def head_query_rms_attention(q_l: np.ndarray, k_l: np.ndarray,
                             extra_lse_l: Optional[np.ndarray] = None) -> np.ndarray:
    """abar_t^{(l)} = sqrt((1 / (|Q| H)) sum_q sum_h alpha_{q,t,l,h}^2), Eq. 4.

    The RMS of the cached-key attention over the same query rows and heads
    that Eq. 6 averages over (Eq. 4 states it for one head; the heads enter
    as Eq. 6 takes them).
    """
    hq, n_q, _ = q_l.shape
    alpha = _attention_rows(q_l, k_l, extra_lse_l)
    return np.sqrt((alpha * alpha).sum(axis=(0, 1)) / (n_q * hq))


def value_norms(v_l: np.ndarray) -> np.ndarray:
    """v_t^{(l)} = ||V_t^{c,(l)}||_2 on the concatenated Hkv*d value vector.

    v_l: [Hkv, N, d] -> [N].
    """
    hkv, n, d = v_l.shape
    concat = np.transpose(v_l, (1, 0, 2)).reshape(n, hkv * d)
    return np.sqrt((concat * concat).sum(axis=1))


# --------------------------------------------------------------------------
# Sec. 3.3, Eq. 7: multi-layer throughput score.
# --------------------------------------------------------------------------
def throughput_score(a: np.ndarray, vn: np.ndarray) -> np.ndarray:
    """s_t = (1/|L|) sum_l a_t^{(l)} v_t^{(l)}; a, vn: [|L|, N] -> [N]."""
    return (a * vn).sum(axis=0) / a.shape[0]


# --------------------------------------------------------------------------
# Sec. 3.4, Eqs. 8 and 9: image-level relevance amplification.
# --------------------------------------------------------------------------
def image_mean_attention(a: np.ndarray, img_off: Sequence[int]) -> np.ndarray:
    """g_j = (1 / (|L| n_j)) sum_l sum_{t in V_j} a_t^{(l)}, Eq. 8.

    img_off: [K+1] request-local token offsets of contiguous image spans.
    """
    n_layers = a.shape[0]
    k_img = len(img_off) - 1
    g = np.zeros(k_img, dtype=np.float64)
    for j in range(k_img):
        lo, hi = int(img_off[j]), int(img_off[j + 1])
        if hi <= lo:
            raise ValueError("image spans must be non-empty")
        g[j] = a[:, lo:hi].sum() / (n_layers * (hi - lo))
    return g


def image_coefficients(g: np.ndarray, lam: float) -> np.ndarray:
    """c_j = (1 - lambda) + lambda * g_j / g_bar, g_bar = mean_j g_j, Eq. 9.

    K == 1 gives c_1 = 1 for every lambda (Sec. 3.5, single-image limit); a
    zero g_bar (all attention underflowed) also gives c = 1.
    """
    if not (0.0 <= lam <= 1.0):
        raise ValueError("lambda must lie in [0, 1]")
    k_img = g.shape[0]
    if k_img == 1:
        return np.ones(1, dtype=np.float64)
    g_bar = g.sum() / k_img
    if g_bar == 0.0:
        return np.ones(k_img, dtype=np.float64)
    return (1.0 - lam) + lam * g / g_bar


# --------------------------------------------------------------------------
# Sec. 3.5, Eqs. 10 and 11: composite score and one global top-k.
# --------------------------------------------------------------------------
def composite_score(s: np.ndarray, c: np.ndarray, img_off: Sequence[int]) -> np.ndarray:
    """s_hat_t = s_t * c_{pi(t)}, Eq. 10."""
    s_hat = np.empty_like(s)
    for j in range(len(img_off) - 1):
        lo, hi = int(img_off[j]), int(img_off[j + 1])
        s_hat[lo:hi] = s[lo:hi] * c[j]
    return s_hat


def topk_select(s_hat: np.ndarray, k: int) -> np.ndarray:
    """T = TopK_t(s_hat, k), Eq. 11; ties go to the lowest index.

    Returns the selected token indices in ascending order (int64).
    """
    n = s_hat.shape[0]
    if not (0 <= k <= n):
        raise ValueError("budget k must lie in [0, N]")
    order = sorted(range(n), key=lambda t: (-float(s_hat[t]), t))
    return np.array(sorted(order[:k]), dtype=np.int64)


# --------------------------------------------------------------------------
# App. D.3 ("explicit" cross-image variant): quotas k_j proportional to
# c_j n_j, then a top-k_j inside each image.
# --------------------------------------------------------------------------
def image_quotas(c: np.ndarray, n: Sequence[int], k: int) -> np.ndarray:
    """k_j proportional to c_j n_j with sum_j k_j = k and 0 <= k_j <= n_j.

    The paper states the proportionality only; the integer rule taken here is
    the largest-remainder (Hamilton) rule in float64: w_j = c_j n_j,
    W = w_0 + w_1 + ... (left to right), ideal_j = (kk w_j) / W over the
    images still open; an image whose ideal exceeds n_j is closed at n_j and
    the rest of the budget is shared again; otherwise k_j = floor(ideal_j)
    and the leftover units go to the largest remainders ideal_j - floor,
    ties to the lower image index. If every open image has weight 0, the
    weights become n_j (size-proportional).
    """
    n = [int(x) for x in n]
    k_img = len(n)
    if not (0 <= k <= sum(n)):
        raise ValueError("budget k must lie in [0, sum n_j]")
    quota = [0] * k_img
    open_ = [j for j in range(k_img)]
    kk = int(k)
    while True:
        w = {j: float(np.float64(c[j]) * float(n[j])) for j in open_}
        if all(w[j] == 0.0 for j in open_):
            w = {j: float(n[j]) for j in open_}
        total = 0.0
        for j in open_:
            total = total + w[j]
        ideal = {j: (float(kk) * w[j]) / total if total > 0 else 0.0 for j in open_}
        over = [j for j in open_ if ideal[j] > n[j]]
        if over:
            for j in over:
                quota[j] = n[j]
                kk -= n[j]
            open_ = [j for j in open_ if j not in over]
            continue
        base = {j: int(math.floor(ideal[j])) for j in open_}
        left = kk - sum(base.values())
        order = sorted(open_, key=lambda j: (-(ideal[j] - base[j]), j))
        for j in open_:
            quota[j] = base[j]
        for j in order[:left]:
            quota[j] += 1
        return np.array(quota, dtype=np.int64)


def quota_select(s: np.ndarray, c: np.ndarray, img_off: Sequence[int], k: int) -> dict:
    """The explicit variant for one request: quotas from image_quotas, then in
    image j the k_j tokens of largest s_t (Eq. 7; c_j is constant inside an
    image, so it decides only the quotas), ties to the lowest index.

    Returns the quotas and the ascending request-local indices.
    """
    n = [int(img_off[j + 1]) - int(img_off[j]) for j in range(len(img_off) - 1)]
    quota = image_quotas(c, n, k)
    idx = []
    for j in range(len(n)):
        lo, hi = int(img_off[j]), int(img_off[j + 1])
        idx.extend((lo + topk_select(np.asarray(s[lo:hi], dtype=np.float64), int(quota[j]))).tolist())
    return {"quota": quota, "idx": np.array(sorted(idx), dtype=np.int64)}


def score_request(q: np.ndarray, k: np.ndarray, v: Optional[np.ndarray],
                  img_off: Sequence[int], layers: Optional[Sequence[int]] = None,
                  vnorm: Optional[np.ndarray] = None, statistic: str = "mean",
                  use_value_norm: bool = True, extra_lse: Optional[np.ndarray] = None) -> dict:
    """The query-conditioned scoring pass for one request (Algorithm 1, scoring loop).

    q: [L, Hq, n_q, d]; k, v: [L, Hkv, N, d] (anything whose [l] gives one
    layer's array); layers: the scored layer set (default all layers, App. A.2).
    vnorm: optional stored norms [L, N] (Sec. 4.3 and App. C.2: the value norm
    depends only on the cached content, so it may be kept per token and layer
    from cache construction); when given, v_t^{(l)} = vnorm[l, t] and v is not
    read (it may be None).
    statistic: "mean" (Eq. 6, the deployed policy) or "rms" (Eq. 4) for the
    attention factor of s; A and g always use the mean.
    use_value_norm: False drops the value norm from s (the factor ablation of
    Sec. 4.4: s ranks by attention alone; v may be None).
    extra_lse: optional [L, Hq, n_q] outside-key log-sum-exps (full-context
    softmax, see softmax_with_outside_keys).
    Returns a, vn ([|L|, N]), stat (the factor used in s), s, A ([N]) and g ([K]).
    """
    f64 = lambda x: np.asarray(x, dtype=np.float64)
    if statistic not in ("mean", "rms"):
        raise ValueError("statistic must be 'mean' or 'rms'")
    if layers is None:
        layers = list(range(len(k)))
    ex = (lambda l: None) if extra_lse is None else (lambda l: f64(extra_lse[l]))
    a = np.stack([head_query_mean_attention(f64(q[l]), f64(k[l]), ex(l)) for l in layers])
    if statistic == "rms":
        stat = np.stack([head_query_rms_attention(f64(q[l]), f64(k[l]), ex(l)) for l in layers])
    else:
        stat = a
    if not use_value_norm:
        vn = np.ones_like(a)
    elif vnorm is None:
        vn = np.stack([value_norms(f64(v[l])) for l in layers])
    else:
        vn = np.stack([f64(vnorm[l]) for l in layers])
    s = throughput_score(stat, vn)
    attn_sum = a.sum(axis=0)
    g = image_mean_attention(a, img_off)
    return {"a": a, "vn": vn, "stat": stat, "s": s, "A": attn_sum, "g": g}


def refresh_mask(q: np.ndarray, k: np.ndarray, v: np.ndarray, img_off: Sequence[int],
                 r: Optional[float] = None, lam: float = 1.0,
                 layers: Optional[Sequence[int]] = None,
                 k_budget: Optional[int] = None) -> dict:
    """Algorithm 1 end to end for one request: budget, scores, c_j, s_hat, TopK, mask.

    Either r (Eq. 2) or an explicit k_budget is given. k == 0 returns the
    all-zero mask without running the scoring pass, as Algorithm 1 does.
    """
    n = np.asarray(k[0]).shape[1]
    kk = budget(r, n) if k_budget is None else int(k_budget)
    if kk == 0:
        return {"k": 0, "idx": np.zeros(0, dtype=np.int64), "mask": np.zeros(n, dtype=np.uint8)}
    sc = score_request(q, k, v, img_off, layers)
    c = image_coefficients(sc["g"], lam)
    s_hat = composite_score(sc["s"], c, img_off)
    idx = topk_select(s_hat, kk)
    mask = np.zeros(n, dtype=np.uint8)
    mask[idx] = 1
    out = dict(sc)
    out.update({"k": kk, "c": c, "s_hat": s_hat, "idx": idx, "mask": mask})
    return out


# --------------------------------------------------------------------------
# App. D (Monte Carlo staleness estimator, isotropic): the error a refresh
# set T leaves, under sampled stale value displacements.
# --------------------------------------------------------------------------
def staleness_iso(q: np.ndarray, k: np.ndarray, v: np.ndarray, refreshed: np.ndarray,
                  z: np.ndarray, kappa: float) -> float:
    """E_iso(T) = sum_{l, h, q} (1/M) sum_m || sum_{t not in T} alpha_{q,t} xi_t^(m) ||^2.

    xi_t^(m) = kappa ||V_t|| / sqrt(d) * z_t^(m), so xi ~ N(0, kappa^2 ||V_t||^2 / d I)
    with z the standard normal draws (an input, the random numbers the
    estimator uses). Readings: xi is drawn per layer, KV head and token with
    ||V_t|| that head's value norm and d its dimension (the local model of
    Sec. 3.2 is one layer and head), the G query heads of a KV group read the
    same xi, alpha is the cached-key softmax over all N visual keys (Eq. 6's
    alpha), and the functional is summed over the layers, query heads and
    scoring rows.
    q: [L, Hq, n_q, d]; k, v: [L, Hkv, N, d]; refreshed: [N] (1 = in T);
    z: [M, L, Hkv, N, d].
    """
    f64 = lambda x: np.asarray(x, dtype=np.float64)
    n_m = z.shape[0]
    n_layers, hq = len(k), np.asarray(q[0]).shape[0]
    keep = 1.0 - f64(refreshed)
    total = 0.0
    for l in range(n_layers):
        q_l, k_l, v_l = f64(q[l]), f64(k[l]), f64(v[l])
        hkv, n, d = k_l.shape
        group = hq // hkv
        for g in range(hkv):
            scale = kappa * np.sqrt((v_l[g] * v_l[g]).sum(axis=1)) / math.sqrt(d)   # [N]
            xi = f64(z[:, l, g]) * (scale * keep)[None, :, None]                    # [M, N, d]
            for h in range(g * group, (g + 1) * group):
                alpha = softmax_over_visual_keys(cached_key_logits(q_l[h], k_l[g]))  # [n_q, N]
                for m in range(n_m):
                    r = alpha @ xi[m]                                                # [n_q, d]
                    total += (r * r).sum() / n_m
    return float(total)


# --------------------------------------------------------------------------
# Selective recompute (Sec. 3.1, Sec. 3.5 refresh mask, Sec. 4.3 serving):
# gather the selected rows, write fresh K/V back, causal attention of the
# refreshed rows over the patched cache.
# --------------------------------------------------------------------------
def kv_gather(cache: np.ndarray, idx: Sequence[int]) -> np.ndarray:
    """rows[l, i, g, :] = cache[l, g, idx[i], :]; cache [L, Hkv, N, d] -> [L, k, Hkv, d]."""
    idx = np.asarray(idx, dtype=np.int64)
    return np.transpose(cache[:, :, idx, :], (0, 2, 1, 3)).copy()


def kv_scatter(cache: np.ndarray, idx: Sequence[int], rows: np.ndarray) -> np.ndarray:
    """Returns a copy of cache with cache[l, g, idx[i], :] = rows[l, i, g, :]."""
    out = np.array(cache, copy=True)
    for i, t in enumerate(np.asarray(idx, dtype=np.int64)):
        out[:, :, t, :] = rows[:, i, :, :]
    return out


def refresh_attention(q_rows: np.ndarray, k_patched: np.ndarray, v_patched: np.ndarray,
                      idx: Sequence[int]) -> np.ndarray:
    """O[l, i, h] = sum_{j <= p_i} softmax_j(<q[l,i,h], K'[l,g(h),j]> / sqrt(d)) V'[l,g(h),j].

    q_rows: [L, k, Hq, d] fresh queries of the refreshed rows; k_patched,
    v_patched: [L, Hkv, N, d] caches after the scatter; p_i = idx[i].
    """
    q_rows = np.asarray(q_rows, dtype=np.float64)
    kp = np.asarray(k_patched, dtype=np.float64)
    vp = np.asarray(v_patched, dtype=np.float64)
    n_layers, n_sel, hq, d = q_rows.shape
    hkv = kp.shape[1]
    group = hq // hkv
    out = np.zeros_like(q_rows)
    for l in range(n_layers):
        for i, p in enumerate(np.asarray(idx, dtype=np.int64)):
            for h in range(hq):
                g = h // group
                x = (kp[l, g, : p + 1, :] @ q_rows[l, i, h]) / math.sqrt(d)
                w = np.exp(x - x.max())
                w = w / w.sum()
                out[l, i, h] = w @ vp[l, g, : p + 1, :]
    return out
