"""Shared helpers of the GPU parity tests: run the C-ABI path and the CPU
oracle on the same seeded inputs and compare them under the stated bar.

Tolerances (written here once, used by every parity test):
  scores s, A, g   |gpu - ref| <= rtol |ref| + 1e-7 max|ref|,
                   rtol = 1e-3 for bf16 inputs, 1e-5 for fp32 inputs
  selection        |T_gpu| = k and T_gpu, T_ref agree outside the band of
                   tokens whose oracle s_hat lies within rtol of the k-th value
  gather/scatter   bitwise (they copy the given rows)
  refresh output   bf16: <= 2e-2 absolute + 2^-8 relative (the output is stored in
                   bf16, whose half-ulp is 2^-8 of the value); fp32: 1e-5
                   relative + 1e-6 absolute
"""

from __future__ import annotations

import math

import numpy as np
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

RTOL = {torch.bfloat16: 1e-3, torch.float32: 1e-5}


def assert_scores_close(gpu, ref, rtol, what="score"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape
    floor = 1e-7 * float(np.abs(ref).max()) if ref.size else 0.0
    err = np.abs(gpu - ref)
    bad = err > rtol * np.abs(ref) + floor
    if bad.any():
        i = int(np.argmax(err / (np.abs(ref) + floor + 1e-300)))
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} outside tolerance; "
                             f"worst at {i}: gpu {gpu[i]!r} ref {ref[i]!r}")


def assert_selection_ok(idx_gpu, mask_gpu, s_hat_ref, idx_ref, k, rtol):
    idx_gpu = np.asarray(idx_gpu, dtype=np.int64)
    assert idx_gpu.size == k, (idx_gpu.size, k)
    assert np.all(np.diff(idx_gpu) > 0), "indices must be strictly ascending"
    if mask_gpu is not None:
        m = np.asarray(mask_gpu)
        assert int(m.sum()) == k and np.all(m[idx_gpu] == 1)
    if k == 0:
        return
    kth = np.sort(s_hat_ref)[::-1][k - 1]
    band = np.abs(s_hat_ref - kth) <= rtol * abs(kth) + 1e-30
    outside_gpu = set(idx_gpu.tolist()) - set(np.nonzero(band)[0].tolist())
    outside_ref = set(np.asarray(idx_ref).tolist()) - set(np.nonzero(band)[0].tolist())
    assert outside_gpu == outside_ref, (
        f"selection differs outside the boundary band: "
        f"{sorted(outside_gpu ^ outside_ref)[:10]}")


def oracle_requests(inputs, lam=1.0, layers=None, budgets=None, requests=None):
    """Oracle Algorithm 1 per request on the same inputs (float64 copies)."""
    tok = inputs["tok_off"].tolist()
    R = len(tok) - 1
    out = {}
    for r in (range(R) if requests is None else requests):
        view = synth.request_view(inputs, r)
        kk = budgets[r] if budgets is not None else O.budget(inputs["ratios"][r], tok[r + 1] - tok[r])
        sc = O.score_request(view["q"], view["k"], view["v"], view["img_off"], layers)
        c = O.image_coefficients(sc["g"], lam)
        s_hat = O.composite_score(sc["s"], c, view["img_off"])
        idx = O.topk_select(s_hat, kk)
        out[r] = dict(sc, c=c, s_hat=s_hat, idx=idx, k=kk, view=view)
    return out


def compare_score_select(pipe, inputs, ref, rtol):
    tok = inputs["tok_off"].tolist()
    rio = inputs["req_img_off"].tolist()
    s = pipe.s.double().cpu().numpy()
    A = pipe.attn_sum.double().cpu().numpy()
    g = pipe.g.double().cpu().numpy()
    coeff = pipe.coeff.double().cpu().numpy()
    idx = pipe.idx.cpu().numpy()
    mask = pipe.mask.cpu().numpy()
    off = pipe.idx_off.tolist()
    for r, o in ref.items():
        t0, t1 = tok[r], tok[r + 1]
        assert_scores_close(s[t0:t1], o["s"], rtol, f"s (request {r})")
        assert_scores_close(A[t0:t1], o["A"], rtol, f"A (request {r})")
        assert_scores_close(g[rio[r]:rio[r + 1]], o["g"], rtol, f"g (request {r})")
        assert_scores_close(coeff[rio[r]:rio[r + 1]], o["c"], 2 * rtol, f"c (request {r})")
        assert_selection_ok(idx[off[r]:off[r + 1]], mask[t0:t1], o["s_hat"], o["idx"], o["k"], rtol)


# ------------------------------------------------ quotas decided by floats
def quota_margins(c, n, k):
    """The fp64 largest-remainder apportionment of App. D.3 (the oracle's rule,
    restated step by step) together with how close each of its decisions came
    to flipping, relative to the ideal share it was taken on.

    Returns (quota, per-image margin, cap margin): an image's margin is the
    smallest of the distance of its ideal share to an integer and of its
    remainder to the remainder on the other side of the leftover cutoff,
    over the largest ideal share of the round; the cap margin is the
    smallest distance of any open image's ideal share to its size, relative
    to that share (a cap decision changes the budget left to every other
    image).
    """
    n = [int(x) for x in n]
    K = len(n)
    quota = [0] * K
    margin = [math.inf] * K
    cap_margin = math.inf
    open_ = list(range(K))
    kk = int(k)
    while True:
        w = {j: float(c[j]) * n[j] for j in open_}
        if all(w[j] == 0.0 for j in open_):
            w = {j: float(n[j]) for j in open_}
        total = sum(w[j] for j in open_)
        ideal = {j: (kk * w[j]) / total if total > 0 else 0.0 for j in open_}
        for j in open_:
            if ideal[j] > 0:
                cap_margin = min(cap_margin, abs(ideal[j] - n[j]) / ideal[j])
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
        rem = {j: ideal[j] - base[j] for j in open_}
        chosen = set(order[:left])
        last_in = rem[order[left - 1]] if left >= 1 else None
        first_out = rem[order[left]] if left < len(order) else None
        scale = max([1.0] + [ideal[j] for j in open_])
        for j in open_:
            quota[j] = base[j] + (1 if j in chosen else 0)
            other = first_out if j in chosen else last_in
            to_cut = abs(rem[j] - other) if other is not None else math.inf
            margin[j] = min(rem[j], 1.0 - rem[j], to_cut) / scale
        return np.array(quota, dtype=np.int64), np.array(margin), cap_margin


def assert_quotas_in_band(q_gpu, c_ref, n, k, rtol_c):
    """Quotas decided on the GPU from binary32 coefficients against the fp64 rule.

    The fp64 quotas of the oracle are the reference. A quota may differ from
    them by one unit, and only for an image whose fp64 decision (its floor or
    its place at the leftover cutoff) lay within 4 rtol_c of flipping, where
    rtol_c bounds the relative error of the coefficients: an ideal share
    k c_j n_j / W moves by at most about 2 rtol_c of itself, so a remainder
    by 2 rtol_c and a difference of two remainders by 4 rtol_c of the
    largest share. If a cap decision lay that close, every image may differ
    by one. The sum is always exact.
    """
    q_gpu = np.asarray(q_gpu, dtype=np.int64)
    n = np.asarray(n, dtype=np.int64)
    q_ref = O.image_quotas(np.asarray(c_ref, dtype=np.float64), n, k)
    q_rep, margin, cap_margin = quota_margins(c_ref, n, k)
    assert np.array_equal(q_rep, q_ref), "test restatement of the quota rule disagrees with the oracle"
    assert int(q_gpu.sum()) == int(k) and np.all(q_gpu >= 0) and np.all(q_gpu <= n)
    diff = np.nonzero(q_gpu != q_ref)[0]
    if diff.size == 0:
        return
    band = 4.0 * rtol_c
    assert np.all(np.abs(q_gpu - q_ref) <= 1), (q_gpu, q_ref)
    if cap_margin <= band:
        return
    far = [int(j) for j in diff if margin[j] > band]
    assert not far, f"quotas differ away from a near-tie: images {far}, gpu {q_gpu[far]}, ref {q_ref[far]}"
