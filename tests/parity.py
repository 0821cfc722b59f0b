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
