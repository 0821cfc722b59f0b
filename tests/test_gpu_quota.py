"""GPU parity of the explicit per-image quota selection (App. D.3).

On the same fp32 scores s and image means g, conduit_select_quota must return
  coeff  Eq. 9 in fp64 (the oracle) within 1e-5 relative (the kernel
         evaluates it in binary32),
  quota  the oracle's fp64 largest-remainder quotas, differing by one unit
         only for an image whose fp64 decision lay within the coefficients'
         tolerance of flipping (tests/parity.py, assert_quotas_in_band),
  idx    exactly the per-image top-k_j of s at the kernel's quotas (integer
         work on the same fp32 s: bitwise, ties to the lowest index),
  mask / s_hat consistent with idx and with s times the kernel's own c.
The crafted batches cover unequal image sizes, a cap (an image whose share
exceeds its size), all-zero weights, lambda 0 / 0.5 / 1, budgets 0 and N_r,
and tied scores. On the full multi-image and long-document workloads the
GPU's scoring pass feeds the rule, and the check is the selection bar of
tests/parity.py per image.
"""

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

from tests import parity as PT

pytestmark = pytest.mark.gpu

# relative error bound of the binary32 c_j of the kernel against Eq. 9 in fp64
# (a sum of up to 5 fp32 means, one division, one fused step: a few ulps)
C_RTOL = 1e-5


@pytest.fixture(scope="module")
def C():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import conduit
    return conduit


# requests as lists of image sizes, with budgets and g per request
CRAFTED = [
    ([1, 500, 37, 1000], 300),     # unequal sizes
    ([64, 64], 128),               # budget = N_r
    ([300], 45),                   # one image: the global top-k
    ([5, 900, 40], 200),           # image 0 is capped when its g dominates
    ([128, 128, 128], 0),          # empty budget
    ([3000, 20, 20, 20, 20], 700), # sizes past 1 024 and 8 192 keys per CTA
    ([9000, 10], 2000),
]


def _crafted(C, seed, g_mode):
    gen = torch.Generator().manual_seed(seed)
    sizes = [n for req, _ in CRAFTED for n in req]
    tok, img, rio = [0], [0], [0]
    for req, _ in CRAFTED:
        for n in req:
            img.append(img[-1] + n)
        tok.append(img[-1])
        rio.append(len(img) - 1)
    n_tot = tok[-1]
    s = torch.rand(n_tot, generator=gen) * 1e-3
    s[torch.rand(n_tot, generator=gen) < 0.2] = 5e-4      # ties: a fifth of the tokens share one score
    K = len(sizes)
    g = torch.rand(K, generator=gen) * 1e-3
    if g_mode == "dominant":
        g[rio[3]] = 1.0                                     # request 3's 5-token image dominates
    elif g_mode == "zeros":
        for r in range(len(CRAFTED)):                       # lambda = 1: c_j = 0 except one image
            g[rio[r]:rio[r + 1]] = 0.0
            g[rio[r + 1] - 1] = 1e-3
    batch = C.Batch(tok, img, rio, list(range(len(CRAFTED) + 1)), device="cuda")
    budgets = [k for _, k in CRAFTED]
    return s, g, batch, budgets, tok, img, rio


@pytest.mark.parametrize("lam", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("g_mode", ["random", "dominant", "zeros"])
def test_quota_selection_crafted(C, lam, g_mode):
    s, g, batch, budgets, tok, img, rio = _crafted(C, 11, g_mode)
    off, off_d = C.idx_offsets(budgets, "cuda")
    n_tot, K = tok[-1], len(img) - 1
    mask = torch.empty(n_tot, dtype=torch.uint8, device="cuda")
    s_hat = torch.empty(n_tot, device="cuda")
    coeff = torch.empty(K, device="cuda")
    quota = torch.empty(K, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    idx, *_ = C.conduit_select_quota(batch, s.cuda(), g.cuda(), lam, off, off_d, None, mask, s_hat,
                                     coeff, quota, status=status)
    torch.cuda.synchronize()
    assert C.conduit_read_status(status) == C.OK
    idx, mask, s_hat = idx.cpu().numpy(), mask.cpu().numpy(), s_hat.cpu().numpy()
    coeff, quota = coeff.cpu().numpy(), quota.cpu().numpy()
    s32, g32 = s.numpy(), g.numpy()
    o = off.tolist()
    for r in range(len(CRAFTED)):
        j0, j1, t0, t1 = rio[r], rio[r + 1], tok[r], tok[r + 1]
        c64 = O.image_coefficients(g32[j0:j1].astype(np.float64), lam)
        PT.assert_scores_close(coeff[j0:j1], c64, C_RTOL, f"c (request {r})")
        spans = [x - t0 for x in img[j0:j1 + 1]]
        n = np.diff(spans)
        PT.assert_quotas_in_band(quota[j0:j1], c64, n, budgets[r], C_RTOL)
        want = []
        for j in range(j1 - j0):  # the per-image top-k_j at the kernel's quotas
            lo, hi = spans[j], spans[j + 1]
            want.extend((lo + O.topk_select(s32[t0 + lo:t0 + hi].astype(np.float64), int(quota[j0 + j]))).tolist())
        assert idx[o[r]:o[r + 1]].tolist() == sorted(want), r
        m = np.zeros(t1 - t0, dtype=np.uint8)
        m[sorted(want)] = 1
        assert np.array_equal(mask[t0:t1], m)
        assert np.array_equal(s_hat[t0:t1], s32[t0:t1] * np.repeat(coeff[j0:j1], n))
    if g_mode == "dominant" and lam == 1.0:
        assert quota[rio[3]] == 5                          # capped at its 5 tokens


def test_global_coefficients_follow_eq9(C):
    """conduit_select_topk's c_j against Eq. 9 in fp64 (binary32 on the GPU)."""
    s, g, batch, budgets, tok, img, rio = _crafted(C, 12, "random")
    off, off_d = C.idx_offsets(budgets, "cuda")
    coeff = torch.empty(len(img) - 1, device="cuda")
    C.conduit_select_topk(batch, s.cuda(), g.cuda(), 0.7, off, off_d, coeff=coeff)
    torch.cuda.synchronize()
    got = coeff.cpu().numpy()
    for r in range(len(CRAFTED)):
        want = O.image_coefficients(g.numpy()[rio[r]:rio[r + 1]].astype(np.float64), 0.7)
        PT.assert_scores_close(got[rio[r]:rio[r + 1]], want, C_RTOL, f"c (request {r})")
        if rio[r + 1] - rio[r] == 1:
            assert got[rio[r]] == 1.0                      # K = 1: c = 1 exactly (Sec. 3.5)


@pytest.mark.parametrize("name", ["multi", "longdoc"])
def test_quota_selection_on_scored_workloads(C, name):
    """The GPU's own scoring pass feeds the quota rule; against the oracle's
    scores: quotas within the band of the fp64 rule (one unit, only near a
    tie, at the score tolerance), exact sums, and per image the selection bar
    of tests/parity.py at the GPU's quota."""
    from paper_2609_05821_gb300 import pipeline
    inputs = synth.make_inputs(synth.workload(name), device="cuda")
    pipe = pipeline.from_inputs(inputs, selection="quota")
    pipe.score_select()
    torch.cuda.synchronize()
    ref = PT.oracle_requests(inputs)[0]
    spans = inputs["img_off"].tolist()
    n = np.diff(spans)
    quota = pipe.quota.cpu().numpy()
    # the GPU's g is within the score tolerance of the oracle's, so its c (and
    # with it each ideal share) within about twice that
    c64 = O.image_coefficients(ref["g"], pipe.lam)
    PT.assert_quotas_in_band(quota, c64, n, ref["k"], 2 * PT.RTOL[torch.bfloat16])
    idx = pipe.idx.cpu().numpy()[:ref["k"]]
    for j in range(len(n)):
        lo, hi = spans[j], spans[j + 1]
        mine = idx[(idx >= lo) & (idx < hi)] - lo
        s_img = ref["s"][lo:hi]
        order = np.argsort(-s_img, kind="stable")
        PT.assert_selection_ok(mine, None, s_img, np.sort(order[:quota[j]]), int(quota[j]),
                               PT.RTOL[torch.bfloat16])
