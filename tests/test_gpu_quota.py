"""GPU parity of the explicit per-image quota selection (App. D.3).

Integer work, so the bar is bitwise: on the same fp32 scores s and image
means g, conduit_select_quota must return
  coeff  bitwise the oracle's binary32 restatement of Eq. 9,
  quota  exactly the oracle's largest-remainder quotas for those coefficients,
  idx    exactly the oracle's per-image top-k_j of s (ties to the lowest index),
  mask / s_hat consistent with idx and s * c.
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
def test_quota_selection_bitwise(C, lam, g_mode):
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
        c32 = O.image_coefficients_f32(g32[j0:j1], lam)
        assert np.array_equal(coeff[j0:j1], c32), r
        spans = [x - t0 for x in img[j0:j1 + 1]]
        want = O.quota_select(s32[t0:t1].astype(np.float64), c32, spans, budgets[r])
        assert quota[j0:j1].tolist() == want["quota"].tolist(), (r, quota[j0:j1], want["quota"])
        assert idx[o[r]:o[r + 1]].tolist() == want["idx"].tolist(), r
        m = np.zeros(t1 - t0, dtype=np.uint8)
        m[want["idx"]] = 1
        assert np.array_equal(mask[t0:t1], m)
        n = np.diff(spans)
        assert np.array_equal(s_hat[t0:t1], s32[t0:t1] * np.repeat(c32, n))
    if g_mode == "dominant" and lam == 1.0:
        assert quota[rio[3]] == 5                          # capped at its 5 tokens


def test_global_coefficients_are_the_binary32_restatement(C):
    s, g, batch, budgets, tok, img, rio = _crafted(C, 12, "random")
    off, off_d = C.idx_offsets(budgets, "cuda")
    coeff = torch.empty(len(img) - 1, device="cuda")
    C.conduit_select_topk(batch, s.cuda(), g.cuda(), 0.7, off, off_d, coeff=coeff)
    torch.cuda.synchronize()
    got = coeff.cpu().numpy()
    for r in range(len(CRAFTED)):
        assert np.array_equal(got[rio[r]:rio[r + 1]], O.image_coefficients_f32(g.numpy()[rio[r]:rio[r + 1]], 0.7))


@pytest.mark.parametrize("name", ["multi", "longdoc"])
def test_quota_selection_on_scored_workloads(C, name):
    """The GPU's own scoring pass feeds the quota rule; against the oracle's
    scores: quotas within one unit of the oracle's, exact sums, and per image
    the selection bar of tests/parity.py at the GPU's quota."""
    from paper_2609_05821_gb300 import pipeline
    inputs = synth.make_inputs(synth.workload(name), device="cuda")
    pipe = pipeline.from_inputs(inputs, selection="quota")
    pipe.score_select()
    torch.cuda.synchronize()
    ref = PT.oracle_requests(inputs)[0]
    spans = inputs["img_off"].tolist()
    n = np.diff(spans)
    quota = pipe.quota.cpu().numpy()
    c32 = O.image_coefficients_f32(ref["g"].astype(np.float32), pipe.lam)
    want_q = O.image_quotas(c32, n, ref["k"])
    assert quota.sum() == ref["k"] and np.all(quota <= n) and np.all(quota >= 0)
    assert np.all(np.abs(quota - want_q) <= 1)
    idx = pipe.idx.cpu().numpy()[:ref["k"]]
    for j in range(len(n)):
        lo, hi = spans[j], spans[j + 1]
        mine = idx[(idx >= lo) & (idx < hi)] - lo
        s_img = ref["s"][lo:hi]
        order = np.argsort(-s_img, kind="stable")
        PT.assert_selection_ok(mine, None, s_img, np.sort(order[:quota[j]]), int(quota[j]),
                               PT.RTOL[torch.bfloat16])
