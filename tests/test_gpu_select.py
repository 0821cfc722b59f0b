"""GPU parity of the global selection (Eqs. 9-11) on requests larger than one
CTA's registers (more than 8 192 tokens), which take a cluster of CTAs each.

Integer work on the kernel's own fp32 keys, so the bar is bitwise: with one
image per request (c = 1 exactly, Sec. 3.5) the keys are s itself and the
selection must be the oracle's top-k of s with ties to the lowest index; with
several images the kernel's s_hat must be s times its own c (binary32), c
within 1e-5 of Eq. 9 in fp64, and the selection the oracle's top-k of that
s_hat. Sizes cut the chunks of the cluster's CTAs unevenly; a fifth of the
scores share one value, so ties straddle chunk boundaries; budgets run from 1
to N_r.
"""

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O

from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import conduit
    return conduit


def _run(C, sizes_per_req, budgets, lam, seed):
    gen = torch.Generator().manual_seed(seed)
    tok, img, rio = [0], [0], [0]
    for req in sizes_per_req:
        for n in req:
            img.append(img[-1] + n)
        tok.append(img[-1])
        rio.append(len(img) - 1)
    n_tot = tok[-1]
    s = torch.rand(n_tot, generator=gen) * 1e-3
    s[torch.rand(n_tot, generator=gen) < 0.2] = 5e-4       # ties across the whole request
    s[torch.rand(n_tot, generator=gen) < 0.05] = 0.0       # exact zeros
    g = torch.rand(len(img) - 1, generator=gen) * 1e-3
    batch = C.Batch(tok, img, rio, list(range(len(sizes_per_req) + 1)), device="cuda")
    off, off_d = C.idx_offsets(budgets, "cuda")
    mask = torch.empty(n_tot, dtype=torch.uint8, device="cuda")
    s_hat = torch.empty(n_tot, device="cuda")
    coeff = torch.empty(len(img) - 1, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    idx, *_ = C.conduit_select_topk(batch, s.cuda(), g.cuda(), lam, off, off_d, None, mask, s_hat, coeff,
                                    status=status)
    torch.cuda.synchronize()
    assert C.conduit_read_status(status) == C.OK
    return (s.numpy(), g.numpy(), tok, img, rio, off.tolist(), idx.cpu().numpy(), mask.cpu().numpy(),
            s_hat.cpu().numpy(), coeff.cpu().numpy())


@pytest.mark.parametrize("seed", [1, 2])
def test_large_single_image_requests_exact(C, seed):
    sizes = [[9000], [41472], [8193], [65536], [8200]]
    budgets = [1, 4147, 8193, 30000, 0]
    s, g, tok, img, rio, off, idx, mask, s_hat, coeff = _run(C, sizes, budgets, 1.0, seed)
    for r, kk in enumerate(budgets):
        t0, t1 = tok[r], tok[r + 1]
        assert coeff[rio[r]] == 1.0                           # one image: c = 1 exactly
        want = O.topk_select(s[t0:t1].astype(np.float64), kk)
        assert idx[off[r]:off[r + 1]].tolist() == want.tolist(), r
        m = np.zeros(t1 - t0, dtype=np.uint8)
        m[want] = 1
        assert np.array_equal(mask[t0:t1], m), r
        assert np.array_equal(s_hat[t0:t1], s[t0:t1])


def test_large_multi_image_request_on_its_own_keys(C):
    sizes = [[1296] * 32, [5000, 7000]]
    budgets = [4147, 1200]
    s, g, tok, img, rio, off, idx, mask, s_hat, coeff = _run(C, sizes, budgets, 0.7, 3)
    for r, kk in enumerate(budgets):
        t0, t1, j0, j1 = tok[r], tok[r + 1], rio[r], rio[r + 1]
        PT.assert_scores_close(coeff[j0:j1], O.image_coefficients(g[j0:j1].astype(np.float64), 0.7), 1e-5,
                               f"c (request {r})")
        n = np.diff(img[j0:j1 + 1])
        assert np.array_equal(s_hat[t0:t1], s[t0:t1] * np.repeat(coeff[j0:j1], n))
        want = O.topk_select(s_hat[t0:t1].astype(np.float64), kk)
        assert idx[off[r]:off[r + 1]].tolist() == want.tolist(), r
