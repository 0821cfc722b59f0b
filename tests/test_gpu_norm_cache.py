"""GPU parity of the value-norm side cache (Sec. 4.3 and App. C.2: the value
norm depends only on the cached content, so it can be stored once per token
and layer and the scores stay exact).

  conduit_value_norms       against the oracle's norms of the same cache:
                            |gpu - ref| <= 1e-5 |ref|. Every square of a bf16
                            value is exact in fp32; each fp32 partial sum adds
                            at most 64 terms, so its relative error is below
                            64 * 2^-24 = 3.8e-6, and the square root halves it.
  conduit_score_with_norms  over that side cache: bitwise the s, A, g of
                            conduit_score (same partial sums, same order), and
                            over an arbitrary side cache: the oracle fed the
                            same stored norms, under the scoring tolerance.
  conduit_value_norms_update after each exchange: bitwise a full rebuild of
                            the side cache over the patched cache.

Cases cover both summation orders (tensor-core kernel: bf16 with head_dim
128, contiguous and paged; CUDA-core kernels: fp32, and bf16 with head_dim
64 over ragged requests including budgets 0 and N_r).
"""

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

from tests import parity as PT

pytestmark = pytest.mark.gpu

NORM_RTOL = 1e-5

CASES = {
    "single": (dict(name="single"), None),
    "batched_paged": (dict(name="batched", num_requests=3), None),
    "tiny_fp32": (dict(name="tiny"), [25]),
    "ragged_bf16_d64": (dict(name="multi", num_layers=3, num_q_heads=6, num_kv_heads=2, head_dim=64,
                             images_per_request=3, tokens_per_image=77, num_requests=3, n_q=None,
                             n_q_lo=1, n_q_hi=13), [0, 30, 231]),
}


@pytest.fixture(scope="module")
def C():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import conduit
    return conduit


@pytest.fixture(scope="module")
def P(C):
    from paper_2609_05821_gb300 import pipeline
    return pipeline


def _inputs(spec):
    spec = dict(spec)
    return synth.make_inputs(synth.workload(spec.pop("name"), **spec), device="cuda")


def _pipe(P, inputs, **kw):
    return P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()}, **kw)


def _oracle_norms(v):
    """Oracle value norms of a contiguous cache [L, Hkv, N_tot, d], one layer at a time."""
    return np.stack([O.value_norms(v[l].double().cpu().numpy()) for l in range(v.shape[0])])


@pytest.mark.parametrize("case", list(CASES))
def test_side_cache_is_exact(C, P, case):
    spec, budgets = CASES[case]
    inputs = _inputs(spec)
    plain = _pipe(P, inputs, budgets=budgets)
    normed = _pipe(P, inputs, budgets=budgets, value_norm="side_cache")
    torch.cuda.synchronize()
    # the side cache built at construction, against the oracle's norms
    PT.assert_scores_close(normed.vnorm.double().cpu().numpy().ravel(),
                           _oracle_norms(inputs["v"]).ravel(), NORM_RTOL, "vnorm")
    names = ("s", "attn_sum", "g", "coeff", "s_hat", "idx", "mask", "k_old", "v_old", "out")
    for step in range(2):  # the second step scores the cache the first one patched
        plain.step()
        normed.step()
        torch.cuda.synchronize()
        for name in names:
            assert torch.equal(getattr(plain, name), getattr(normed, name)), (step, name)
        rebuilt = C.conduit_value_norms(normed.kv, normed.batch)
        torch.cuda.synchronize()
        assert torch.equal(normed.vnorm, rebuilt), step
    assert C.conduit_read_status(normed.status) == C.OK


def test_score_with_norms_reads_the_given_norms(C, P):
    """An arbitrary stored-norm table (not V's norms), scored layers 1 and 3
    of 4, three ragged requests: against the oracle fed the same table."""
    w = synth.workload("multi", num_layers=4, images_per_request=3, tokens_per_image=150,
                       num_requests=3, n_q=None, n_q_lo=3, n_q_hi=40)
    inputs = synth.make_inputs(w, device="cuda")
    pipe = _pipe(P, inputs)
    gen = torch.Generator(device="cpu").manual_seed(1234)
    table = (torch.rand((4, pipe.batch.n_tot), generator=gen, dtype=torch.float64) * 8 + 0.25)
    vn = table.float().cuda()
    layers = [1, 3]
    s, A, g = C.conduit_score_with_norms(pipe.kv, pipe.batch, pipe.q, vn, layers=layers)
    torch.cuda.synchronize()
    ref = PT.oracle_requests(inputs, layers=layers)
    tok, rio = inputs["tok_off"].tolist(), inputs["req_img_off"].tolist()
    stored = vn.double().cpu().numpy()  # the fp32 values the GPU read
    for r, o in ref.items():
        t0, t1 = tok[r], tok[r + 1]
        view = o["view"]
        want = O.score_request(view["q"], view["k"], None, view["img_off"], layers,
                               vnorm=stored[:, t0:t1])
        PT.assert_scores_close(s[t0:t1].double().cpu().numpy(), want["s"], PT.RTOL[torch.bfloat16],
                               f"s (request {r})")
        PT.assert_scores_close(A[t0:t1].double().cpu().numpy(), want["A"], PT.RTOL[torch.bfloat16],
                               f"A (request {r})")
        PT.assert_scores_close(g[rio[r]:rio[r + 1]].double().cpu().numpy(), want["g"],
                               PT.RTOL[torch.bfloat16], f"g (request {r})")


def test_update_touches_only_the_selected_rows(C, P):
    """conduit_value_norms_update after a scatter: the selected rows get the
    patched cache's norms, every other entry keeps its stored value."""
    inputs = _inputs(CASES["ragged_bf16_d64"][0])
    pipe = _pipe(P, inputs, budgets=[5, 0, 40], value_norm="side_cache")
    pipe.score_select()
    sentinel = torch.full_like(pipe.vnorm, -1.0)
    C.conduit_kv_scatter(pipe.kv, pipe.batch, pipe.idx, pipe.idx_off, pipe.idx_off_dev,
                         pipe.k_rows, pipe.v_rows)
    C.conduit_value_norms_update(pipe.kv, pipe.batch, pipe.idx, pipe.idx_off, pipe.idx_off_dev,
                                 sentinel)
    full = C.conduit_value_norms(pipe.kv, pipe.batch)
    torch.cuda.synchronize()
    tok, off = inputs["tok_off"].tolist(), pipe.idx_off.tolist()
    idx = pipe.idx.cpu().tolist()
    rows = [tok[r] + t for r in range(3) for t in idx[off[r]:off[r + 1]]]
    assert len(rows) == 45
    touched = torch.zeros(pipe.batch.n_tot, dtype=torch.bool)
    touched[rows] = True
    got = sentinel.cpu()
    assert torch.equal(got[:, touched], full.cpu()[:, touched])
    assert torch.all(got[:, ~touched] == -1.0)
    # the patched rows' norms are those of the fresh value rows (oracle)
    fresh = pipe.v_rows.double().cpu().numpy()                 # [L, n_sel, Hkv, d]
    want = np.stack([O.value_norms(np.transpose(fresh[l], (1, 0, 2))) for l in range(fresh.shape[0])])
    PT.assert_scores_close(got[:, rows].double().numpy().ravel(), want.ravel(), NORM_RTOL, "updated")
