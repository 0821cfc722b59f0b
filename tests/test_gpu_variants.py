"""GPU parity of the scoring variants of conduit_score_ex against the oracle.

  statistic RMS (Eq. 4)      s against the oracle's RMS statistic; attn_sum and
                             g are the mean of Eq. 6 and stay bitwise those of
                             conduit_score (the same partial sums are formed)
  value norm NONE            s = attn_sum / |L| (fp32 division), i.e. the
                             factor ablation that ranks by attention alone
  full-context softmax       extra_lse rows (some -inf) against the oracle fed
                             the same values; all -inf gives bitwise the
                             visual-only pass
  combined                   RMS + side cache + extra_lse against the oracle
Tolerance: the scoring bar of tests/parity.py (1e-3 relative for bf16 inputs,
1e-5 for fp32, plus 1e-7 of the largest value).
"""

import pytest
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

from tests import parity as PT

pytestmark = pytest.mark.gpu

CASES = {
    "single": (dict(name="single"), None),
    "multi_ragged_subset": (dict(name="multi", num_layers=3, images_per_request=3, tokens_per_image=150,
                                 num_requests=3, n_q=None, n_q_lo=3, n_q_hi=40), [0, 2]),
    "tiny_fp32": (dict(name="tiny"), None),
    "ragged_bf16_d64": (dict(name="multi", num_layers=3, num_q_heads=6, num_kv_heads=2, head_dim=64,
                             images_per_request=3, tokens_per_image=77, num_requests=3, n_q=None,
                             n_q_lo=1, n_q_hi=13), None),
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


def _setup(P, case):
    spec, layers = CASES[case]
    spec = dict(spec)
    inputs = synth.make_inputs(synth.workload(spec.pop("name"), **spec), device="cuda")
    pipe = P.from_inputs(inputs)
    return inputs, pipe, layers


def _extra_lse(inputs, seed=7):
    """Outside-key log-sum-exps per scoring row (seeded, host copy)."""
    return synth.make_extra_lse(inputs, seed).cpu()


def _compare(pipe, inputs, got, layers, rtol, **oracle_kw):
    s, A, g = (x.double().cpu().numpy() for x in got)
    tok, rio, qo = inputs["tok_off"].tolist(), inputs["req_img_off"].tolist(), inputs["q_off"].tolist()
    extra = oracle_kw.pop("extra_lse", None)
    vnorm = oracle_kw.pop("vnorm", None)
    for r in range(len(tok) - 1):
        view = synth.request_view(inputs, r)
        t0, t1 = tok[r], tok[r + 1]
        kw = dict(oracle_kw)
        if extra is not None:
            kw["extra_lse"] = extra[:, :, qo[r]:qo[r + 1]].double().numpy()
        if vnorm is not None:
            kw["vnorm"] = vnorm[:, t0:t1].double().cpu().numpy()
        want = O.score_request(view["q"], view["k"], view["v"], view["img_off"], layers, **kw)
        PT.assert_scores_close(s[t0:t1], want["s"], rtol, f"s (request {r})")
        PT.assert_scores_close(A[t0:t1], want["A"], rtol, f"A (request {r})")
        PT.assert_scores_close(g[rio[r]:rio[r + 1]], want["g"], rtol, f"g (request {r})")


def _rtol(inputs):
    return PT.RTOL[inputs["k"].dtype]


@pytest.mark.parametrize("case", list(CASES))
def test_rms_statistic(C, P, case):
    inputs, pipe, layers = _setup(P, case)
    got = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, statistic="rms")
    base = C.conduit_score(pipe.kv, pipe.batch, pipe.q, layers)
    torch.cuda.synchronize()
    assert torch.equal(got[1], base[1]) and torch.equal(got[2], base[2])
    assert torch.all(got[0] > 0)
    _compare(pipe, inputs, got, layers, _rtol(inputs), statistic="rms")


@pytest.mark.parametrize("case", list(CASES))
def test_attention_alone(C, P, case):
    inputs, pipe, layers = _setup(P, case)
    s, A, g = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, value_norm="none")
    torch.cuda.synchronize()
    n_l = len(layers) if layers is not None else inputs["k"].shape[0]
    assert torch.equal(s, (A.double() / n_l).float())   # fp64 quotient rounds once more: exact
    _compare(pipe, inputs, (s, A, g), layers, _rtol(inputs), use_value_norm=False)


@pytest.mark.parametrize("case", list(CASES))
def test_full_context_softmax(C, P, case):
    inputs, pipe, layers = _setup(P, case)
    extra = _extra_lse(inputs)
    got = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, extra_lse=extra.cuda())
    torch.cuda.synchronize()
    A = got[1].double().cpu().numpy()
    n_l = len(layers) if layers is not None else inputs["k"].shape[0]
    assert A.sum() < n_l * (len(inputs["tok_off"]) - 1)   # every row now sums to less than 1
    _compare(pipe, inputs, got, layers, _rtol(inputs), extra_lse=extra)
    # no outside keys anywhere: bitwise the visual-only pass
    none = torch.full_like(extra, -float("inf")).cuda()
    a = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, extra_lse=none)
    b = C.conduit_score(pipe.kv, pipe.batch, pipe.q, layers)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(x, y)


@pytest.mark.parametrize("case", ["single", "ragged_bf16_d64"])
def test_rms_side_cache_full_context_together(C, P, case):
    inputs, pipe, layers = _setup(P, case)
    extra = _extra_lse(inputs, seed=8)
    vn = C.conduit_value_norms(pipe.kv, pipe.batch)
    got = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, statistic="rms",
                             value_norm="side_cache", vnorm=vn, extra_lse=extra.cuda())
    same_from_v = C.conduit_score_ex(pipe.kv, pipe.batch, pipe.q, layers, statistic="rms",
                                     extra_lse=extra.cuda())
    torch.cuda.synchronize()
    for x, y in zip(got, same_from_v):
        assert torch.equal(x, y)
    _compare(pipe, inputs, got, layers, _rtol(inputs), statistic="rms", extra_lse=extra)
