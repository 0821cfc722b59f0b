"""GPU parity of the isotropic Monte Carlo staleness estimator (App. D).

The refresh sets are the oracle's own Conduit selection and seeded uniform
random sets (no input of the oracle comes from the CUDA path); the standard
normal draws z are seeded and rounded to the cache dtype before both sides
see them. Bar: per request and per layer, |gpu - ref| <= rtol |ref| with
rtol = 1e-2 for bf16 caches (xi, P and the attention output are bf16 there,
three roundings of 2^-9 relative on each term of a sum of squares) and 1e-4
for fp32 caches (fp32 accumulation of up to a few thousand terms).
Covers both refresh kernels (tensor-core bf16 head_dim 128, contiguous and
paged; CUDA-core fp32 and bf16 head_dim 64) and, on the full multi-image
workload, two sampled layers.
"""

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

from tests import parity as PT

pytestmark = pytest.mark.gpu

CASES = {
    "multi_small": dict(name="multi", num_layers=2, images_per_request=3, tokens_per_image=150,
                        num_requests=3, n_q=None, n_q_lo=3, n_q_hi=40),
    "batched_paged": dict(name="batched", num_requests=3, num_layers=2, tokens_per_image=300),
    "tiny_fp32": dict(name="tiny"),
    "ragged_bf16_d64": dict(name="multi", num_layers=2, num_q_heads=6, num_kv_heads=2, head_dim=64,
                            images_per_request=3, tokens_per_image=77, num_requests=3, n_q=None,
                            n_q_lo=1, n_q_hi=13),
}
M = 3
KAPPA = 0.5


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


def _draws(inputs, M, seed):
    L, Hkv, n_tot, d = inputs["k"].shape
    gen = torch.Generator().manual_seed(seed)
    return torch.randn((M, L, Hkv, n_tot, d), generator=gen).to(inputs["k"].dtype)


def _sets(inputs, seed):
    """Per request: the oracle's Conduit selection and a uniform random set of the same size."""
    tok = inputs["tok_off"].tolist()
    ref = PT.oracle_requests(inputs)
    rng = np.random.default_rng(seed)
    conduit_mask = np.zeros(tok[-1], dtype=np.uint8)
    uniform_mask = np.zeros(tok[-1], dtype=np.uint8)
    for r, o in ref.items():
        conduit_mask[tok[r] + o["idx"]] = 1
        n_r = tok[r + 1] - tok[r]
        uniform_mask[tok[r] + rng.choice(n_r, o["k"], replace=False)] = 1
    return {"conduit": conduit_mask, "uniform": uniform_mask}


def _oracle(inputs, mask, z, layers=None):
    tok = inputs["tok_off"].tolist()
    L = inputs["k"].shape[0]
    out = {}
    for r in range(len(tok) - 1):
        view = synth.request_view(inputs, r)
        t0, t1 = tok[r], tok[r + 1]
        zr = z[:, :, :, t0:t1].double().numpy()
        ls = range(L) if layers is None else layers
        out[r] = [O.staleness_iso(view["q"][l:l + 1], view["k"][l:l + 1], view["v"][l:l + 1],
                                  mask[t0:t1], zr[:, l:l + 1], KAPPA) for l in ls]
    return out


@pytest.mark.parametrize("case", list(CASES))
def test_staleness_matches_oracle(C, P, case):
    spec = dict(CASES[case])
    inputs = synth.make_inputs(synth.workload(spec.pop("name"), **spec), device="cuda")
    pipe = P.from_inputs(inputs)
    z = _draws(inputs, M, 5)
    rtol = 1e-2 if inputs["k"].dtype == torch.bfloat16 else 1e-4
    L = inputs["k"].shape[0]
    R = len(inputs["tok_off"]) - 1
    for rule, mask in _sets(inputs, 6).items():
        layers = torch.empty((R, L), dtype=torch.float64, device="cuda")
        err, _ = C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, torch.as_tensor(mask).cuda(),
                                         z.cuda(), KAPPA, err_layers=layers)
        torch.cuda.synchronize()
        want = _oracle(inputs, mask, z)
        got_l = layers.cpu().numpy()
        for r in range(R):
            np.testing.assert_allclose(got_l[r], want[r], rtol=rtol, err_msg=f"{rule} request {r}")
            np.testing.assert_allclose(err[r].item(), sum(want[r]), rtol=rtol)
    # refreshing every token leaves no error; kappa scales the error by kappa^2
    all_in = torch.ones(pipe.batch.n_tot, dtype=torch.uint8, device="cuda")
    zero, _ = C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, all_in, z.cuda(), KAPPA)
    mask = torch.as_tensor(_sets(inputs, 6)["uniform"]).cuda()
    e1, _ = C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, mask, z.cuda(), 1.0)
    e2, _ = C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, mask, z.cuda(), 2.0)
    torch.cuda.synchronize()
    assert torch.all(zero == 0)
    np.testing.assert_allclose(e2.cpu().numpy(), 4 * e1.cpu().numpy(), rtol=2 * rtol)


def test_staleness_full_multi_sampled_layers(C, P):
    inputs = synth.make_inputs(synth.workload("multi"), device="cuda")
    pipe = P.from_inputs(inputs)
    z = _draws(inputs, 2, 7)
    mask = _sets(inputs, 8)["conduit"]
    L = inputs["k"].shape[0]
    layers = torch.empty((1, L), dtype=torch.float64, device="cuda")
    C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, torch.as_tensor(mask).cuda(), z.cuda(), KAPPA,
                            err_layers=layers)
    torch.cuda.synchronize()
    sample = [3, 21]
    want = _oracle(inputs, mask, z, layers=sample)[0]
    np.testing.assert_allclose(layers[0, sample].cpu().numpy(), want, rtol=1e-2)
