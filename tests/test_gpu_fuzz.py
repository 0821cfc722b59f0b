"""Seeded shape fuzz of the whole step against the oracle.

Each case draws a geometry the named workloads never use: query heads per KV
group G in {1, 3, 5, 16} (query tiles of 128, 126, 125 and 128 rows),
requests of 1 to 255 tokens (one ragged key tile, or a single key), 1 to 300
scoring rows per request (one to several row groups), budgets 0, 1, N_r and
in between, bf16 head_dim 128 (tensor-core kernels) and bf16 head_dim 64 /
fp32 (CUDA-core kernels). The bar is that of tests/parity.py: scores within
1e-3 (bf16) / 1e-5 (fp32) relative, selections exact outside the tie band,
gather / scatter bitwise, refresh output within 2e-2 + 2^-8 relative (bf16)
or 1e-5 (fp32).
"""

import numpy as np
import pytest
import torch

from paper_2609_05821_gb300 import synth

from tests import parity as PT
from tests.test_gpu_parity import _check_refresh, _oracle, _patched_equals_scatter, _run

pytestmark = pytest.mark.gpu

# (Hq, Hkv, d, dtype, tokens per image, images, requests, n_q range, budget per request)
# budget "N" = every token, "rand" = a seeded draw from 2..N_r-1
CASES = [
    (16, 16, 128, "bf16", 1, 1, 2, (1, 3), (1, 0)),                  # G = 1, one-token requests
    (12, 4, 128, "bf16", 7, 3, 3, (1, 2), ("N", "rand", 1)),         # G = 3, 21 tokens, 1-2 queries
    (20, 4, 128, "bf16", 100, 2, 2, (40, 60), ("rand", "N")),        # G = 5: 125-row query tiles
    (32, 2, 128, "bf16", 129, 1, 2, (5, 20), ("rand", "N")),         # G = 16: 8 rows per tile
    (8, 8, 128, "bf16", 255, 1, 1, (200, 300), ("rand",)),           # G = 1, up to 2 400 score rows
    (6, 2, 64, "bf16", 50, 3, 3, (2, 9), (0, "rand", "N")),          # CUDA-core bf16
    (4, 1, 128, "f32", 90, 2, 2, (3, 6), ("N", "rand")),             # CUDA-core fp32, one KV head
]


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


@pytest.mark.parametrize("case", range(len(CASES)))
def test_fuzzed_shapes(C, P, case):
    hq, hkv, d, dtype, tpi, imgs, reqs, (lo, hi), modes = CASES[case]
    w = synth.workload("multi", num_layers=2, num_q_heads=hq, num_kv_heads=hkv, head_dim=d, dtype=dtype,
                       tokens_per_image=tpi, images_per_request=imgs, num_requests=reqs, n_q=None,
                       n_q_lo=lo, n_q_hi=hi, seed=100 + case)
    inputs = synth.make_inputs(w, device="cuda")
    tok = inputs["tok_off"].tolist()
    n_r = [tok[r + 1] - tok[r] for r in range(reqs)]
    rng = np.random.default_rng(200 + case)
    budgets = [n if m == "N" else int(rng.integers(2, n)) if m == "rand" else m for m, n in zip(modes, n_r)]
    pipe = _run(P, inputs, budgets=budgets)
    ref = _oracle(inputs, budgets=budgets)
    rtol = PT.RTOL[torch.float32 if dtype == "f32" else torch.bfloat16]
    PT.compare_score_select(pipe, inputs, ref, rtol)
    _check_refresh(P, pipe, inputs, ref, 1e-5 if dtype == "f32" else None)
    _patched_equals_scatter(C, pipe, inputs)
    assert C.conduit_read_status(pipe.status) == C.OK
