"""conduit_select_topk_noalloc: selection for callers that cannot allocate.

Some callers cannot hand the library device scratch memory (a serving engine
that has given all free memory to its KV pool, plain C code without a device
allocator). For them the selection keeps its scratch in a static device
array of the library. This test calls that entry point through the C ABI and
checks it against conduit_select_topk, which takes a caller workspace, on two
calls in a row (the second reuses the array the first call left behind).
It lives in its own file, collected last, and works alone or after the rest.
"""

import pytest
import torch

from paper_2609_05821_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import conduit
    return conduit


def _scores(C, seed):
    w = synth.workload("batched", num_requests=3, num_layers=2, tokens_per_image=96)
    inputs = synth.make_inputs(w, device="cuda", seed=seed)
    kv = C.KvCache(inputs["k"], inputs["v"], w.num_q_heads)
    b = C.Batch(inputs["tok_off"], inputs["img_off"], inputs["req_img_off"], inputs["q_off"], "cuda")
    s, attn, g = C.conduit_score(kv, b, inputs["q"])
    tok = inputs["tok_off"].tolist()
    budgets = [C.conduit_budget(r, tok[i + 1] - tok[i]) for i, r in enumerate(inputs["ratios"])]
    budgets[1] = tok[2] - tok[1]          # one request selects all of its tokens
    return b, s, g, budgets


def _outputs(b, n_sel):
    n = b.n_tot
    return (torch.full((max(n_sel, 1),), -1, dtype=torch.int32, device="cuda"),
            torch.full((n,), 7, dtype=torch.uint8, device="cuda"),
            torch.full((n,), -1.0, device="cuda"),
            torch.full((b.num_images,), -1.0, device="cuda"))


def test_noalloc_matches_workspace_selection_twice(C):
    for call, seed in enumerate((4, 5)):
        b, s, g, budgets = _scores(C, seed)
        off, off_d = C.idx_offsets(budgets, "cuda")
        n_sel = int(off[-1])
        lam = 1.0 if call == 0 else 0.5
        want = C.conduit_select_topk(b, s, g, lam, off, off_d, *_outputs(b, n_sel))
        idx, mask, s_hat, coeff = _outputs(b, n_sel)
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        C.conduit_select_topk_noalloc(b, s, g, lam, off, off_d, idx, mask, s_hat, coeff, status)
        torch.cuda.synchronize()
        assert torch.equal(idx[:n_sel], want[0][:n_sel])
        assert torch.equal(mask, want[1])
        assert torch.equal(s_hat, want[2])
        assert torch.equal(coeff, want[3])
        assert int(mask.sum()) == n_sel
        assert C.conduit_read_status(status) == C.OK


def test_noalloc_rejects_batches_beyond_its_scratch(C):
    n = C.NOALLOC_MAX_TOKENS + 16
    b = C.Batch([0, n], [0, n], [0, 1], [0, 1], "cuda")
    s = torch.zeros(1, device="cuda")
    off, off_d = C.idx_offsets([1], "cuda")
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(C.ConduitError) as ei:
        C.conduit_select_topk_noalloc(b, s, s, 1.0, off, off_d, idx)
    assert ei.value.code == C.ERR_UNSUPPORTED and "static scratch" in str(ei.value)
