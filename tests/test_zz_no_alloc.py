"""conduit_select_topk_noalloc: selection for callers that cannot allocate.

Some callers cannot hand the library device scratch memory: a serving
engine that has given all free device memory to its paged KV pool and keeps
no allocator on this path, or plain C code with no device allocator. For
them the selection keeps its scratch (the sortable keys of requests too large
for registers) in a static device array of the library. These tests call
that entry point through the C ABI and check it against conduit_select_topk,
which takes a caller workspace:
  * batches whose largest request exceeds 8 192 tokens, so the selection
    kernel keeps its keys in the static array (smaller requests keep them in
    registers), on two calls in a row, the second with fewer tokens than the
    first (it runs over what the first call left in the array);
  * small batches (keys in registers), also twice;
  * a batch of exactly the array's size is accepted, one token more rejected.
The file is collected last and works alone or after the rest of the suite.
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


def _scores(C, seed, workload, full_request=1, **kw):
    w = synth.workload(workload, **kw)
    inputs = synth.make_inputs(w, device="cuda", seed=seed)
    kv = C.KvCache(inputs["k"], inputs["v"], w.num_q_heads)
    b = C.Batch(inputs["tok_off"], inputs["img_off"], inputs["req_img_off"], inputs["q_off"], "cuda")
    s, attn, g = C.conduit_score(kv, b, inputs["q"])
    tok = inputs["tok_off"].tolist()
    budgets = [C.conduit_budget(r, tok[i + 1] - tok[i]) for i, r in enumerate(inputs["ratios"])]
    if full_request is not None and full_request < len(budgets):
        budgets[full_request] = tok[full_request + 1] - tok[full_request]  # selects all its tokens
    return b, s, g, budgets


def _outputs(b, n_sel):
    n = b.n_tot
    return (torch.full((max(n_sel, 1),), -1, dtype=torch.int32, device="cuda"),
            torch.full((n,), 7, dtype=torch.uint8, device="cuda"),
            torch.full((n,), -1.0, device="cuda"),
            torch.full((b.num_images,), -1.0, device="cuda"))


def _same_as_workspace_selection(C, b, s, g, budgets, lam):
    off, off_d = C.idx_offsets(budgets, "cuda")
    n_sel = int(off[-1])
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


def test_noalloc_large_requests_use_the_static_array_twice(C):
    # 3 x 4096 = 12 288 tokens per request, then 2 x 4500 = 9 000: both above
    # the 8 192 keys a selection CTA keeps in registers
    b, s, g, budgets = _scores(C, 6, "multi", None, num_layers=1, images_per_request=3,
                               tokens_per_image=4096, num_requests=2)
    _same_as_workspace_selection(C, b, s, g, budgets, 1.0)
    b, s, g, budgets = _scores(C, 7, "multi", 0, num_layers=1, images_per_request=2,
                               tokens_per_image=4500, num_requests=1)
    budgets[0] = 901
    _same_as_workspace_selection(C, b, s, g, budgets, 0.5)


def test_noalloc_small_requests_twice(C):
    for call, seed in enumerate((4, 5)):
        b, s, g, budgets = _scores(C, seed, "batched", 1, num_requests=3, num_layers=2,
                                   tokens_per_image=96)
        _same_as_workspace_selection(C, b, s, g, budgets, 1.0 if call == 0 else 0.5)


def test_noalloc_limit_is_inclusive(C):
    n = C.NOALLOC_MAX_TOKENS
    b = C.Batch([0, n], [0, n], [0, 1], [0, 1], "cuda")
    s = torch.rand(n, device="cuda")
    g = torch.ones(1, device="cuda")
    off, off_d = C.idx_offsets([0], "cuda")
    idx, mask, s_hat, coeff = _outputs(b, 0)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    C.conduit_select_topk_noalloc(b, s, g, 1.0, off, off_d, idx, mask, s_hat, coeff, status)
    torch.cuda.synchronize()
    assert int(mask.sum()) == 0 and C.conduit_read_status(status) == C.OK


def test_noalloc_rejects_batches_beyond_its_scratch(C):
    n = C.NOALLOC_MAX_TOKENS + 1
    b = C.Batch([0, n], [0, n], [0, 1], [0, 1], "cuda")
    s = torch.zeros(1, device="cuda")
    off, off_d = C.idx_offsets([1], "cuda")
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(C.ConduitError) as ei:
        C.conduit_select_topk_noalloc(b, s, s, 1.0, off, off_d, idx)
    assert ei.value.code == C.ERR_UNSUPPORTED and "static scratch" in str(ei.value)
