"""conduit_score_select_topk: scoring and the global selection in one call.

The call promises the results of conduit_score_ex followed by
conduit_select_topk (Eqs. 6-11), bit for bit, in fewer launches: batches
whose requests hold at most 8192 tokens and whose 32-token blocks fit one
wave of SMs take the fused tail (the per-token reductions, the image means
g_j, c_j, s_hat and the top-k in one launch, the last block to finish a
request selecting it), others the separate launches. Checked on the GPU
against the two separate calls, bitwise:
  * the bench workloads (single image: fused; multi-image and paged batched
    serving: separate);
  * ragged batches whose requests start inside a 32-token block, down to
    requests of one token, so that one block completes many requests;
  * a request above 8192 tokens beside small ones (separate launches);
  * bf16 tensor-core and fp32 CUDA-core scoring, every scoring variant (RMS,
    side cache, no value norm, full-context softmax);
  * budgets 0 and N_r, lambda 0 and 1, and repeated calls (the arrival
    counters start from zero every call).
The pipeline's step runs this call, so the oracle comparisons of
test_gpu_parity.py and test_gpu_fuzz.py cover it against the paper's
definitions; one ragged case is also checked against the oracle here.
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


def _ragged(C, sizes, nq, dtype=torch.bfloat16, d=128, L=3, Hq=8, Hkv=2, seed=0):
    tok, img, rio = [0], [0], [0]
    for req in sizes:
        for n in req:
            img.append(img[-1] + n)
        tok.append(img[-1])
        rio.append(len(img) - 1)
    q_off = [0]
    for n in nq:
        q_off.append(q_off[-1] + n)
    gen = torch.Generator(device="cuda").manual_seed(seed)
    q = (torch.randn((L, Hq, q_off[-1], d), generator=gen, device="cuda") * 1.5).to(dtype)
    k = torch.randn((L, Hkv, tok[-1], d), generator=gen, device="cuda").to(dtype)
    v = torch.randn((L, Hkv, tok[-1], d), generator=gen, device="cuda").to(dtype)
    inputs = {"q": q, "k": k, "v": v, "tok_off": torch.tensor(tok, dtype=torch.int32),
              "img_off": torch.tensor(img, dtype=torch.int32),
              "req_img_off": torch.tensor(rio, dtype=torch.int32),
              "q_off": torch.tensor(q_off, dtype=torch.int32)}
    return C.KvCache(k, v, Hq), C.Batch(tok, img, rio, q_off, device="cuda"), inputs


def _garbage(shape, dtype):
    return torch.full(shape, 7 if dtype == torch.uint8 else -3.0, dtype=dtype, device="cuda")


def _both(C, kv, batch, q, lam, budgets, layers=None, **variant):
    """The separate calls and the fused one on the same inputs; returns both result tuples."""
    off, off_d = C.idx_offsets(budgets, "cuda")
    n, K = batch.n_tot, batch.num_images
    st1 = torch.zeros(1, dtype=torch.int32, device="cuda")
    s1, a1, g1 = C.conduit_score_ex(kv, batch, q, layers, status=st1, **variant)
    m1, h1, c1 = _garbage((n,), torch.uint8), _garbage((n,), torch.float32), _garbage((K,), torch.float32)
    i1, *_ = C.conduit_select_topk(batch, s1, g1, lam, off, off_d, None, m1, h1, c1, status=st1)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    m2, h2, c2 = _garbage((n,), torch.uint8), _garbage((n,), torch.float32), _garbage((K,), torch.float32)
    s2, a2, g2 = (_garbage((n,), torch.float32), _garbage((n,), torch.float32), _garbage((K,), torch.float32))
    i2 = torch.full((max(int(off[-1]), 1),), -5, dtype=torch.int32, device="cuda")
    C.conduit_score_select_topk(kv, batch, q, lam, off, off_d, layers, s=s2, attn_sum=a2, g=g2, idx=i2,
                                mask=m2, s_hat=h2, coeff=c2, status=st2, **variant)
    torch.cuda.synchronize()
    i2 = i2[:int(off[-1])]
    return (s1, a1, g1, i1, m1, h1, c1, st1), (s2, a2, g2, i2, m2, h2, c2, st2)


def _assert_bitwise(one, two, what=""):
    names = ("s", "attn_sum", "g", "idx", "mask", "s_hat", "coeff", "status")
    for name, x, y in zip(names, one, two):
        assert x.shape == y.shape and torch.equal(x, y), f"{what}: {name} differs"
    assert int(one[-1].item()) == 0, f"{what}: status {int(one[-1].item()):#x}"


def _budgets(batch, ratio=0.1):
    tok = batch.tok_off.tolist()
    return [int(ratio * (b - a)) for a, b in zip(tok[:-1], tok[1:])]


@pytest.mark.parametrize("name", ["single", "multi", "batched"])
def test_bench_workloads_bitwise(C, name):
    from paper_2609_05821_gb300 import pipeline
    inputs = synth.make_inputs(synth.workload(name), device="cuda")
    pipe = pipeline.from_inputs(inputs)
    one, two = _both(C, pipe.kv, pipe.batch, pipe.q, pipe.lam, pipe.budgets)
    _assert_bitwise(one, two, name)
    # the pipeline's step runs the fused call: same selection again
    pipe.score_select()
    torch.cuda.synchronize()
    assert torch.equal(pipe.idx[:pipe.n_sel], two[3]) and torch.equal(pipe.s, two[0])


def test_requests_inside_one_block_bitwise(C):
    # 40 one-token requests, then 1-37 token requests and a few images each:
    # the first 32-token block completes 32 requests, later blocks straddle
    # request boundaries
    sizes = [[1]] * 40 + [[5, 3], [37], [2, 1, 30], [33], [64], [31, 1], [1000, 24], [2049, 1, 7]]
    nq = [1 + (i % 5) for i in range(40)] + [16, 1, 9, 7, 3, 2, 40, 64]
    kv, batch, inputs = _ragged(C, sizes, nq)
    tok = batch.tok_off.tolist()
    n_r = [b - a for a, b in zip(tok[:-1], tok[1:])]
    for lam, budgets in ((1.0, [max(0, n // 3) for n in n_r]), (0.0, n_r), (0.7, [0] * len(n_r)),
                         (1.0, [min(n, 1) for n in n_r])):
        one, two = _both(C, kv, batch, inputs["q"], lam, budgets)
        _assert_bitwise(one, two, f"lambda {lam}")


def test_fused_path_is_one_launch_and_large_requests_take_the_separate_ones(C):
    kv, batch, inputs = _ragged(C, [[700, 300], [33]], [20, 5], L=2)
    n0 = C.conduit_launch_count()
    one, two = _both(C, kv, batch, inputs["q"], 1.0, _budgets(batch))
    _assert_bitwise(one, two, "small")
    separate = 4        # scoring kernel, finalize, image means, select
    assert C.conduit_launch_count() - n0 == separate + 2
    kv, batch, inputs = _ragged(C, [[9000], [100, 50], [8193]], [8, 3, 2], L=2)
    n0 = C.conduit_launch_count()
    one, two = _both(C, kv, batch, inputs["q"], 1.0, _budgets(batch, 0.2))
    _assert_bitwise(one, two, "large")
    assert C.conduit_launch_count() - n0 == 2 * separate


def test_fp32_cuda_core_scoring_bitwise(C):
    kv, batch, inputs = _ragged(C, [[256], [77, 13], [1], [300, 200]], [16, 3, 1, 9], dtype=torch.float32,
                                d=64, L=2, Hq=4, Hkv=2)
    one, two = _both(C, kv, batch, inputs["q"], 1.0, _budgets(batch, 0.25))
    _assert_bitwise(one, two, "fp32")


@pytest.mark.parametrize("variant", ["rms", "none", "side_cache", "extra_lse"])
def test_scoring_variants_bitwise(C, variant):
    kv, batch, inputs = _ragged(C, [[150, 150, 90], [1], [33, 64], [500]], [12, 2, 7, 30], L=3)
    kw = {}
    if variant == "rms":
        kw["statistic"] = "rms"
    elif variant == "none":
        kw["value_norm"] = "none"
    elif variant == "side_cache":
        kw["value_norm"] = "side_cache"
        kw["vnorm"] = C.conduit_value_norms(kv, batch)
    else:
        gen = torch.Generator(device="cuda").manual_seed(5)
        e = torch.randn((kv.num_layers, kv.num_q_heads, int(batch.q_off[-1])), generator=gen, device="cuda") * 2
        e[:, :, ::3] = -float("inf")
        kw["extra_lse"] = e
    one, two = _both(C, kv, batch, inputs["q"], 0.8, _budgets(batch, 0.15), [0, 2], **kw)
    _assert_bitwise(one, two, variant)


def test_repeated_calls_are_bitwise_equal(C):
    kv, batch, inputs = _ragged(C, [[1]] * 7 + [[400, 80], [9]], [2] * 7 + [24, 3])
    off, off_d = C.idx_offsets(_budgets(batch, 0.3), "cuda")
    outs = []
    ws = torch.empty(C.conduit_score_select_topk_workspace_size(kv, batch), dtype=torch.uint8, device="cuda")
    for _ in range(3):
        res = C.conduit_score_select_topk(kv, batch, inputs["q"], 1.0, off, off_d,
                                          mask=torch.empty(batch.n_tot, dtype=torch.uint8, device="cuda"),
                                          workspace=ws)
        torch.cuda.synchronize()
        outs.append([x.clone() for x in res if x is not None])
    for other in outs[1:]:
        assert all(torch.equal(x, y) for x, y in zip(outs[0], other))


def test_ragged_case_against_the_oracle(C):
    kv, batch, inputs = _ragged(C, [[37, 5], [1], [300], [64, 64, 1]], [9, 1, 17, 4], L=2)
    tok, rio = batch.tok_off.tolist(), batch.req_img_off.tolist()
    budgets = _budgets(batch, 0.2)
    off, off_d = C.idx_offsets(budgets, "cuda")
    s, A, g, idx, _, s_hat, coeff = C.conduit_score_select_topk(
        kv, batch, inputs["q"], 1.0, off, off_d, s_hat=torch.empty(batch.n_tot, device="cuda"),
        coeff=torch.empty(batch.num_images, device="cuda"))
    torch.cuda.synchronize()
    s, g, idx, s_hat, coeff = (x.cpu().numpy() for x in (s, g, idx, s_hat, coeff))
    off = off.tolist()
    for r in range(len(tok) - 1):
        view = synth.request_view(inputs, r)
        want = O.score_request(view["q"], view["k"], view["v"], view["img_off"])
        t0, t1, j0, j1 = tok[r], tok[r + 1], rio[r], rio[r + 1]
        PT.assert_scores_close(s[t0:t1], want["s"], 1e-3, f"s (request {r})")
        PT.assert_scores_close(g[j0:j1], want["g"], 1e-3, f"g (request {r})")
        # the selection is exact on the kernel's own keys (integer work)
        assert idx[off[r]:off[r + 1]].tolist() == O.topk_select(s_hat[t0:t1].astype(np.float64),
                                                                budgets[r]).tolist()


def test_non_finite_scores_flag_both_paths_alike(C):
    """A NaN query makes its request's scores NaN: the fused call flags
    CONDUIT_FLAG_NONFINITE as the separate calls do and returns the same bits."""
    kv, batch, inputs = _ragged(C, [[200, 56], [1], [90]], [6, 2, 5], L=2)
    q = inputs["q"].clone()
    q[1, 3, 0, 5] = float("nan")                      # layer 1, head 3, request 0's first query
    one, two = _both(C, kv, batch, q, 1.0, _budgets(batch, 0.2))
    names = ("s", "attn_sum", "g", "idx", "mask", "s_hat", "coeff", "status")
    for name, x, y in zip(names, one, two):
        bits = lambda t: t.view(torch.int32) if t.dtype == torch.float32 else t
        assert x.shape == y.shape and torch.equal(bits(x), bits(y)), name
    assert int(one[-1].item()) & C.FLAG_NONFINITE and int(one[-1].item()) == int(two[-1].item())
    tok = batch.tok_off.tolist()
    assert torch.isnan(one[0][tok[0]:tok[1]]).all() and torch.isfinite(one[0][tok[1]:]).all()
