"""GPU parity: every C-ABI call against the CPU oracle on the same seeded inputs.

Sizes: the five workloads at their full sizes (long-document and batched
compare whole requests drawn from the batch, refresh rows sampled), plus
ragged small shapes that cut tiles and warps unevenly. Tolerances are in
tests/parity.py.
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


@pytest.fixture(scope="module")
def P(C):
    from paper_2609_05821_gb300 import pipeline
    return pipeline


class _Layers:
    """Lazily widened per-layer numpy views of one request (keeps host memory low)."""

    def __init__(self, t, lo, hi):
        self.t, self.lo, self.hi = t, lo, hi

    def __len__(self):
        return self.t.shape[0]

    def __getitem__(self, l):
        return self.t[l, :, self.lo:self.hi, :].double().cpu().numpy()


def _oracle(inputs, lam=1.0, layers=None, budgets=None, requests=None):
    tok, qo = inputs["tok_off"].tolist(), inputs["q_off"].tolist()
    img, rio = inputs["img_off"].tolist(), inputs["req_img_off"].tolist()
    out = {}
    for r in (range(len(tok) - 1) if requests is None else requests):
        t0, t1 = tok[r], tok[r + 1]
        spans = [x - t0 for x in img[rio[r]:rio[r + 1] + 1]]
        kk = budgets[r] if budgets is not None else O.budget(inputs["ratios"][r], t1 - t0)
        sc = O.score_request(_Layers(inputs["q"], qo[r], qo[r + 1]), _Layers(inputs["k"], t0, t1),
                             _Layers(inputs["v"], t0, t1), spans, layers)
        c = O.image_coefficients(sc["g"], lam)
        s_hat = O.composite_score(sc["s"], c, spans)
        out[r] = dict(sc, c=c, s_hat=s_hat, idx=O.topk_select(s_hat, kk), k=kk)
    return out


def _check_refresh(P, pipe, inputs, ref, rtol_out, layers_sample=None, rows_sample=None, seed=0):
    """gather / scatter / refresh against the oracle on the oracle's own selection.

    A GPU selection may differ from the oracle's inside the tie band, so the
    index-driven calls are run again on a fresh copy of the cache (same fresh
    rows, same paging) with every request of ``ref`` given the oracle's
    indices; every such request with k > 0 is then compared (sampled layers
    and rows at full size). Returns the (request, layer, row) triples
    compared and asserts that there was at least one whenever some k > 0.
    """
    tok = inputs["tok_off"].tolist()
    off = pipe.idx_off.tolist()
    fresh = {"q_rows": pipe.q_rows, "k_rows": pipe.k_rows, "v_rows": pipe.v_rows}
    twin = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()},
                         paged=pipe.kv.page_table is not None and pipe.kv.k.dim() == 5,
                         budgets=pipe.budgets, fresh=fresh)
    twin.idx.copy_(pipe.idx)
    for r, o in ref.items():
        assert len(o["idx"]) == off[r + 1] - off[r] == o["k"]
        if o["k"]:
            twin.idx[off[r]:off[r + 1]] = torch.as_tensor(o["idx"], dtype=torch.int32, device=twin.idx.device)
    twin.refresh()
    torch.cuda.synchronize()
    L = inputs["k"].shape[0]
    rng = np.random.default_rng(seed)
    k_old, v_old = twin.k_old.cpu(), twin.v_old.cpu()
    out = twin.out.double().cpu().numpy()
    compared = 0
    for r, o in ref.items():
        if o["k"] == 0:
            continue
        t0, t1 = tok[r], tok[r + 1]
        ls = range(L) if layers_sample is None else sorted(rng.choice(L, layers_sample, replace=False))
        rows = np.arange(o["k"])
        if rows_sample is not None and rows_sample < o["k"]:
            rows = np.sort(rng.choice(o["k"], rows_sample, replace=False))
        for l in ls:
            kc = inputs["k"][l:l + 1, :, t0:t1].double().cpu().numpy()
            vc = inputs["v"][l:l + 1, :, t0:t1].double().cpu().numpy()
            # gather: bitwise copies of the stale rows
            want_k = O.kv_gather(kc, o["idx"])[0]
            np.testing.assert_array_equal(k_old[l, off[r]:off[r + 1]].double().numpy(), want_k)
            want_v = O.kv_gather(vc, o["idx"])[0]
            np.testing.assert_array_equal(v_old[l, off[r]:off[r + 1]].double().numpy(), want_v)
            fk = twin.k_rows[l:l + 1, off[r]:off[r + 1]].double().cpu().numpy()
            fv = twin.v_rows[l:l + 1, off[r]:off[r + 1]].double().cpu().numpy()
            kp = O.kv_scatter(kc, o["idx"], fk)
            vp = O.kv_scatter(vc, o["idx"], fv)
            qr = twin.q_rows[l:l + 1, off[r]:off[r + 1]].double().cpu().numpy()
            want = O.refresh_attention(qr[:, rows], kp, vp, o["idx"][rows])[0]
            got = out[l, off[r] + rows]
            if rtol_out is None:
                # bf16 output: 2e-2 plus half a bf16 ulp of the value (2^-8 relative)
                np.testing.assert_allclose(got, want, rtol=2.0 ** -8, atol=2e-2)
            else:
                np.testing.assert_allclose(got, want, rtol=rtol_out, atol=1e-6)
            compared += len(rows)
    if any(o["k"] for o in ref.values()):
        assert compared > 0, "no refresh row was compared"
    if twin.kv.k.dim() == 4:  # contiguous cache: the whole patched cache, bitwise
        _patched_equals_scatter(None, twin, inputs)
    del twin
    return compared


def _patched_equals_scatter(C, pipe, inputs):
    """After the step the cache holds the fresh rows at the selected positions, the stale rows elsewhere."""
    tok = inputs["tok_off"].tolist()
    off = pipe.idx_off.tolist()
    idx = pipe.idx.cpu().numpy()
    k_now, v_now = pipe.kv.k.cpu(), pipe.kv.v.cpu()
    for r in range(len(tok) - 1):
        sel = idx[off[r]:off[r + 1]]
        t0, t1 = tok[r], tok[r + 1]
        want_k = inputs["k"][:, :, t0:t1].clone().cpu()
        want_v = inputs["v"][:, :, t0:t1].clone().cpu()
        want_k[:, :, sel] = pipe.k_rows[:, off[r]:off[r + 1]].cpu().transpose(1, 2)
        want_v[:, :, sel] = pipe.v_rows[:, off[r]:off[r + 1]].cpu().transpose(1, 2)
        assert torch.equal(k_now[:, :, t0:t1], want_k)
        assert torch.equal(v_now[:, :, t0:t1], want_v)


def _run(P, inputs, **kw):
    pipe = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()}, **kw)
    pipe.step()
    torch.cuda.synchronize()
    return pipe


# ------------------------------------------------------------------ workloads
@pytest.mark.parametrize("k_budget", [25, 26])
def test_tiny_fp32(C, P, k_budget):
    w = synth.workload("tiny")
    inputs = synth.make_inputs(w, device="cuda")
    pipe = _run(P, inputs, budgets=[k_budget])
    ref = _oracle(inputs, budgets=[k_budget])
    PT.compare_score_select(pipe, inputs, ref, PT.RTOL[torch.float32])
    assert pipe.coeff.item() == 1.0
    _check_refresh(P, pipe, inputs, ref, rtol_out=1e-5)
    _patched_equals_scatter(C, pipe, inputs)
    assert C.conduit_read_status(pipe.status) == C.OK


def test_single_image_full(C, P):
    inputs = synth.make_inputs(synth.workload("single"), device="cuda")
    pipe = _run(P, inputs)
    ref = _oracle(inputs)
    assert ref[0]["k"] == 102
    PT.compare_score_select(pipe, inputs, ref, PT.RTOL[torch.bfloat16])
    assert pipe.coeff.item() == 1.0                        # K = 1: c = 1 exactly (Sec. 3.5)
    _check_refresh(P, pipe, inputs, ref, None, layers_sample=6)
    _patched_equals_scatter(C, pipe, inputs)


def test_multi_image_full(C, P):
    inputs = synth.make_inputs(synth.workload("multi"), device="cuda")
    pipe = _run(P, inputs)
    ref = _oracle(inputs)
    assert ref[0]["k"] == 819
    PT.compare_score_select(pipe, inputs, ref, PT.RTOL[torch.bfloat16])
    _check_refresh(P, pipe, inputs, ref, None, layers_sample=3, rows_sample=48)


def test_long_document_full_three_budgets(C, P):
    inputs = synth.make_inputs(synth.workload("longdoc"), device="cuda")
    ref = _oracle(inputs, budgets=[2073])
    for r_ratio, kk in ((0.05, 2073), (0.10, 4147), (0.20, 8294)):
        pipe = _run(P, inputs, budgets=[kk])
        assert C.conduit_budget(r_ratio, 41472) == kk == O.budget(r_ratio, 41472)
        o = dict(ref[0])
        o.update(k=kk, idx=O.topk_select(o["s_hat"], kk))
        PT.compare_score_select(pipe, inputs, {0: o}, PT.RTOL[torch.bfloat16])
        if kk == 4147:
            _check_refresh(P, pipe, inputs, {0: o}, None, layers_sample=2, rows_sample=32)
        del pipe


def test_batched_paged_sampled_requests(C, P):
    w = synth.workload("batched")
    inputs = synth.make_inputs(w, device="cuda")
    pipe = _run(P, inputs)                                 # paged, as the workload says
    ref = _oracle(inputs, requests=[0, 11])
    PT.compare_score_select(pipe, inputs, ref, PT.RTOL[torch.bfloat16])
    _check_refresh(P, pipe, inputs, ref, None, layers_sample=2, rows_sample=24)
    flat = _run(P, inputs, paged=False)                    # contiguous twin: bitwise equal
    for name in ("s", "attn_sum", "g", "coeff", "s_hat", "idx", "mask", "k_old", "v_old", "out"):
        assert torch.equal(getattr(pipe, name), getattr(flat, name)), name


# ------------------------------------------------------------ ragged shapes
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_ragged_multi_request(C, P, dtype):
    w = synth.workload("multi", num_layers=3, num_q_heads=6, num_kv_heads=2, head_dim=64,
                       images_per_request=3, tokens_per_image=77, num_requests=3, n_q=None,
                       n_q_lo=1, n_q_hi=13, dtype=dtype)
    inputs = synth.make_inputs(w, device="cuda")
    budgets = [0, 30, 231]                                  # k = 0, ragged, k = N_r
    pipe = _run(P, inputs, budgets=budgets)
    ref = _oracle(inputs, budgets=budgets)
    rt = PT.RTOL[torch.float32 if dtype == "f32" else torch.bfloat16]
    PT.compare_score_select(pipe, inputs, ref, rt)
    _check_refresh(P, pipe, inputs, ref, 1e-5 if dtype == "f32" else None)
    _patched_equals_scatter(C, pipe, inputs)


def test_head_dim_128_ragged_tokens(C, P):
    w = synth.workload("single", num_layers=2, tokens_per_image=1000, n_q=5, n_q_lo=5, n_q_hi=5)
    inputs = synth.make_inputs(w, device="cuda")
    pipe = _run(P, inputs, budgets=[333])
    PT.compare_score_select(pipe, inputs, _oracle(inputs, budgets=[333]), PT.RTOL[torch.bfloat16])


# --------------------------------------------------------------- edge cases
def _small_multi(**kw):
    base = dict(num_layers=2, tokens_per_image=128, images_per_request=4)
    base.update(kw)
    return synth.make_inputs(synth.workload("multi", **base), device="cuda")


def test_budget_zero_and_full(C, P):
    inputs = _small_multi()
    n = inputs["tok_off"].tolist()[-1]
    for kk in (0, n):
        pipe = _run(P, inputs, budgets=[kk])
        assert int(pipe.mask.sum()) == kk
        if kk:
            assert pipe.idx[:kk].tolist() == list(range(n))


def test_lambda_zero_and_single_image_coefficients(C, P):
    inputs = _small_multi()
    pipe = _run(P, inputs, lam=0.0)
    assert torch.all(pipe.coeff == 1.0)
    ref = _oracle(inputs, lam=0.0)
    PT.compare_score_select(pipe, inputs, ref, 1e-3)
    pipe1 = _run(P, inputs, lam=1.0)
    c = pipe1.coeff.double()
    assert abs(c.mean().item() - 1.0) < 1e-6               # App. B.2: mean c_j = 1


def test_zero_value_norm_scores_exactly_zero(C, P):
    inputs = _small_multi()
    zero = [0, 5, 300, 511]
    inputs["v"][:, :, zero, :] = 0
    pipe = _run(P, inputs)
    assert torch.all(pipe.s[zero] == 0)
    assert torch.all(pipe.s[[1, 2, 3]] > 0)


def test_deterministic_bitwise(C, P):
    inputs = _small_multi()
    a, b = _run(P, inputs), _run(P, inputs)
    for name in ("s", "attn_sum", "g", "s_hat", "idx", "mask", "out"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name


def test_batched_equals_per_request(C, P):
    w = synth.workload("batched", num_requests=3, num_layers=2, tokens_per_image=64)
    inputs = synth.make_inputs(w, device="cuda")
    whole = _run(P, inputs, paged=False)
    tok, qo, rio = inputs["tok_off"].tolist(), inputs["q_off"].tolist(), inputs["req_img_off"].tolist()
    off = whole.idx_off.tolist()
    for r in range(3):
        one = {
            "workload": w, "q": inputs["q"][:, :, qo[r]:qo[r + 1]].contiguous(),
            "k": inputs["k"][:, :, tok[r]:tok[r + 1]].contiguous(),
            "v": inputs["v"][:, :, tok[r]:tok[r + 1]].contiguous(),
            "tok_off": torch.tensor([0, tok[r + 1] - tok[r]], dtype=torch.int32),
            "img_off": torch.tensor([x - tok[r] for x in inputs["img_off"].tolist()[rio[r]:rio[r + 1] + 1]],
                                    dtype=torch.int32),
            "req_img_off": torch.tensor([0, rio[r + 1] - rio[r]], dtype=torch.int32),
            "q_off": torch.tensor([0, qo[r + 1] - qo[r]], dtype=torch.int32),
            "ratios": [inputs["ratios"][r]],
        }
        single = _run(P, one, paged=False)
        assert torch.equal(single.s, whole.s[tok[r]:tok[r + 1]])
        assert torch.equal(single.g, whole.g[rio[r]:rio[r + 1]])
        assert torch.equal(single.idx[:off[r + 1] - off[r]], whole.idx[off[r]:off[r + 1]])


def test_scored_layer_subset(C, P):
    inputs = _small_multi(num_layers=4)
    pipe = _run(P, inputs, layers=[1, 3])
    PT.compare_score_select(pipe, inputs, _oracle(inputs, layers=[1, 3]), 1e-3)


def test_index_driven_refresh_with_oracle_indices(C, P):
    """gather / scatter / refresh fed the oracle's own selection."""
    inputs = _small_multi(tokens_per_image=100)
    ref = _oracle(inputs)
    kk = ref[0]["k"]
    pipe = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    pipe.idx[:kk] = torch.as_tensor(ref[0]["idx"], dtype=torch.int32, device="cuda")
    pipe.refresh()
    torch.cuda.synchronize()
    _check_refresh(P, pipe, inputs, ref, None)
    _patched_equals_scatter(C, pipe, inputs)


@pytest.mark.parametrize("paged", [False, True])
def test_exchange_equals_gather_then_scatter(C, P, paged):
    """conduit_kv_exchange (the pipeline's call) against conduit_kv_gather
    followed by conduit_kv_scatter on a copy of the cache: bitwise."""
    inputs = synth.make_inputs(synth.workload("batched" if paged else "multi",
                                              **({"num_requests": 3} if paged else {})), device="cuda")
    a = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    b = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    a.score_select()
    b.score_select()
    C.conduit_kv_exchange(a.kv, a.batch, a.idx, a.idx_off, a.idx_off_dev, a.k_old, a.v_old,
                          a.k_rows, a.v_rows)
    C.conduit_kv_gather(b.kv, b.batch, b.idx, b.idx_off, b.idx_off_dev, b.k_old, b.v_old)
    C.conduit_kv_scatter(b.kv, b.batch, b.idx, b.idx_off, b.idx_off_dev, b.k_rows, b.v_rows)
    torch.cuda.synchronize()
    assert torch.equal(a.idx, b.idx)
    for x, y in ((a.k_old, b.k_old), (a.v_old, b.v_old), (a.kv.k, b.kv.k), (a.kv.v, b.kv.v)):
        assert torch.equal(x, y)
    assert not torch.equal(a.k_old, a.k_rows)  # the stale rows differ from the fresh ones


def test_refresh_late_max_jump_in_some_heads(C, P):
    """Rows whose running max jumps far (> 2^8) at a late key tile while other
    rows of the same warp do not: the lazy O rescale must stay correct."""
    inputs = _small_multi(num_layers=1, tokens_per_image=128)   # N = 512, G = 7
    d = inputs["k"].shape[-1]
    u = torch.nn.functional.normalize(torch.randn(d, device="cuda"), dim=0)
    k = inputs["k"].clone()
    k[0, :, 400, :] = (45.0 * u).to(k.dtype)                    # planted key, not refreshed
    base = {**inputs, "k": k, "v": inputs["v"].clone()}
    sel = list(range(401, 481))
    pipe = P.from_inputs(base, budgets=[len(sel)])
    q_rows = pipe.q_rows.clone()
    q_rows[:, :, 0::2, :] = (8.0 * u).to(q_rows.dtype)          # even heads aim at the planted key
    pipe.q_rows.copy_(q_rows)
    pipe.idx[:len(sel)] = torch.tensor(sel, dtype=torch.int32, device="cuda")
    pipe.refresh()
    torch.cuda.synchronize()
    assert C.conduit_read_status(pipe.status) == C.OK
    kp = O.kv_scatter(k[:, :, :512].double().cpu().numpy(), sel, pipe.k_rows.double().cpu().numpy())
    vp = O.kv_scatter(inputs["v"][:, :, :512].double().cpu().numpy(), sel, pipe.v_rows.double().cpu().numpy())
    want = O.refresh_attention(pipe.q_rows.double().cpu().numpy(), kp, vp, sel)
    np.testing.assert_allclose(pipe.out.double().cpu().numpy(), want, rtol=2.0 ** -8, atol=2e-2)


def test_nonfinite_input_sets_status_word(C, P):
    inputs = _small_multi()
    inputs["v"][0, 0, 7, 3] = float("nan")
    pipe = _run(P, inputs)
    assert C.conduit_read_status(pipe.status) == C.ERR_NONFINITE
    C.conduit_clear_status(pipe.status)
    assert C.conduit_read_status(pipe.status) == C.OK


def test_step_from_host_equals_step(C, P):
    """The end-to-end form (host copies on their own stream, the step as two
    graphs) gives bitwise the selection and output of the plain step."""
    inputs = _small_multi(num_layers=3)
    a = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    b = P.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    host = a.host_buffers()          # the cache before any step
    a.capture()                      # the capture runs one step on a's buffers
    a.step_from_host(host)           # the copies restore them first
    b.step()
    torch.cuda.synchronize()
    assert torch.equal(host["idx"].cuda(), b.idx)
    assert torch.equal(host["out"].cuda(), b.out)
    assert torch.equal(a.kv.k, b.kv.k) and torch.equal(a.kv.v, b.kv.v)


def test_double_buffered_steps_equal_plain_steps(C, P):
    """Two pipelines stepped alternately, back to back, from two different
    host batches: every step's selection, output and patched cache are
    bitwise those of a plain step on a fresh pipeline over that batch."""
    from paper_2609_05821_gb300 import synth
    w = synth.workload("multi", num_layers=3, tokens_per_image=128, images_per_request=4)
    batches = [synth.make_inputs(w, device="cuda", seed=s) for s in (21, 22)]
    fresh = [synth.make_fresh_rows(w, 51, device="cuda", seed=s) for s in (31, 32)]
    own = lambda x: {n: t.clone() if torch.is_tensor(t) else t for n, t in x.items()}
    # a pipeline keeps the tensors it is given (q, fresh rows), so each gets copies
    pipes = [P.from_inputs(own(x), fresh=own(f), budgets=[51]) for x, f in zip(batches, fresh)]
    hosts = [p.host_buffers() for p in pipes]  # each batch's cache before any step
    for p in pipes:
        p.capture()
    stepper = P.DoubleBuffered(*pipes)
    order = [0, 1, 0, 1, 1, 0]
    outs = []
    for j in order:
        ran = stepper.step_from_host(hosts[j])
        host_copy = {"idx": torch.empty_like(hosts[j]["idx"]), "out": torch.empty_like(hosts[j]["out"])}
        torch.cuda.current_stream().synchronize()
        host_copy["idx"].copy_(hosts[j]["idx"])
        host_copy["out"].copy_(hosts[j]["out"])
        outs.append((j, host_copy, ran.kv.k.clone(), ran.kv.v.clone()))
    for j, got, k_now, v_now in outs:
        ref = P.from_inputs(own(batches[j]), fresh=own(fresh[j]), budgets=[51])
        ref.step()
        torch.cuda.synchronize()
        assert torch.equal(got["idx"].cuda(), ref.idx)
        assert torch.equal(got["out"].cuda(), ref.out)
        assert torch.equal(k_now, ref.kv.k) and torch.equal(v_now, ref.kv.v)


def test_double_buffered_back_to_back_equals_plain(C, P):
    """Back to back with no synchronisation between steps (each step's copies
    overlapping the previous step's kernels), the last step's results are
    bitwise those of a plain step."""
    inputs = _small_multi(num_layers=3)
    own = lambda x: {n: t.clone() if torch.is_tensor(t) else t for n, t in x.items()}
    pipes = [P.from_inputs(own(inputs)) for _ in range(2)]
    host = pipes[0].host_buffers()
    for p in pipes:
        p.capture()
    stepper = P.DoubleBuffered(*pipes)
    last = None
    for _ in range(5):
        last = stepper.step_from_host(host)
    torch.cuda.synchronize()
    ref = P.from_inputs(own(inputs))
    ref.step()
    torch.cuda.synchronize()
    assert torch.equal(host["idx"].cuda(), ref.idx)
    assert torch.equal(host["out"].cuda(), ref.out)
    assert torch.equal(last.kv.k, ref.kv.k)


@pytest.mark.parametrize("page_size,tokens_per_image", [(8, 208), (32, 208), (64, 224), (128, 192)])
def test_paged_caches_of_every_page_size_equal_contiguous(C, P, page_size, tokens_per_image):
    """Scoring, selection, exchange and refresh over a paged cache (pages in a
    seeded shuffled pool order) give bitwise the results of the contiguous
    cache, for every page size the tensor-core kernels take (one TMA copy per
    page half: 32 copies per tile at page size 8). Requests of 416 and 448
    tokens end in a ragged key tile."""
    w = synth.workload("multi", num_layers=2, images_per_request=2, tokens_per_image=tokens_per_image,
                       num_requests=3, n_q=None, n_q_lo=5, n_q_hi=40, page_size=page_size)
    inputs = synth.make_inputs(w, device="cuda")
    paged = _run(P, inputs, paged=True)
    flat = _run(P, inputs, paged=False)
    assert paged.kv.k.dim() == 5 and paged.kv.k.shape[3] == page_size
    for name in ("s", "attn_sum", "g", "coeff", "s_hat", "idx", "mask", "k_old", "v_old", "out"):
        assert torch.equal(getattr(paged, name), getattr(flat, name)), name


def test_tensor_core_refresh_mixed_budgets(C, P):
    """One launch of the tensor-core path over requests with budgets 0, N_r,
    1 and 17: items of a single row, whole requests and empty requests share
    the persistent grid and its work counter."""
    w = synth.workload("multi", num_layers=2, images_per_request=2, tokens_per_image=128, num_requests=4,
                       n_q=None, n_q_lo=3, n_q_hi=30)
    inputs = synth.make_inputs(w, device="cuda")
    budgets = [0, 256, 1, 17]
    pipe = _run(P, inputs, budgets=budgets)
    ref = _oracle(inputs, budgets=budgets)
    PT.compare_score_select(pipe, inputs, ref, PT.RTOL[torch.bfloat16])
    _check_refresh(P, pipe, inputs, ref, None)
    _patched_equals_scatter(C, pipe, inputs)
    assert C.conduit_read_status(pipe.status) == C.OK
