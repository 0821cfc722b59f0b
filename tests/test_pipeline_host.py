"""Host logic of the double-buffered end-to-end stepper (no kernels run).

DoubleBuffered alternates two pipelines so that one step's host-to-device
copies overlap the previous step's kernels; that is only sound when the two
pipelines share no buffer the copies write and have the same batch shape.
"""

import pytest
import torch

from paper_2609_05821_gb300 import synth


@pytest.fixture(scope="module")
def P():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import pipeline
    return pipeline


def _inputs(**kw):
    base = dict(num_layers=1, tokens_per_image=32, images_per_request=2, n_q=4, n_q_lo=4, n_q_hi=4)
    base.update(kw)
    return synth.make_inputs(synth.workload("multi", **base))


def _own(x):
    return {n: t.clone() if torch.is_tensor(t) else t for n, t in x.items()}


def test_separate_pipelines_alternate(P):
    x = _inputs()
    a, b = P.from_inputs(_own(x)), P.from_inputs(_own(x))
    d = P.DoubleBuffered(a, b)
    assert d.pipes == (a, b) and d._next == 0 and d._done == [None, None]


def test_pipelines_sharing_a_buffer_are_refused(P):
    x = _inputs()
    a = P.from_inputs(_own(x))
    shared_q = P.from_inputs({**_own(x), "q": a.q})  # the same query buffer
    with pytest.raises(ValueError, match="separate device buffers"):
        P.DoubleBuffered(a, shared_q)
    fresh = {"q_rows": a.q_rows, "k_rows": a.k_rows, "v_rows": a.v_rows}
    shared_rows = P.from_inputs(_own(x), fresh=fresh)  # the same fresh-row buffers
    with pytest.raises(ValueError, match="separate device buffers"):
        P.DoubleBuffered(a, shared_rows)


def test_pipelines_of_different_shapes_are_refused(P):
    a = P.from_inputs(_inputs())
    with pytest.raises(ValueError, match="same batch shape"):
        P.DoubleBuffered(a, P.from_inputs(_inputs(tokens_per_image=48)))
    with pytest.raises(ValueError, match="same batch shape"):
        P.DoubleBuffered(a, P.from_inputs(_inputs(), budgets=[5]))


def test_bench_work_model_matches_closed_forms(P):
    """The algorithmic bytes and FLOPs behind bench.py's roofline figures, on
    a hand-fixed selection: scoring reads K, V and Q once and writes s, A, g;
    the exchange reads and writes K and V rows twice (gather, scatter);
    refresh reads its query rows, writes its output and reads the K/V prefix
    up to the largest selected position, with causal FLOPs 4 Hq d (p + 1)."""
    import bench
    x = _inputs(num_layers=2)
    k = 5
    pipe = P.from_inputs(_own(x), budgets=[k])
    sel = [1, 7, 20, 33, 60]
    pipe.idx[:k] = torch.tensor(sel, dtype=torch.int32)
    m = bench.work_model(pipe)
    L, Hq, Hkv, d, b = 2, 28, 4, 128, 2
    N, nq, K = 64, 4, 2
    assert m["score"]["bytes"] == 2 * L * Hkv * N * d * b + L * Hq * nq * d * b + 8 * N + 4 * K
    assert m["score"]["flops"] == 2 * L * Hq * nq * N * d
    assert m["exchange"]["bytes"] == 8 * L * k * Hkv * d * b
    assert m["refresh"]["flops"] == L * sum(4 * Hq * d * (p + 1) for p in sel)
    assert m["refresh"]["bytes"] == 2 * L * k * Hq * d * b + 2 * L * Hkv * (max(sel) + 1) * d * b
    # scoring by attention alone drops the V read
    alone = P.from_inputs(_own(x), budgets=[k], value_norm="none")
    alone.idx[:k] = torch.tensor(sel, dtype=torch.int32)
    assert m["score"]["bytes"] - bench.work_model(alone)["score"]["bytes"] == L * Hkv * N * d * b
    # over several timed calls (the cache, and so the selection, changes from
    # step to step) the refresh work is the mean over their selections
    sel2 = [0, 2, 4, 6, 8]
    m2 = bench.work_model(pipe, [sel, sel2])
    f1 = L * sum(4 * Hq * d * (p + 1) for p in sel)
    f2 = L * sum(4 * Hq * d * (p + 1) for p in sel2)
    assert m2["refresh"]["flops"] == (f1 + f2) / 2
    assert m2["refresh"]["bytes"] == 2 * L * k * Hq * d * b + L * Hkv * (max(sel) + max(sel2) + 2) * d * b
    assert m2["score"] == m["score"] and m2["exchange"] == m["exchange"]
