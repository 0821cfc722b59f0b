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
