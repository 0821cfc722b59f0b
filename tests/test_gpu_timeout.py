"""The bounded-wait path of the tensor-core kernels, made to run out on purpose.

Every wait of the kernels on an mbarrier is bounded; a role whose wait runs
out raises an abort flag, the kernel sets CONDUIT_FLAG_TIMEOUT with a site bit
in the caller's status word, drains the copies it issued, frees its tensor
memory and returns, so the context stays usable. To reach that path without
any fault, the test uses a separate test-only build of the library
(libconduit_testhooks.so: waits give up after 1 ms, and
conduit_test_withhold_v_tile(n) makes the scoring kernel's V producer skip
V tile n of each CTA: no copy and no arrive, an ordinary missed arrive). It
checks through the C ABI that
  * the scoring call returns CONDUIT_OK (the launch itself is fine) and the
    status word then reads CONDUIT_ERR_TIMEOUT with a site bit naming the
    first wait that ran out (the epilogue's for the tile, or the MMA thread's
    or producer's behind it, whichever started waiting first); the scores of
    a timed-out call are undefined, so the finalize step may add
    CONDUIT_FLAG_NONFINITE, and no other bit appears;
  * the same test library, hook off, scores the same batch to the product
    library's result, bitwise;
  * the product library then runs a whole step in the same process and
    matches the oracle, with a clean status word.
"""

import ctypes

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O
from paper_2609_05821_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def libs():
    from paper_2609_05821_gb300 import _build
    _build.build()
    path = _build.build_test_hooks()
    from paper_2609_05821_gb300 import conduit
    test_lib = ctypes.CDLL(path)
    test_lib.conduit_test_withhold_v_tile.argtypes = [ctypes.c_int32]
    test_lib.conduit_test_withhold_v_tile.restype = None
    P = ctypes.c_void_p
    test_lib.conduit_score.argtypes = [P, P, P, P, ctypes.c_int32, P, P, P, P, ctypes.c_size_t, P, P]
    test_lib.conduit_score.restype = ctypes.c_int32
    test_lib.conduit_read_status.argtypes = [P, P, ctypes.POINTER(ctypes.c_int32)]
    test_lib.conduit_read_status.restype = ctypes.c_int32
    return conduit, test_lib


def _batch(C):
    # one layer, 3 images x 256 tokens: 6 key tiles per slab, so each CTA's
    # V producer reaches tile 3
    w = synth.workload("multi", num_layers=1, images_per_request=3, tokens_per_image=256, n_q=16,
                       n_q_lo=16, n_q_hi=16)
    inputs = synth.make_inputs(w, device="cuda")
    kv = C.KvCache(inputs["k"], inputs["v"], w.num_q_heads)
    b = C.Batch(inputs["tok_off"], inputs["img_off"], inputs["req_img_off"], inputs["q_off"], "cuda")
    return w, inputs, kv, b


def _score_with(lib, C, kv, b, q):
    n = b.n_tot
    s = torch.full((n,), -1.0, device="cuda")
    attn = torch.full((n,), -1.0, device="cuda")
    g = torch.full((b.num_images,), -1.0, device="cuda")
    need = C.conduit_score_workspace_size(kv, b, 0)
    ws = torch.empty(max(need, 1), dtype=torch.uint8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    code = lib.conduit_score(kv.ref(), b.ref(), p(q), None, 0, p(s), p(attn), p(g), p(ws), ws.numel(),
                             p(status), stream)
    word = ctypes.c_int32(0)
    read = lib.conduit_read_status(p(status), stream, ctypes.byref(word))
    return code, read, int(word.value), s, attn, g


def test_withheld_tile_times_out_and_the_context_stays_usable(libs):
    C, T = libs
    w, inputs, kv, b = _batch(C)
    T.conduit_test_withhold_v_tile(3)
    try:
        code, read, word, *_ = _score_with(T, C, kv, b, inputs["q"])
    finally:
        T.conduit_test_withhold_v_tile(-1)
    assert code == C.OK                       # the launch itself succeeded
    assert read == C.ERR_TIMEOUT              # the status word reports the wait that ran out
    sites = C.SITE_LOAD | C.SITE_MMA | C.SITE_FINAL
    assert word & C.FLAG_TIMEOUT and word & sites, hex(word)
    assert word & ~(C.FLAG_TIMEOUT | C.FLAG_NONFINITE | sites) == 0, hex(word)

    # the test library, hook off: the same scores as the product library, bitwise
    code, read, word, s_t, a_t, g_t = _score_with(T, C, kv, b, inputs["q"])
    assert code == C.OK and read == C.OK and word == 0
    s_p, a_p, g_p = C.conduit_score(kv, b, inputs["q"])
    torch.cuda.synchronize()
    assert torch.equal(s_t, s_p) and torch.equal(a_t, a_p) and torch.equal(g_t, g_p)

    # the product library runs a whole step after the timeout and matches the oracle
    from paper_2609_05821_gb300 import pipeline
    pipe = pipeline.from_inputs({**inputs, "k": inputs["k"].clone(), "v": inputs["v"].clone()})
    pipe.step()
    torch.cuda.synchronize()
    assert C.conduit_read_status(pipe.status) == C.OK
    view = synth.request_view(inputs, 0)
    ref = O.score_request(view["q"], view["k"], view["v"], view["img_off"])
    s = pipe.s.double().cpu().numpy()
    assert np.all(np.abs(s - ref["s"]) <= 1e-3 * np.abs(ref["s"]) + 1e-7 * np.abs(ref["s"]).max())
