"""Seeded generators: determinism, shapes, and the paged re-layout."""

import torch

from paper_2609_05821_gb300 import synth


def _small(name, **kw):
    return synth.workload(name, **kw)


def test_deterministic_and_shaped():
    w = _small("multi", num_layers=2, tokens_per_image=64, images_per_request=3)
    a = synth.make_inputs(w)
    b = synth.make_inputs(w)
    for key in ("q", "k", "v"):
        assert torch.equal(a[key], b[key])
    assert a["k"].shape == (2, 4, 192, 128) and a["k"].dtype == torch.bfloat16
    assert a["q"].shape == (2, 28, 64, 128)
    assert a["img_off"].tolist() == [0, 64, 128, 192]
    c = synth.make_inputs(w, seed=99)
    assert not torch.equal(a["k"], c["k"])


def test_tiny_is_fp32_with_planted_tokens():
    a = synth.make_inputs(synth.workload("tiny"))
    assert a["k"].dtype == torch.float32 and a["k"].shape == (1, 2, 256, 64)
    n = a["k"].float().norm(dim=-1)                       # planted keys are long: 3 sqrt(d)
    assert int((n[0, 0] > 20).sum()) == 8


def test_batched_offsets_and_paged_relayout():
    w = _small("batched", num_requests=3, num_layers=2, tokens_per_image=32)
    a = synth.make_inputs(w)
    assert a["tok_off"].tolist() == [0, 128, 256, 384]
    assert all(32 <= n <= 128 for n in a["n_q"])
    assert a["q_off"].tolist()[-1] == sum(a["n_q"])
    pool, table = synth.to_paged(a["k"], a["tok_off"].tolist(), 16, w.seed)
    L, P, Hkv, ps, d = pool.shape
    assert (L, P, Hkv, ps, d) == (2, 24, 4, 16, 128)
    tok = a["tok_off"].tolist()
    for r in range(3):
        for t in (0, 17, 127):
            page = int(table[r, t // 16])
            assert torch.equal(pool[:, page, :, t % 16, :], a["k"][:, :, tok[r] + t, :])
    assert sorted(table.flatten().tolist()) == list(range(P))
