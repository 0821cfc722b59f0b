"""The C ABI on the host: exported symbols and argument checks (no GPU needed).

Every call here fails its host-side checks, which run before anything is
enqueued, so none of them touches a device.
"""

import ctypes
import os
import re
import subprocess

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "conduit.h")


@pytest.fixture(scope="module")
def C():
    from paper_2609_05821_gb300 import _build
    _build.build()
    from paper_2609_05821_gb300 import conduit
    return conduit


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(conduit_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared()
    for want in ("conduit_score", "conduit_select_topk", "conduit_refresh_attn", "conduit_kv_scatter",
                 "conduit_kv_gather", "conduit_budget", "conduit_score_workspace_size",
                 "conduit_read_status", "conduit_value_norms", "conduit_value_norms_update",
                 "conduit_score_with_norms", "conduit_score_with_norms_workspace_size",
                 "conduit_score_ex", "conduit_score_ex_workspace_size",
                 "conduit_select_quota", "conduit_select_quota_workspace_size",
                 "conduit_staleness_iso", "conduit_staleness_iso_workspace_size",
                 "conduit_score_select_topk", "conduit_score_select_topk_workspace_size"):
        assert want in names


def test_library_exports_every_declared_symbol(C):
    lib = ctypes.CDLL(C.LIB_PATH)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert missing == []
    nm = subprocess.run(["nm", "-D", "--defined-only", C.LIB_PATH], capture_output=True, text=True)
    exported = set(re.findall(r"\bT (conduit_[a-z_]+)\b", nm.stdout))
    assert set(_declared()) <= exported


def test_version_and_budget(C):
    assert C.conduit_version() == 100
    assert C.conduit_budget(0.10, 256) == 25
    assert C.conduit_budget(0.10, 1024) == 102
    assert C.conduit_budget(0.05, 41472) == 2073
    assert C.conduit_budget(0.20, 41472) == 8294
    assert C.conduit_budget(0.3, 10) == 3
    assert C.conduit_budget(0.0, 999) == 0
    assert C.conduit_budget(1.0, 999) == 999
    assert C.conduit_budget(-0.01, 10) == -1
    assert C.conduit_budget(1.01, 10) == -1
    assert C.conduit_budget(float("nan"), 10) == -1
    assert C.conduit_budget(0.5, -1) == -1


def test_budget_matches_oracle(C):
    from oracle import conduit_oracle as O
    for r in (0.0, 0.01, 0.05, 0.1, 0.125, 0.2, 0.3, 0.7, 0.99, 1.0):
        for n in (1, 7, 10, 256, 1000, 1024, 8192, 41472):
            assert C.conduit_budget(r, n) == O.budget(r, n)


def _batch(C, tok=(0, 64, 128), img=(0, 32, 64, 128), rio=(0, 2, 3), qo=(0, 4, 8)):
    return C.Batch(list(tok), list(img), list(rio), list(qo), device="cpu")


def _kv(C, L=2, Hq=4, Hkv=2, d=64, n=128, dtype=torch.bfloat16, **kw):
    k = torch.zeros((L, Hkv, n, d), dtype=dtype)
    return C.KvCache(k, torch.zeros_like(k), Hq, **kw)


def _expect(C, code, fn, *args, match=None):
    with pytest.raises(C.ConduitError) as ei:
        fn(*args)
    assert ei.value.code == code, str(ei.value)
    if match:
        assert re.search(match, str(ei.value)), str(ei.value)


def test_score_rejects_bad_arguments(C):
    kv, b = _kv(C), _batch(C)
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    ws = torch.zeros(1, dtype=torch.uint8)
    # workspace too small / missing
    _expect(C, C.ERR_WORKSPACE, C.conduit_score, kv, b, q, None, None, None, None, ws)
    # unsorted images
    bad = _batch(C, img=(0, 70, 64, 128))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="empty or out of order")
    # images that do not tile the request
    bad = _batch(C, img=(0, 32, 60, 128))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="tile")
    # empty request
    bad = _batch(C, tok=(0, 0, 128), img=(0, 0, 64, 128))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q)
    # empty scoring span
    bad = _batch(C, qo=(0, 0, 8))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="scoring span")
    # layer ids
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, b, q, [1, 0], match="increasing")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, b, q, [5], match="out of range")
    # head mismatch
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, _kv(C, Hq=5), b, q, match="multiple")
    # head_dim
    _expect(C, C.ERR_UNSUPPORTED, C.conduit_score, _kv(C, d=12), b, q, match="head_dim")
    # null query
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, b, None)


def test_batch_structure_is_checked(C):
    """Reading c7: every request has visual tokens and images, images are
    non-empty spans that tile their request, offsets start at 0."""
    kv = _kv(C)
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    # a request with tokens but no images
    bad = _batch(C, img=(0, 32, 64), rio=(0, 2, 2))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="no images")
    # the image count of the last request does not close the image list
    bad = _batch(C, rio=(0, 2, 2))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="num_images")
    # offsets that do not start at 0
    bad = _batch(C, tok=(1, 64, 128), img=(1, 32, 64, 128))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score, kv, bad, q, match="start at 0")
    # more images in one request than the selection keeps in shared memory
    n = 4097
    many = C.Batch([0, n], list(range(n + 1)), [0, n], [0, 4], device="cpu")
    _expect(C, C.ERR_UNSUPPORTED, C.conduit_score, _kv(C, n=n), many,
            torch.zeros((2, 4, 4, 64), dtype=torch.bfloat16), match="more than 4096 images")


def test_select_rejects_bad_budgets_and_lambda(C):
    b = _batch(C)
    s = torch.zeros(128)
    g = torch.zeros(3)
    off, off_d = C.idx_offsets([10, 65], "cpu")          # 65 > 64 tokens of request 1
    _expect(C, C.ERR_INVALID_ARG, C.conduit_select_topk, b, s, g, 1.0, off, off_d, match="budget")
    off, off_d = C.idx_offsets([10, 5], "cpu")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_select_topk, b, s, g, 1.5, off, off_d, match="lambda")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_select_topk, b, s, g, float("nan"), off, off_d)
    ws = torch.zeros(8, dtype=torch.uint8)
    _expect(C, C.ERR_WORKSPACE, C.conduit_select_topk, b, s, g, 1.0, off, off_d, None, None, None,
            None, ws)


def test_score_select_rejects_bad_arguments(C):
    """conduit_score_select_topk checks both calls' arguments before it enqueues anything."""
    kv, b = _kv(C), _batch(C)
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    off, off_d = C.idx_offsets([10, 65], "cpu")          # 65 > 64 tokens of request 1
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_select_topk, kv, b, q, 1.0, off, off_d, match="budget")
    off, off_d = C.idx_offsets([10, 5], "cpu")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_select_topk, kv, b, q, 1.5, off, off_d, match="lambda")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_select_topk, kv, b, None, 1.0, off, off_d)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_select_topk, kv, b, q, 1.0, off, off_d, [1, 0],
            match="increasing")
    opts = C.score_opts()
    opts.statistic = 7
    n = ctypes.c_size_t(0)
    assert C._lib.conduit_score_select_topk_workspace_size(kv.ref(), b.ref(), 0, ctypes.byref(opts),
                                                           ctypes.byref(n)) == C.ERR_INVALID_ARG
    bad = _batch(C, qo=(0, 0, 8))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_select_topk, kv, bad, q, 1.0, off, off_d,
            match="scoring span")
    # the workspace is the scoring call's plus a counter per request and the selection's keys
    need = C.conduit_score_select_topk_workspace_size(kv, b)
    assert need >= C.conduit_score_workspace_size(kv, b) + 256 + C.conduit_select_workspace_size(b)
    ws = torch.zeros(need - 256, dtype=torch.uint8)
    _expect(C, C.ERR_WORKSPACE, C.conduit_score_select_topk, kv, b, q, 1.0, off, off_d, None, "mean", "v",
            None, None, None, None, None, None, None, None, None, ws)


def test_quota_select_rejects_bad_arguments(C):
    b = _batch(C)
    s = torch.zeros(128)
    g = torch.zeros(3)
    off, off_d = C.idx_offsets([10, 65], "cpu")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_select_quota, b, s, g, 1.0, off, off_d, match="budget")
    off, off_d = C.idx_offsets([10, 5], "cpu")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_select_quota, b, s, g, -0.5, off, off_d, match="lambda")
    idx = torch.zeros(15, dtype=torch.int32)
    assert C._lib.conduit_select_quota(b.ref(), None, C._ptr(g), 1.0, C._ptr(off), C._ptr(off_d),
                                       C._ptr(idx), None, None, None, None, None, 0, None,
                                       None) == C.ERR_INVALID_ARG
    need = C.conduit_select_quota_workspace_size(b)
    assert need > C.conduit_select_workspace_size(b)        # plus coefficients, quotas, offsets
    ws = torch.zeros(need - 256, dtype=torch.uint8)
    _expect(C, C.ERR_WORKSPACE, C.conduit_select_quota, b, s, g, 1.0, off, off_d, None, None, None,
            None, None, ws)


def test_staleness_rejects_bad_arguments(C):
    kv, b = _kv(C), _batch(C)
    lib = C._lib
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    mask = torch.zeros(128, dtype=torch.uint8)
    z = torch.zeros((2, 2, 2, 128, 64), dtype=torch.bfloat16)
    err = torch.zeros(2, dtype=torch.float64)
    n = ctypes.c_size_t(0)
    assert lib.conduit_staleness_iso_workspace_size(kv.ref(), b.ref(), 0, ctypes.byref(n)) == C.ERR_INVALID_ARG
    assert lib.conduit_staleness_iso_workspace_size(kv.ref(), b.ref(), 2, ctypes.byref(n)) == C.OK
    need = n.value
    assert need > 0

    def call(mq=q, mz=z, M=2, kappa=1.0, ws_bytes=need):
        ws = torch.zeros(max(ws_bytes, 1), dtype=torch.uint8)
        return lib.conduit_staleness_iso(kv.ref(), b.ref(), C._ptr(mq), C._ptr(mask), C._ptr(mz), M, kappa,
                                         C._ptr(err), None, C._ptr(ws) if ws_bytes else None, ws_bytes,
                                         None, None)

    assert call(mz=None) == C.ERR_INVALID_ARG
    assert call(M=0) == C.ERR_INVALID_ARG
    assert call(kappa=-1.0) == C.ERR_INVALID_ARG
    assert call(kappa=float("nan")) == C.ERR_INVALID_ARG
    assert call(ws_bytes=0) == C.ERR_WORKSPACE
    assert call(ws_bytes=need - 256) == C.ERR_WORKSPACE


def test_kv_copy_and_refresh_reject_bad_arguments(C):
    kv, b = _kv(C), _batch(C)
    off, off_d = C.idx_offsets([3, 4], "cpu")
    idx = torch.zeros(7, dtype=torch.int32)
    rows = torch.zeros((2, 7, 2, 64), dtype=torch.bfloat16)
    bad_off = torch.tensor([1, 3, 7], dtype=torch.int32)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_kv_scatter, kv, b, idx, bad_off, off_d, rows, rows)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_kv_gather, kv, b, idx, off, None, rows, rows)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_kv_exchange, kv, b, idx, off, off_d, rows, rows, None, rows)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_kv_exchange, kv, b, idx, bad_off, off_d, rows, rows, rows, rows)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_refresh_attn, kv, b, None, off, off_d, rows)
    paged = torch.zeros((2, 8, 2, 16, 64), dtype=torch.bfloat16)
    table = torch.zeros((2, 3), dtype=torch.int32)      # 3 pages x 16 < 64 tokens
    kvp = C.KvCache(paged, torch.zeros_like(paged), 4, 16, table)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_kv_scatter, kvp, b, idx, off, off_d, rows, rows,
            match="page-table")


def test_norm_side_cache_rejects_bad_arguments(C):
    kv, b = _kv(C), _batch(C)
    lib = C._lib
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    vn = torch.zeros((2, 128))
    # a NULL or misaligned side cache
    assert lib.conduit_value_norms(kv.ref(), b.ref(), None, None) == C.ERR_INVALID_ARG
    assert "vnorm" in lib.conduit_last_error_string().decode()
    odd = ctypes.c_void_p(vn.data_ptr() + 2)
    assert lib.conduit_value_norms(kv.ref(), b.ref(), odd, None) == C.ERR_INVALID_ARG
    # the batch and cache checks of the scoring pass apply
    bad = _batch(C, img=(0, 70, 64, 128))
    _expect(C, C.ERR_INVALID_ARG, C.conduit_value_norms, kv, bad, vn, match="empty or out of order")
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_with_norms, kv, bad, q, vn)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_score_with_norms, kv, b, q, vn, [1, 0], match="increasing")
    # the update takes a selection like the scatter
    off, off_d = C.idx_offsets([3, 4], "cpu")
    bad_off = torch.tensor([1, 3, 7], dtype=torch.int32)
    idx = torch.zeros(7, dtype=torch.int32)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_value_norms_update, kv, b, idx, bad_off, off_d, vn)
    _expect(C, C.ERR_INVALID_ARG, C.conduit_value_norms_update, kv, b, None, off, off_d, vn)
    assert lib.conduit_value_norms_update(kv.ref(), b.ref(), C._ptr(idx), C._ptr(off), C._ptr(off_d),
                                          None, None) == C.ERR_INVALID_ARG
    # workspace: the normed pass has no value partials, so it needs less
    full = C.conduit_score_workspace_size(kv, b)
    normed = C.conduit_score_with_norms_workspace_size(kv, b)
    assert 0 < normed < full
    ws = torch.zeros(normed - 256, dtype=torch.uint8)
    _expect(C, C.ERR_WORKSPACE, C.conduit_score_with_norms, kv, b, q, vn, None, None, None, None, ws)
    assert lib.conduit_score_with_norms(kv.ref(), b.ref(), C._ptr(q), None, 0, None, C._ptr(vn),
                                        C._ptr(vn), C._ptr(vn), None, 0, None, None) == C.ERR_INVALID_ARG


def test_score_options_are_checked(C):
    kv, b = _kv(C), _batch(C)
    lib = C._lib
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    vn = torch.zeros((2, 128))
    out = torch.zeros(128)

    def call(opts, ws=None):
        n = ctypes.c_size_t(0)
        rc = lib.conduit_score_ex_workspace_size(kv.ref(), b.ref(), 0, ctypes.byref(opts), ctypes.byref(n))
        if ws is None:
            return rc
        return lib.conduit_score_ex(kv.ref(), b.ref(), C._ptr(q), None, 0, ctypes.byref(opts), C._ptr(out),
                                    C._ptr(out), C._ptr(out), C._ptr(ws), ws.numel(), None, None)

    bad = C.score_opts()
    bad.statistic = 7
    assert call(bad) == C.ERR_INVALID_ARG and "statistic" in lib.conduit_last_error_string().decode()
    bad = C.score_opts()
    bad.value_norm = 3
    assert call(bad) == C.ERR_INVALID_ARG
    assert call(C.score_opts(value_norm="side_cache")) == C.ERR_INVALID_ARG      # no vnorm
    assert call(C.score_opts(value_norm="v", vnorm=vn)) == C.ERR_INVALID_ARG     # vnorm not used
    odd = C.score_opts()
    odd.extra_lse = vn.data_ptr() + 2
    assert call(odd) == C.ERR_INVALID_ARG
    # workspace sizes: NULL options = conduit_score; RMS adds, dropping V's partials removes
    n = ctypes.c_size_t(0)
    assert lib.conduit_score_ex_workspace_size(kv.ref(), b.ref(), 0, None, ctypes.byref(n)) == C.OK
    base = C.conduit_score_workspace_size(kv, b)
    assert n.value == base
    rms = C.conduit_score_ex_workspace_size(kv, b, 0, C.score_opts(statistic="rms"))
    none = C.conduit_score_ex_workspace_size(kv, b, 0, C.score_opts(value_norm="none"))
    side = C.conduit_score_ex_workspace_size(kv, b, 0, C.score_opts(value_norm="side_cache", vnorm=vn))
    assert rms > base > none == side == C.conduit_score_with_norms_workspace_size(kv, b)
    # a workspace sized for the mean is short for the RMS statistic
    ws = torch.zeros(base, dtype=torch.uint8)
    assert call(C.score_opts(statistic="rms"), ws) == C.ERR_WORKSPACE


def test_kv_cache_python_checks(C):
    k = torch.zeros((1, 2, 8, 64), dtype=torch.float16)
    _expect(C, C.ERR_UNSUPPORTED, C.KvCache, k, k.clone(), 2)
    k = torch.zeros((1, 2, 8, 64))
    _expect(C, C.ERR_INVALID_ARG, C.KvCache, k, torch.zeros((1, 2, 8, 32)), 2)


def test_last_error_is_thread_local(C):
    import threading
    kv, b = _kv(C), _batch(C)
    q = torch.zeros((2, 4, 8, 64), dtype=torch.bfloat16)
    with pytest.raises(C.ConduitError):
        C.conduit_score(kv, b, q, [9])
    main_msg = C._lib.conduit_last_error_string().decode()
    seen = []
    t = threading.Thread(target=lambda: seen.append(C._lib.conduit_last_error_string().decode()))
    t.start()
    t.join()
    assert seen == [""] and "out of range" in main_msg


def test_noalloc_limit_is_the_header_value(C):
    """The binding's limit of conduit_select_topk_noalloc is the header's
    CONDUIT_NOALLOC_MAX_TOKENS (the library sizes its static array from it)."""
    m = re.search(r"#define\s+CONDUIT_NOALLOC_MAX_TOKENS\s+\(1\s*<<\s*(\d+)\)", open(HEADER).read())
    assert m is not None
    assert C.NOALLOC_MAX_TOKENS == 1 << int(m.group(1))
    src = open(os.path.join(ROOT, "paper_2609_05821_gb300", "csrc", "select.cu")).read()
    assert re.search(r"kNoAllocMaxTokens\s*=\s*CONDUIT_NOALLOC_MAX_TOKENS\s*;", src)


def test_status_bits_are_the_header_values(C):
    text = open(HEADER).read()
    for name, val in (("CONDUIT_FLAG_NONFINITE", C.FLAG_NONFINITE), ("CONDUIT_FLAG_TIMEOUT", C.FLAG_TIMEOUT),
                      ("CONDUIT_SITE_LOAD", C.SITE_LOAD), ("CONDUIT_SITE_MMA", C.SITE_MMA),
                      ("CONDUIT_SITE_FINAL", C.SITE_FINAL)):
        m = re.search(name + r"\s*=\s*([0-9]+)(?:\s*<<\s*([0-9]+))?", text)
        assert m is not None, name
        assert val == int(m.group(1)) << int(m.group(2) or 0), name


def test_product_library_has_no_test_hooks(C):
    lib = ctypes.CDLL(C.LIB_PATH)
    assert not hasattr(lib, "conduit_test_withhold_v_tile")
