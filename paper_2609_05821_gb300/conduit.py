"""Thin Python binding of the libconduit C ABI (include/conduit.h).

Each ``conduit_*`` function here marshals torch tensors into the pointers and
sizes of the C call of the same name and raises ``ConduitError`` on a non-OK
status. Every step of the computation runs in the CUDA library; this module
only allocates outputs and workspaces with torch when the caller passes none.
There is no fallback: a missing library raises on import.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libconduit.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_NONFINITE, ERR_TIMEOUT, ERR_WORKSPACE = range(7)
FLAG_NONFINITE, FLAG_TIMEOUT = 1, 2
# with FLAG_TIMEOUT, the wait that ran out: a TMA tile, an MMA completion, an item's final MMA
SITE_LOAD, SITE_MMA, SITE_FINAL = 1 << 8, 1 << 9, 1 << 10
F32, BF16 = 0, 1
MAX_LAYERS = 512
STAT_MEAN, STAT_RMS = 0, 1
VNORM_FROM_V, VNORM_SIDE_CACHE, VNORM_NONE = 0, 1, 2
_STATS = {"mean": STAT_MEAN, "rms": STAT_RMS}
_VNORMS = {"v": VNORM_FROM_V, "side_cache": VNORM_SIDE_CACHE, "none": VNORM_NONE}

_STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "NONFINITE",
                 5: "TIMEOUT", 6: "WORKSPACE"}


class ConduitError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"conduit {_STATUS_NAMES.get(code, code)}: {message}")
        self.code = code


class ConduitKV(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("dtype", ctypes.c_int32), ("page_size", ctypes.c_int32),
        ("num_pages", ctypes.c_int32), ("max_pages_per_req", ctypes.c_int32),
        ("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
    ]


class ConduitScoreOpts(ctypes.Structure):
    _fields_ = [
        ("statistic", ctypes.c_int32), ("value_norm", ctypes.c_int32),
        ("vnorm", ctypes.c_void_p), ("extra_lse", ctypes.c_void_p),
    ]


class ConduitBatch(ctypes.Structure):
    _fields_ = [
        ("num_requests", ctypes.c_int32), ("num_images", ctypes.c_int32),
        ("tok_off", ctypes.c_void_p), ("img_off", ctypes.c_void_p),
        ("req_img_off", ctypes.c_void_p), ("q_off", ctypes.c_void_p),
        ("tok_off_dev", ctypes.c_void_p), ("img_off_dev", ctypes.c_void_p),
        ("req_img_off_dev", ctypes.c_void_p), ("q_off_dev", ctypes.c_void_p),
    ]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"libconduit.so is not built ({LIB_PATH}); run "
            "`python -c 'import __graft_entry__ as g; g.build()'` first")
    lib = ctypes.CDLL(LIB_PATH)
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    st = ctypes.c_int32
    sig = {
        "conduit_version": (I32, []),
        "conduit_last_error_string": (ctypes.c_char_p, []),
        "conduit_budget": (I32, [ctypes.c_double, ctypes.c_int64]),
        "conduit_score_workspace_size": (st, [P, P, I32, ctypes.POINTER(SZ)]),
        "conduit_score": (st, [P, P, P, P, I32, P, P, P, P, SZ, P, P]),
        "conduit_score_ex_workspace_size": (st, [P, P, I32, P, ctypes.POINTER(SZ)]),
        "conduit_score_ex": (st, [P, P, P, P, I32, P, P, P, P, P, SZ, P, P]),
        "conduit_staleness_iso_workspace_size": (st, [P, P, I32, ctypes.POINTER(SZ)]),
        "conduit_staleness_iso": (st, [P, P, P, P, P, I32, ctypes.c_float, P, P, P, SZ, P, P]),
        "conduit_value_norms": (st, [P, P, P, P]),
        "conduit_value_norms_update": (st, [P, P, P, P, P, P, P]),
        "conduit_score_with_norms_workspace_size": (st, [P, P, I32, ctypes.POINTER(SZ)]),
        "conduit_score_with_norms": (st, [P, P, P, P, I32, P, P, P, P, P, SZ, P, P]),
        "conduit_score_select_topk_workspace_size": (st, [P, P, I32, P, ctypes.POINTER(SZ)]),
        "conduit_score_select_topk": (st, [P, P, P, P, I32, P, ctypes.c_float, P, P, P, P, P, P, P, P,
                                           P, P, SZ, P, P]),
        "conduit_select_workspace_size": (st, [P, ctypes.POINTER(SZ)]),
        "conduit_select_topk": (st, [P, P, P, ctypes.c_float, P, P, P, P, P, P, P, SZ, P, P]),
        "conduit_select_topk_noalloc": (st, [P, P, P, ctypes.c_float, P, P, P, P, P, P, P, P]),
        "conduit_select_quota_workspace_size": (st, [P, ctypes.POINTER(SZ)]),
        "conduit_select_quota": (st, [P, P, P, ctypes.c_float, P, P, P, P, P, P, P, P, SZ, P, P]),
        "conduit_kv_gather": (st, [P, P, P, P, P, P, P, P]),
        "conduit_kv_scatter": (st, [P, P, P, P, P, P, P, P]),
        "conduit_kv_exchange": (st, [P, P, P, P, P, P, P, P, P, P]),
        "conduit_refresh_workspace_size": (st, [P, P, P, ctypes.POINTER(SZ)]),
        "conduit_refresh_attn": (st, [P, P, P, P, P, P, P, P, SZ, P, P]),
        "conduit_launch_count": (ctypes.c_int64, []),
        "conduit_clear_status": (st, [P, P]),
        "conduit_read_status": (st, [P, P, ctypes.POINTER(I32)]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype, fn.argtypes = res, args
    return lib


_lib = _load()


def _check(code: int):
    if code != OK:
        raise ConduitError(code, _lib.conduit_last_error_string().decode())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream_ptr(stream) -> Optional[ctypes.c_void_p]:
    if stream is None:
        if not torch.cuda.is_available():
            return None  # argument checks run before any stream use
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise ConduitError(ERR_UNSUPPORTED, f"dtype {t.dtype} (fp32 and bf16 only)")


class Batch:
    """Request / image / query offsets on host and device (conduit_batch)."""

    def __init__(self, tok_off, img_off, req_img_off, q_off, device="cuda"):
        as_host = lambda x: torch.as_tensor(x, dtype=torch.int32).contiguous().cpu()
        self.tok_off, self.img_off = as_host(tok_off), as_host(img_off)
        self.req_img_off, self.q_off = as_host(req_img_off), as_host(q_off)
        dev = torch.device(device)
        self.tok_off_dev = self.tok_off.to(dev)
        self.img_off_dev = self.img_off.to(dev)
        self.req_img_off_dev = self.req_img_off.to(dev)
        self.q_off_dev = self.q_off.to(dev)
        self.num_requests = self.tok_off.numel() - 1
        self.num_images = self.img_off.numel() - 1
        self.struct = ConduitBatch(
            self.num_requests, self.num_images,
            self.tok_off.data_ptr(), self.img_off.data_ptr(),
            self.req_img_off.data_ptr(), self.q_off.data_ptr(),
            self.tok_off_dev.data_ptr(), self.img_off_dev.data_ptr(),
            self.req_img_off_dev.data_ptr(), self.q_off_dev.data_ptr())

    @property
    def n_tot(self) -> int:
        return int(self.tok_off[-1])

    @property
    def q_tot(self) -> int:
        return int(self.q_off[-1])

    def ref(self):
        return ctypes.byref(self.struct)


class KvCache:
    """A contiguous [L][Hkv][N_tot][d] or paged [L][P][Hkv][page][d] K/V cache (conduit_kv)."""

    def __init__(self, k: torch.Tensor, v: torch.Tensor, num_q_heads: int, page_size: int = 0,
                 page_table: Optional[torch.Tensor] = None):
        if k.shape != v.shape or k.dtype != v.dtype:
            raise ConduitError(ERR_INVALID_ARG, "k and v must have equal shapes and dtypes")
        if not (k.is_contiguous() and v.is_contiguous()):
            raise ConduitError(ERR_INVALID_ARG, "k and v must be contiguous")
        self.k, self.v, self.page_table = k, v, page_table
        L = k.shape[0]
        if page_size:
            _, P, Hkv, ps, d = k.shape
            if ps != page_size:
                raise ConduitError(ERR_INVALID_ARG, "pool page dimension != page_size")
            if page_table is None:
                raise ConduitError(ERR_INVALID_ARG, "a paged cache needs a page table")
            self.page_table = page_table.to(device=k.device, dtype=torch.int32).contiguous()
            max_pages = self.page_table.shape[1]
        else:
            _, Hkv, _, d = k.shape
            P, max_pages = 0, 0
        self.num_layers, self.num_kv_heads, self.head_dim = L, Hkv, d
        self.num_q_heads = num_q_heads
        self.struct = ConduitKV(L, num_q_heads, Hkv, d, _dtype_code(k), page_size, P, max_pages,
                                k.data_ptr(), v.data_ptr(),
                                self.page_table.data_ptr() if page_size else None)

    @property
    def dtype(self):
        return self.k.dtype

    def ref(self):
        return ctypes.byref(self.struct)


def conduit_version() -> int:
    return int(_lib.conduit_version())


def conduit_launch_count() -> int:
    """Kernels the library has enqueued in this process (launched or captured)."""
    return int(_lib.conduit_launch_count())


def conduit_budget(r: float, n_vis: int) -> int:
    return int(_lib.conduit_budget(float(r), int(n_vis)))


def _layer_array(layers: Optional[Sequence[int]]):
    if layers is None:
        return None, 0
    arr = (ctypes.c_int32 * len(layers))(*[int(x) for x in layers])
    return arr, len(layers)


def conduit_score_workspace_size(kv: KvCache, batch: Batch, n_layers: int = 0) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_score_workspace_size(kv.ref(), batch.ref(), int(n_layers), ctypes.byref(n)))
    return int(n.value)


def _workspace(nbytes: int, device, ws: Optional[torch.Tensor]) -> torch.Tensor:
    if ws is not None:
        return ws
    return torch.empty(max(nbytes, 1), dtype=torch.uint8, device=device)


def conduit_score(kv: KvCache, batch: Batch, q: torch.Tensor, layers=None, s=None, attn_sum=None,
                  g=None, workspace=None, status=None, stream=None):
    """Scoring pass (Eqs. 6-8). Returns (s [N_tot], attn_sum [N_tot], g [K]) fp32."""
    dev = kv.k.device
    larr, nl = _layer_array(layers)
    s = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if s is None else s
    attn_sum = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if attn_sum is None else attn_sum
    g = torch.empty(batch.num_images, dtype=torch.float32, device=dev) if g is None else g
    need = conduit_score_workspace_size(kv, batch, nl)
    ws = _workspace(need, dev, workspace)
    _check(_lib.conduit_score(kv.ref(), batch.ref(), _ptr(q), larr, nl, _ptr(s), _ptr(attn_sum),
                              _ptr(g), _ptr(ws), ws.numel(), _ptr(status), _stream_ptr(stream)))
    return s, attn_sum, g


def score_opts(statistic: str = "mean", value_norm: str = "v", vnorm=None, extra_lse=None):
    """conduit_score_opts: statistic "mean" | "rms", value_norm "v" | "side_cache" | "none"."""
    o = ConduitScoreOpts()
    o.statistic = _STATS[statistic]
    o.value_norm = _VNORMS[value_norm]
    o.vnorm = None if vnorm is None else vnorm.data_ptr()
    o.extra_lse = None if extra_lse is None else extra_lse.data_ptr()
    return o


def conduit_score_ex_workspace_size(kv: KvCache, batch: Batch, n_layers: int = 0,
                                    opts: Optional[ConduitScoreOpts] = None) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_score_ex_workspace_size(kv.ref(), batch.ref(), int(n_layers),
                                                None if opts is None else ctypes.byref(opts),
                                                ctypes.byref(n)))
    return int(n.value)


def conduit_score_ex(kv: KvCache, batch: Batch, q: torch.Tensor, layers=None, statistic="mean",
                     value_norm="v", vnorm=None, extra_lse=None, s=None, attn_sum=None, g=None,
                     workspace=None, status=None, stream=None):
    """Scoring pass with the variants of conduit_score_opts. Returns (s, attn_sum, g)."""
    dev = kv.k.device
    larr, nl = _layer_array(layers)
    opts = score_opts(statistic, value_norm, vnorm, extra_lse)
    s = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if s is None else s
    attn_sum = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if attn_sum is None else attn_sum
    g = torch.empty(batch.num_images, dtype=torch.float32, device=dev) if g is None else g
    ws = _workspace(conduit_score_ex_workspace_size(kv, batch, nl, opts), dev, workspace)
    _check(_lib.conduit_score_ex(kv.ref(), batch.ref(), _ptr(q), larr, nl, ctypes.byref(opts),
                                 _ptr(s), _ptr(attn_sum), _ptr(g), _ptr(ws), ws.numel(),
                                 _ptr(status), _stream_ptr(stream)))
    return s, attn_sum, g


def conduit_score_select_topk_workspace_size(kv: KvCache, batch: Batch, n_layers: int = 0,
                                             opts: Optional[ConduitScoreOpts] = None) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_score_select_topk_workspace_size(kv.ref(), batch.ref(), int(n_layers),
                                                         None if opts is None else ctypes.byref(opts),
                                                         ctypes.byref(n)))
    return int(n.value)


def conduit_score_select_topk(kv: KvCache, batch: Batch, q: torch.Tensor, lam: float,
                              idx_off: torch.Tensor, idx_off_dev: torch.Tensor, layers=None,
                              statistic="mean", value_norm="v", vnorm=None, extra_lse=None, s=None,
                              attn_sum=None, g=None, idx=None, mask=None, s_hat=None, coeff=None,
                              workspace=None, status=None, stream=None):
    """Scoring and global top-k in one call (Eqs. 6-11): conduit_score_ex then
    conduit_select_topk, bitwise, in fewer launches.
    Returns (s, attn_sum, g, idx, mask, s_hat, coeff)."""
    dev = kv.k.device
    larr, nl = _layer_array(layers)
    opts = score_opts(statistic, value_norm, vnorm, extra_lse)
    s = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if s is None else s
    attn_sum = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if attn_sum is None else attn_sum
    g = torch.empty(batch.num_images, dtype=torch.float32, device=dev) if g is None else g
    n_sel = int(idx_off[-1])
    idx = torch.empty(max(n_sel, 1), dtype=torch.int32, device=dev) if idx is None else idx
    ws = _workspace(conduit_score_select_topk_workspace_size(kv, batch, nl, opts), dev, workspace)
    _check(_lib.conduit_score_select_topk(kv.ref(), batch.ref(), _ptr(q), larr, nl, ctypes.byref(opts),
                                          float(lam), _ptr(idx_off), _ptr(idx_off_dev), _ptr(s),
                                          _ptr(attn_sum), _ptr(g), _ptr(idx), _ptr(mask), _ptr(s_hat),
                                          _ptr(coeff), _ptr(ws), ws.numel(), _ptr(status),
                                          _stream_ptr(stream)))
    return s, attn_sum, g, idx[:n_sel], mask, s_hat, coeff


def conduit_staleness_iso_workspace_size(kv: KvCache, batch: Batch, M: int) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_staleness_iso_workspace_size(kv.ref(), batch.ref(), int(M), ctypes.byref(n)))
    return int(n.value)


def conduit_staleness_iso(kv: KvCache, batch: Batch, q: torch.Tensor, refreshed: torch.Tensor,
                          z: torch.Tensor, kappa: float, err=None, err_layers=None, workspace=None,
                          status=None, stream=None):
    """Isotropic Monte Carlo staleness of a refresh set (App. D). z: [M][L][Hkv][N_tot][d].
    Returns (err [R], err_layers [R, L] or None), float64."""
    dev = kv.k.device
    M = int(z.shape[0])
    err = torch.empty(batch.num_requests, dtype=torch.float64, device=dev) if err is None else err
    ws = _workspace(conduit_staleness_iso_workspace_size(kv, batch, M), dev, workspace)
    _check(_lib.conduit_staleness_iso(kv.ref(), batch.ref(), _ptr(q), _ptr(refreshed), _ptr(z), M,
                                      float(kappa), _ptr(err), _ptr(err_layers), _ptr(ws), ws.numel(),
                                      _ptr(status), _stream_ptr(stream)))
    return err, err_layers


def conduit_value_norms(kv: KvCache, batch: Batch, vnorm=None, stream=None) -> torch.Tensor:
    """Value-norm side cache vnorm[l][t] = ||concat_g V[l][g][t]|| (fp32 [L, N_tot])."""
    if vnorm is None:
        vnorm = torch.empty((kv.num_layers, batch.n_tot), dtype=torch.float32, device=kv.k.device)
    _check(_lib.conduit_value_norms(kv.ref(), batch.ref(), _ptr(vnorm), _stream_ptr(stream)))
    return vnorm


def conduit_value_norms_update(kv: KvCache, batch: Batch, idx, idx_off, idx_off_dev, vnorm,
                               stream=None):
    """Recompute the side-cache entries of the selected rows (after a scatter or exchange)."""
    _check(_lib.conduit_value_norms_update(kv.ref(), batch.ref(), _ptr(idx), _ptr(idx_off),
                                           _ptr(idx_off_dev), _ptr(vnorm), _stream_ptr(stream)))


def conduit_score_with_norms_workspace_size(kv: KvCache, batch: Batch, n_layers: int = 0) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_score_with_norms_workspace_size(kv.ref(), batch.ref(), int(n_layers),
                                                        ctypes.byref(n)))
    return int(n.value)


def conduit_score_with_norms(kv: KvCache, batch: Batch, q: torch.Tensor, vnorm: torch.Tensor,
                             layers=None, s=None, attn_sum=None, g=None, workspace=None,
                             status=None, stream=None):
    """Scoring pass with the value norms from the side cache; V is not read."""
    dev = kv.k.device
    larr, nl = _layer_array(layers)
    s = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if s is None else s
    attn_sum = torch.empty(batch.n_tot, dtype=torch.float32, device=dev) if attn_sum is None else attn_sum
    g = torch.empty(batch.num_images, dtype=torch.float32, device=dev) if g is None else g
    need = conduit_score_with_norms_workspace_size(kv, batch, nl)
    ws = _workspace(need, dev, workspace)
    _check(_lib.conduit_score_with_norms(kv.ref(), batch.ref(), _ptr(q), larr, nl, _ptr(vnorm),
                                         _ptr(s), _ptr(attn_sum), _ptr(g), _ptr(ws), ws.numel(),
                                         _ptr(status), _stream_ptr(stream)))
    return s, attn_sum, g


def conduit_select_workspace_size(batch: Batch) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_select_workspace_size(batch.ref(), ctypes.byref(n)))
    return int(n.value)


def idx_offsets(budgets: Sequence[int], device="cuda"):
    """Host and device prefix sums [R+1] of per-request budgets."""
    off = [0]
    for k in budgets:
        off.append(off[-1] + int(k))
    host = torch.tensor(off, dtype=torch.int32)
    return host, host.to(device)


def conduit_select_topk(batch: Batch, s: torch.Tensor, g: torch.Tensor, lam: float,
                        idx_off: torch.Tensor, idx_off_dev: torch.Tensor, idx=None, mask=None,
                        s_hat=None, coeff=None, workspace=None, status=None, stream=None):
    """Amplification + global top-k (Eqs. 9-11). Returns (idx, mask, s_hat, coeff)."""
    dev = s.device
    n_sel = int(idx_off[-1])
    idx = torch.empty(max(n_sel, 1), dtype=torch.int32, device=dev) if idx is None else idx
    need = conduit_select_workspace_size(batch)
    ws = _workspace(need, dev, workspace)
    _check(_lib.conduit_select_topk(batch.ref(), _ptr(s), _ptr(g), float(lam), _ptr(idx_off),
                                    _ptr(idx_off_dev), _ptr(idx), _ptr(mask), _ptr(s_hat),
                                    _ptr(coeff), _ptr(ws), ws.numel(), _ptr(status),
                                    _stream_ptr(stream)))
    return idx[:n_sel], mask, s_hat, coeff


def conduit_select_quota_workspace_size(batch: Batch) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_select_quota_workspace_size(batch.ref(), ctypes.byref(n)))
    return int(n.value)


def conduit_select_quota(batch: Batch, s: torch.Tensor, g: torch.Tensor, lam: float,
                         idx_off: torch.Tensor, idx_off_dev: torch.Tensor, idx=None, mask=None,
                         s_hat=None, coeff=None, quota=None, workspace=None, status=None,
                         stream=None):
    """Explicit per-image quotas (App. D.3). Returns (idx, mask, s_hat, coeff, quota)."""
    dev = s.device
    n_sel = int(idx_off[-1])
    idx = torch.empty(max(n_sel, 1), dtype=torch.int32, device=dev) if idx is None else idx
    ws = _workspace(conduit_select_quota_workspace_size(batch), dev, workspace)
    _check(_lib.conduit_select_quota(batch.ref(), _ptr(s), _ptr(g), float(lam), _ptr(idx_off),
                                     _ptr(idx_off_dev), _ptr(idx), _ptr(mask), _ptr(s_hat),
                                     _ptr(coeff), _ptr(quota), _ptr(ws), ws.numel(), _ptr(status),
                                     _stream_ptr(stream)))
    return idx[:n_sel], mask, s_hat, coeff, quota


NOALLOC_MAX_TOKENS = 1 << 20


def conduit_select_topk_noalloc(batch: Batch, s: torch.Tensor, g: torch.Tensor, lam: float,
                                idx_off: torch.Tensor, idx_off_dev: torch.Tensor, idx: torch.Tensor,
                                mask=None, s_hat=None, coeff=None, status=None, stream=None):
    """conduit_select_topk with the library's static scratch instead of a workspace.

    For callers that cannot give the library device scratch memory. Outputs
    must be preallocated by the caller; nothing here or in the C call allocates.
    """
    _check(_lib.conduit_select_topk_noalloc(batch.ref(), _ptr(s), _ptr(g), float(lam),
                                            _ptr(idx_off), _ptr(idx_off_dev), _ptr(idx),
                                            _ptr(mask), _ptr(s_hat), _ptr(coeff), _ptr(status),
                                            _stream_ptr(stream)))
    return idx, mask, s_hat, coeff


def conduit_kv_gather(kv: KvCache, batch: Batch, idx, idx_off, idx_off_dev, k_rows=None,
                      v_rows=None, stream=None):
    n_sel = int(idx_off[-1])
    shape = (kv.num_layers, n_sel, kv.num_kv_heads, kv.head_dim)
    k_rows = torch.empty(shape, dtype=kv.dtype, device=kv.k.device) if k_rows is None else k_rows
    v_rows = torch.empty(shape, dtype=kv.dtype, device=kv.k.device) if v_rows is None else v_rows
    _check(_lib.conduit_kv_gather(kv.ref(), batch.ref(), _ptr(idx), _ptr(idx_off),
                                  _ptr(idx_off_dev), _ptr(k_rows), _ptr(v_rows), _stream_ptr(stream)))
    return k_rows, v_rows


def conduit_kv_scatter(kv: KvCache, batch: Batch, idx, idx_off, idx_off_dev, k_rows, v_rows,
                       stream=None):
    _check(_lib.conduit_kv_scatter(kv.ref(), batch.ref(), _ptr(idx), _ptr(idx_off),
                                   _ptr(idx_off_dev), _ptr(k_rows), _ptr(v_rows), _stream_ptr(stream)))


def conduit_kv_exchange(kv: KvCache, batch: Batch, idx, idx_off, idx_off_dev, k_old, v_old,
                        k_rows, v_rows, stream=None):
    """Stale rows of the selected tokens into k_old / v_old, fresh rows into the cache."""
    _check(_lib.conduit_kv_exchange(kv.ref(), batch.ref(), _ptr(idx), _ptr(idx_off),
                                    _ptr(idx_off_dev), _ptr(k_old), _ptr(v_old), _ptr(k_rows),
                                    _ptr(v_rows), _stream_ptr(stream)))


def conduit_refresh_workspace_size(kv: KvCache, batch: Batch, idx_off) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.conduit_refresh_workspace_size(kv.ref(), batch.ref(), _ptr(idx_off), ctypes.byref(n)))
    return int(n.value)


def conduit_refresh_attn(kv: KvCache, batch: Batch, idx, idx_off, idx_off_dev, q_rows, out=None,
                         workspace=None, status=None, stream=None):
    """Causal attention of the refreshed rows over the patched cache."""
    out = torch.empty_like(q_rows) if out is None else out
    need = conduit_refresh_workspace_size(kv, batch, idx_off)
    ws = workspace if (workspace is not None or need == 0) else _workspace(need, kv.k.device, None)
    _check(_lib.conduit_refresh_attn(kv.ref(), batch.ref(), _ptr(idx), _ptr(idx_off),
                                     _ptr(idx_off_dev), _ptr(q_rows), _ptr(out), _ptr(ws),
                                     0 if ws is None else ws.numel(), _ptr(status),
                                     _stream_ptr(stream)))
    return out


def conduit_clear_status(status: torch.Tensor, stream=None):
    _check(_lib.conduit_clear_status(_ptr(status), _stream_ptr(stream)))


def conduit_read_status(status: torch.Tensor, stream=None) -> int:
    """Synchronises the stream; returns OK, ERR_NONFINITE or ERR_TIMEOUT (no raise)."""
    word = ctypes.c_int32(0)
    code = _lib.conduit_read_status(_ptr(status), _stream_ptr(stream), ctypes.byref(word))
    if code not in (OK, ERR_NONFINITE, ERR_TIMEOUT):
        _check(code)
    return int(code)
