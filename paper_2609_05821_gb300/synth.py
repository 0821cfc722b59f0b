"""Seeded synthetic visual KV caches shaped like the paper's workloads.

This module only draws random inputs and lays them out; it holds none of the
scoring, selection or attention arithmetic, and both the CUDA path's tests and
the CPU oracle's tests take their inputs from it.

Workloads (they stand in for the benchmark suites of Sec. 4.1, which are not
used): a tiny fp32 case, one high-resolution image (thousand-plus tokens per
image, Sec. 1), a multi-image prompt, a long document of page images, and a
batch of paged serving requests (paged KV storage, Sec. 4.3).

Value laws:
  * tiny: Q, K ~ N(0, 1); V_t = rho_t z_t/||z_t|| on the concatenated Hkv*d
    vector, rho_t ~ sqrt(Hkv d) LogNormal(0, 0.5); eight planted tokens take
    K = 3 sqrt(d) u_g + N(0, 0.1^2) (u_g the unit mean of KV group g's query
    rows) and rho x 0.05 (high attention, small value norm).
  * others: per (layer, KV head) a unit direction u; queries of that group are
    0.5 sqrt(d) u + N(0, I); keys N(0, I) with 5 % of tokens replaced by
    ||k|| (0.6 u + 0.8 w), w a unit vector orthogonal to u (cosine 0.6 with
    the query direction); query-relevant images add 0.25 sqrt(d) u to every
    key; rho ~ sqrt(Hkv d) LogNormal(0, 0.7). Long-document pages start with
    four sink tokens, K = 1.5 sqrt(d) u + N(0, I) and rho x 0.02.
  * fresh rows for the refresh step (queries, keys and values of the
    recomputed tokens) are N(0, 1).
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence

import torch

__all__ = ["Workload", "WORKLOADS", "workload", "make_inputs", "make_fresh_rows",
           "make_extra_lse", "to_paged", "request_view"]


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    images_per_request: int
    tokens_per_image: int
    num_requests: int
    n_q: Optional[int]             # fixed query-span length, or None for U{n_q_lo..n_q_hi}
    n_q_lo: int
    n_q_hi: int
    dtype: str                     # "f32" or "bf16"
    seed: int
    ratios: Sequence[float]        # refresh ratios r (per request drawn from this set when batched)
    relevant_images: int           # query-relevant images per request
    sinks_per_image: int
    planted: int                   # tiny-case planted tokens
    page_size: int                 # 0 = contiguous cache
    rho_sigma: float

    @property
    def tokens_per_request(self) -> int:
        return self.images_per_request * self.tokens_per_image


WORKLOADS = {
    "tiny": Workload("tiny", 1, 4, 2, 64, 1, 256, 1, 16, 16, 16, "f32", 0, (0.10,), 0, 0, 8, 0, 0.5),
    "single": Workload("single", 28, 28, 4, 128, 1, 1024, 1, 32, 32, 32, "bf16", 1, (0.10,), 0, 0, 0, 0, 0.7),
    "multi": Workload("multi", 28, 28, 4, 128, 8, 1024, 1, 64, 64, 64, "bf16", 2, (0.10,), 2, 0, 0, 0, 0.7),
    "longdoc": Workload("longdoc", 36, 32, 8, 128, 32, 1296, 1, 48, 48, 48, "bf16", 3,
                        (0.05, 0.10, 0.20), 3, 4, 0, 0, 0.7),
    "batched": Workload("batched", 28, 28, 4, 128, 4, 2048, 16, None, 32, 128, "bf16", 4,
                        (0.05, 0.10, 0.20), 1, 0, 0, 16, 0.7),
}


def workload(name: str, **overrides) -> Workload:
    """A named workload, optionally with fields replaced (smaller test variants)."""
    return dataclasses.replace(WORKLOADS[name], **overrides)


def _torch_dtype(name: str) -> torch.dtype:
    return torch.float32 if name == "f32" else torch.bfloat16


def _unit(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True)


def make_inputs(w: Workload, device="cpu", seed: Optional[int] = None) -> dict:
    """Draw one batch of the workload on ``device`` with a seeded generator.

    Returns contiguous tensors in the library's layouts:
      q [L][Hq][sum n_q][d], k / v [L][Hkv][N_tot][d] (dtype of the workload)
    and int32 offset arrays tok_off [R+1], img_off [K_tot+1] (global token
    offsets), req_img_off [R+1], q_off [R+1], plus the per-request ratios r.
    """
    seed = w.seed if seed is None else seed
    dev = torch.device(device)
    gen = torch.Generator(device=dev).manual_seed(seed)
    cpu_gen = torch.Generator().manual_seed(seed + 7919)
    L, Hq, Hkv, d = w.num_layers, w.num_q_heads, w.num_kv_heads, w.head_dim
    G = Hq // Hkv
    R = w.num_requests
    n_tok = w.tokens_per_request

    if w.n_q is not None:
        nq = [w.n_q] * R
    else:
        nq = torch.randint(w.n_q_lo, w.n_q_hi + 1, (R,), generator=cpu_gen).tolist()
    ratios = [float(w.ratios[int(i)]) for i in
              torch.randint(0, len(w.ratios), (R,), generator=cpu_gen).tolist()] \
        if R > 1 else [float(w.ratios[0])] * R
    tok_off = [i * n_tok for i in range(R + 1)]
    q_off = [0]
    for n in nq:
        q_off.append(q_off[-1] + n)
    img_off = [i * w.tokens_per_image for i in range(R * w.images_per_request + 1)]
    req_img_off = [i * w.images_per_request for i in range(R + 1)]
    n_tot, nq_tot = tok_off[-1], q_off[-1]

    dt = _torch_dtype(w.dtype)
    f32 = torch.float32
    q = torch.empty((L, Hq, nq_tot, d), dtype=dt, device=dev)
    k = torch.empty((L, Hkv, n_tot, d), dtype=dt, device=dev)
    v = torch.empty((L, Hkv, n_tot, d), dtype=dt, device=dev)

    # Per-request choices of planted / aligned tokens and relevant images.
    plans = []
    for r in range(R):
        perm_img = torch.randperm(w.images_per_request, generator=cpu_gen)
        relevant = sorted(perm_img[: w.relevant_images].tolist())
        n_al = int(round(0.05 * n_tok)) if w.planted == 0 else 0
        aligned = torch.randperm(n_tok, generator=cpu_gen)[:n_al].sort().values
        planted = torch.randperm(n_tok, generator=cpu_gen)[: w.planted].sort().values
        plans.append((relevant, aligned, planted))

    for l in range(L):
        for r in range(R):
            t0, t1 = tok_off[r], tok_off[r + 1]
            q0, q1 = q_off[r], q_off[r + 1]
            relevant, aligned, planted = plans[r]
            ql = torch.randn((Hq, q1 - q0, d), generator=gen, device=dev, dtype=f32)
            kl = torch.randn((Hkv, n_tok, d), generator=gen, device=dev, dtype=f32)
            if w.name == "tiny" or w.planted:
                u = _unit(ql.view(Hkv, G * (q1 - q0), d).mean(dim=1))            # [Hkv, d]
            else:
                u = _unit(torch.randn((Hkv, d), generator=gen, device=dev, dtype=f32))
                ql = ql + 0.5 * math.sqrt(d) * u.repeat_interleave(G, dim=0)[:, None, :]
                if aligned.numel():
                    a_idx = aligned.to(dev)
                    wv = torch.randn((Hkv, a_idx.numel(), d), generator=gen, device=dev, dtype=f32)
                    wv = _unit(wv - (wv * u[:, None, :]).sum(-1, keepdim=True) * u[:, None, :])
                    kn = kl[:, a_idx, :].norm(dim=-1, keepdim=True)
                    kl[:, a_idx, :] = kn * (0.6 * u[:, None, :] + 0.8 * wv)
                for j in relevant:
                    s0 = j * w.tokens_per_image
                    kl[:, s0:s0 + w.tokens_per_image, :] += 0.25 * math.sqrt(d) * u[:, None, :]
                if w.sinks_per_image:
                    for j in range(w.images_per_request):
                        s0 = j * w.tokens_per_image
                        ns = w.sinks_per_image
                        kl[:, s0:s0 + ns, :] = 1.5 * math.sqrt(d) * u[:, None, :] + torch.randn(
                            (Hkv, ns, d), generator=gen, device=dev, dtype=f32)
            if planted.numel():
                p_idx = planted.to(dev)
                kl[:, p_idx, :] = 3.0 * math.sqrt(d) * u[:, None, :] + 0.1 * torch.randn(
                    (Hkv, p_idx.numel(), d), generator=gen, device=dev, dtype=f32)
            # Values: direction uniform on the concatenated Hkv*d sphere, log-normal radius.
            z = _unit(torch.randn((n_tok, Hkv * d), generator=gen, device=dev, dtype=f32))
            rho = math.sqrt(Hkv * d) * torch.exp(
                w.rho_sigma * torch.randn((n_tok,), generator=gen, device=dev, dtype=f32))
            if planted.numel():
                rho[planted.to(dev)] *= 0.05
            if w.sinks_per_image:
                for j in range(w.images_per_request):
                    s0 = j * w.tokens_per_image
                    rho[s0:s0 + w.sinks_per_image] *= 0.02
            vl = (rho[:, None] * z).view(n_tok, Hkv, d).transpose(0, 1)
            q[l, :, q0:q1, :] = ql.to(dt)
            k[l, :, t0:t1, :] = kl.to(dt)
            v[l, :, t0:t1, :] = vl.to(dt)

    i32 = lambda xs: torch.tensor(xs, dtype=torch.int32)
    return {
        "workload": w, "q": q, "k": k, "v": v,
        "tok_off": i32(tok_off), "img_off": i32(img_off), "req_img_off": i32(req_img_off),
        "q_off": i32(q_off), "ratios": ratios, "n_q": nq,
    }


def make_fresh_rows(w: Workload, n_sel_total: int, device="cpu", seed: Optional[int] = None) -> dict:
    """Fresh queries / keys / values of the recomputed rows, N(0, 1).

    q_rows [L][n_sel][Hq][d], k_rows / v_rows [L][n_sel][Hkv][d]; n_sel is the
    total number of selected rows over all requests.
    """
    seed = (w.seed if seed is None else seed) + 104729
    dev = torch.device(device)
    gen = torch.Generator(device=dev).manual_seed(seed)
    dt = _torch_dtype(w.dtype)
    L, Hq, Hkv, d = w.num_layers, w.num_q_heads, w.num_kv_heads, w.head_dim
    shape_q, shape_kv = (L, n_sel_total, Hq, d), (L, n_sel_total, Hkv, d)
    return {
        "q_rows": torch.randn(shape_q, generator=gen, device=dev, dtype=torch.float32).to(dt),
        "k_rows": torch.randn(shape_kv, generator=gen, device=dev, dtype=torch.float32).to(dt),
        "v_rows": torch.randn(shape_kv, generator=gen, device=dev, dtype=torch.float32).to(dt),
    }


def make_extra_lse(inputs: dict, seed: int = 7) -> torch.Tensor:
    """Outside-key log-sum-exps for the full-context softmax, fp32 [L, Hq, Q_tot].

    A stand-in for what a prefill over the text and query-span keys would
    return per scoring row: the request's own visual scale log(N_r) plus a
    N(0, 4) spread, and one row in ten with no outside keys (-inf). Seeded.
    """
    L, Hq, q_tot, _ = inputs["q"].shape
    tok = inputs["tok_off"].tolist()
    q_off = inputs["q_off"].tolist()
    gen = torch.Generator(device="cpu").manual_seed(seed)
    e = torch.randn((L, Hq, q_tot), generator=gen, dtype=torch.float32) * 2.0
    for r in range(len(tok) - 1):
        e[:, :, q_off[r]:q_off[r + 1]] += float(math.log(max(tok[r + 1] - tok[r], 2)))
    e[torch.rand((L, Hq, q_tot), generator=gen) < 0.1] = -float("inf")
    return e.to(inputs["q"].device)


def to_paged(k: torch.Tensor, tok_off: Sequence[int], page_size: int, seed: int) -> tuple:
    """Re-lay a contiguous cache [L][Hkv][N_tot][d] into a shuffled page pool.

    Returns (pool [L][P][Hkv][page_size][d], page_table int32 [R][max_pages]).
    Request r's logical page p holds its tokens [p*page_size, (p+1)*page_size);
    physical pages follow a seeded permutation. Token counts must be multiples
    of page_size.
    """
    L, Hkv, n_tot, d = k.shape
    tok_off = [int(x) for x in tok_off]
    R = len(tok_off) - 1
    pages = [(tok_off[r + 1] - tok_off[r]) // page_size for r in range(R)]
    if any((tok_off[r + 1] - tok_off[r]) % page_size for r in range(R)):
        raise ValueError("token counts must be multiples of the page size")
    P = sum(pages)
    perm = torch.randperm(P, generator=torch.Generator().manual_seed(seed + 31337))
    max_pages = max(pages) if pages else 0
    table = torch.full((R, max_pages), -1, dtype=torch.int32)
    # logical (request, page) -> physical page
    flat = 0
    logical = torch.empty(P, dtype=torch.long)
    for r in range(R):
        for p in range(pages[r]):
            table[r, p] = int(perm[flat])
            logical[int(perm[flat])] = flat
            flat += 1
    # contiguous page blocks: [L][Hkv][P][page][d] in logical order
    blocks = k.view(L, Hkv, P, page_size, d)
    pool = blocks[:, :, logical.to(k.device), :, :].permute(0, 2, 1, 3, 4).contiguous()
    return pool, table


def request_view(inputs: dict, r: int) -> dict:
    """Host float64 numpy views of request r's tensors, for the CPU oracle."""
    tok_off = inputs["tok_off"].tolist()
    q_off = inputs["q_off"].tolist()
    img_off = inputs["img_off"].tolist()
    rio = inputs["req_img_off"].tolist()
    t0, t1 = tok_off[r], tok_off[r + 1]
    q0, q1 = q_off[r], q_off[r + 1]
    spans = [x - t0 for x in img_off[rio[r]: rio[r + 1] + 1]]
    return {
        "q": inputs["q"][:, :, q0:q1, :].double().cpu().numpy(),
        "k": inputs["k"][:, :, t0:t1, :].double().cpu().numpy(),
        "v": inputs["v"][:, :, t0:t1, :].double().cpu().numpy(),
        "img_off": spans,
    }
