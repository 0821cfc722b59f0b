"""Planted mistakes in the CPU oracle must each fail at least one pin.

Every mutant below replaces one oracle function with a plausible wrong
version (a dropped term, a wrong index or axis, a flipped tie rule); the test
re-runs the pins of test_oracle_pins against the mutant and requires that one
of them fails. The mistakes are planted in the oracle, on the CPU only.
"""

import math

import numpy as np
import pytest

from oracle import conduit_oracle as O
from tests import test_oracle_pins as P


def _softmax_wrong_axis(x):
    m = x.max(axis=0, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=0, keepdims=True)


def _logits_no_scale(q_h, k_g):
    return q_h @ k_g.T


def _head_mean_wrong_gqa(q_l, k_l, extra_lse_l=None):
    hq, n_q, _ = q_l.shape
    hkv = k_l.shape[0]
    total = np.zeros(k_l.shape[1])
    for h in range(hq):
        total += O.softmax_over_visual_keys(O.cached_key_logits(q_l[h], k_l[h % hkv])).sum(axis=0)
    return total / (n_q * hq)


def _head_mean_wrong_divisor(q_l, k_l, extra_lse_l=None):
    hq, n_q, _ = q_l.shape
    hkv = k_l.shape[0]
    total = np.zeros(k_l.shape[1])
    for h in range(hq):
        total += O.softmax_over_visual_keys(O.cached_key_logits(q_l[h], k_l[h // (hq // hkv)])).sum(axis=0)
    return total / (n_q * hkv)


def _outside_keys_dropped(x, extra_lse):
    return O.softmax_over_visual_keys(x)


def _outside_keys_twice(x, extra_lse):
    c = np.maximum(x.max(axis=1), extra_lse)[:, None]
    e = np.exp(x - c)
    return e / (e.sum(axis=1, keepdims=True) + 2 * np.exp(extra_lse[:, None] - c))


def _rms_without_root(q_l, k_l, extra_lse_l=None):
    hq, n_q, _ = q_l.shape
    alpha = O._attention_rows(q_l, k_l, extra_lse_l)
    return (alpha * alpha).sum(axis=(0, 1)) / (n_q * hq)


def _rms_over_queries_only(q_l, k_l, extra_lse_l=None):
    hq, n_q, _ = q_l.shape
    alpha = O._attention_rows(q_l, k_l, extra_lse_l)
    return np.sqrt((alpha * alpha).sum(axis=(0, 1)) / n_q)


def _quotas_floor_only(c, n, k):
    w = np.asarray(c, dtype=np.float64) * np.asarray(n, dtype=np.float64)
    return np.floor(k * w / w.sum()).astype(np.int64)


def _quotas_ties_high(c, n, k):
    w = np.asarray(c, dtype=np.float64) * np.asarray(n, dtype=np.float64)
    ideal = k * w / w.sum()
    base = np.floor(ideal).astype(np.int64)
    order = sorted(range(len(n)), key=lambda j: (-(ideal[j] - base[j]), -j))
    for j in order[:k - int(base.sum())]:
        base[j] += 1
    return np.minimum(base, np.asarray(n))


def _quotas_ignore_sizes(c, n, k):
    return _quotas_ties_high_free(np.asarray(c, dtype=np.float64), len(n), k)


def _quotas_ties_high_free(w, K, k):
    ideal = k * w / w.sum()
    base = np.floor(ideal).astype(np.int64)
    order = sorted(range(K), key=lambda j: (-(ideal[j] - base[j]), j))
    for j in order[:k - int(base.sum())]:
        base[j] += 1
    return base


_staleness_iso = O.staleness_iso  # the original, for the mutants that wrap it


def _staleness_no_dim_divisor(q, k, v, refreshed, z, kappa):
    return _staleness_iso(q, k, v, refreshed, z, kappa) * np.asarray(q).shape[-1]


def _staleness_keeps_refreshed(q, k, v, refreshed, z, kappa):
    return _staleness_iso(q, k, v, np.zeros_like(np.asarray(refreshed, dtype=float)), z, kappa)


def _value_norm_mean_of_heads(v_l):
    return np.sqrt((v_l * v_l).sum(axis=2)).mean(axis=0)


def _throughput_sum(a, vn):
    return (a * vn).sum(axis=0)


def _image_mean_no_layer_divisor(a, img_off):
    return np.array([a[:, img_off[j]:img_off[j + 1]].sum() / (img_off[j + 1] - img_off[j])
                     for j in range(len(img_off) - 1)])


def _coefficients_ignore_lambda(g, lam):
    if g.shape[0] == 1:
        return np.ones(1)
    return g / g.mean()


def _coefficients_inverted(g, lam):
    if g.shape[0] == 1:
        return np.ones(1)
    return (1 - lam) + lam * g.mean() / g


def _composite_shifted_image(s, c, img_off):
    out = np.empty_like(s)
    for j in range(len(img_off) - 1):
        out[img_off[j]:img_off[j + 1]] = s[img_off[j]:img_off[j + 1]] * c[(j + 1) % len(c)]
    return out


def _topk_highest_index_ties(s_hat, k):
    order = sorted(range(len(s_hat)), key=lambda t: (-float(s_hat[t]), -t))
    return np.array(sorted(order[:k]), dtype=np.int64)


def _topk_ascending(s_hat, k):
    order = sorted(range(len(s_hat)), key=lambda t: (float(s_hat[t]), t))
    return np.array(sorted(order[:k]), dtype=np.int64)


def _budget_round(r, n):
    if not 0.0 <= r <= 1.0:
        raise ValueError
    return int(round(r * n))


def _refresh_exclusive(q_rows, kp, vp, idx):
    out = np.zeros_like(np.asarray(q_rows, dtype=np.float64))
    L, n_sel, hq, d = out.shape
    G = hq // kp.shape[1]
    for l in range(L):
        for i, p in enumerate(idx):
            for h in range(hq):
                hi = max(int(p), 1)
                x = kp[l, h // G, :hi] @ q_rows[l, i, h] / math.sqrt(d)
                w = np.exp(x - x.max())
                out[l, i, h] = (w / w.sum()) @ vp[l, h // G, :hi]
    return out


def _scatter_wrong_axis(cache, idx, rows):
    out = np.array(cache, copy=True)
    for i, t in enumerate(idx):
        out[:, :, t, :] = rows[:, i, ::-1, :]
    return out


MUTANTS = {
    "softmax over queries": ("softmax_over_visual_keys", _softmax_wrong_axis),
    "no 1/sqrt(d) scale": ("cached_key_logits", _logits_no_scale),
    "GQA head h -> h % Hkv": ("head_query_mean_attention", _head_mean_wrong_gqa),
    "divide by Hkv": ("head_query_mean_attention", _head_mean_wrong_divisor),
    "mean of per-head norms": ("value_norms", _value_norm_mean_of_heads),
    "staleness without the 1/d variance": ("staleness_iso", _staleness_no_dim_divisor),
    "staleness counts refreshed tokens": ("staleness_iso", _staleness_keeps_refreshed),
    "quotas floored, leftover dropped": ("image_quotas", _quotas_floor_only),
    "quota remainder ties to the higher index": ("image_quotas", _quotas_ties_high),
    "quotas ignore image sizes": ("image_quotas", _quotas_ignore_sizes),
    "outside keys dropped": ("softmax_with_outside_keys", _outside_keys_dropped),
    "outside keys counted twice": ("softmax_with_outside_keys", _outside_keys_twice),
    "RMS without the root": ("head_query_rms_attention", _rms_without_root),
    "RMS divides by |Q| only": ("head_query_rms_attention", _rms_over_queries_only),
    "layer sum instead of mean": ("throughput_score", _throughput_sum),
    "g without 1/|L|": ("image_mean_attention", _image_mean_no_layer_divisor),
    "lambda ignored": ("image_coefficients", _coefficients_ignore_lambda),
    "inverted ratio": ("image_coefficients", _coefficients_inverted),
    "wrong image coefficient": ("composite_score", _composite_shifted_image),
    "ties to highest index": ("topk_select", _topk_highest_index_ties),
    "bottom-k": ("topk_select", _topk_ascending),
    "budget rounds": ("budget", _budget_round),
    "refresh excludes itself": ("refresh_attention", _refresh_exclusive),
    "scatter transposes heads": ("kv_scatter", _scatter_wrong_axis),
}

PINS = [getattr(P, n) for n in dir(P) if n.startswith("test_")]


def _run_pins():
    failed = []
    for pin in PINS:
        params = getattr(pin, "pytestmark", [])
        arg_sets = [{}]
        for mark in params:
            if mark.name == "parametrize":
                names = [s.strip() for s in mark.args[0].split(",")]
                arg_sets = [dict(zip(names, vals if isinstance(vals, tuple) else (vals,)))
                            for vals in mark.args[1]]
        for kwargs in arg_sets:
            try:
                pin(**kwargs)
            except (AssertionError, ValueError, IndexError):
                failed.append(pin.__name__)
                break
    return failed


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(O, attr, fn)
    assert _run_pins(), f"no pin catches the planted mistake: {name}"


def test_unmutated_oracle_passes_every_pin():
    assert _run_pins() == []
