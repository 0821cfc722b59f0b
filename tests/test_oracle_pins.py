"""Pins of the CPU oracle against facts the paper and the mathematics fix.

None of these tests re-types an oracle formula: each checks the oracle
against a hand-derived closed form, a brute-force enumeration, a library
routine (scipy / torch softmax and attention), or an invariant stated in the
paper (Sec. 3.5 single-image limit, App. B.1 Lemma 1, App. B.2 normalisation).
"""

import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import conduit_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example.json")


def _worked_inputs():
    ex = json.load(open(GOLDEN))
    inp = ex["inputs"]
    w = np.array(inp["weights_w"], dtype=np.float64)
    L, Hq, Hkv, nq, N = inp["num_layers"], inp["num_q_heads"], inp["num_kv_heads"], inp["n_q"], len(w)
    q = np.zeros((L, Hq, nq, 1))
    q[0, :, :, 0] = np.array(inp["queries"]["layer0"])
    q[1, :, :, 0] = np.array(inp["queries"]["layer1"])
    k = np.zeros((L, Hkv, N, 1))
    k[:, 0, :, 0] = np.log(w)
    v = np.zeros((L, Hkv, N, 1))
    v[0, 0, :, 0] = inp["values"]["layer0"]
    v[1, 0, :, 0] = inp["values"]["layer1"]
    return ex, q, k, v, inp["img_off"]


# ---------------------------------------------------------------- closed form
def test_worked_example_scores():
    ex, q, k, v, img_off = _worked_inputs()
    e = ex["expected"]
    sc = O.score_request(q, k, v, img_off)
    np.testing.assert_allclose(sc["a"], e["a"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(sc["vn"], e["vn"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(sc["s"], e["s"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(sc["A"], e["A"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(sc["g"], e["g"], rtol=0, atol=1e-14)
    c = O.image_coefficients(sc["g"], 1.0)
    np.testing.assert_allclose(c, e["c_lambda1"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(O.composite_score(sc["s"], c, img_off), e["s_hat_lambda1"], rtol=0, atol=1e-14)


@pytest.mark.parametrize("lam,key", [(1.0, "topk_lambda1"), (0.0, "topk_lambda0")])
def test_worked_example_selection(lam, key):
    ex, q, k, v, img_off = _worked_inputs()
    for kk, want in ex["expected"][key].items():
        out = O.refresh_mask(q, k, v, img_off, lam=lam, k_budget=int(kk))
        assert out["idx"].tolist() == want
        assert out["mask"].tolist() == [1 if t in want else 0 for t in range(4)]


# ------------------------------------------------------------------- budget
def test_budget_eq2():
    assert O.budget(0.0, 1000) == 0
    assert O.budget(1.0, 1000) == 1000
    assert O.budget(0.10, 256) == 25          # floor(25.6)
    assert O.budget(0.10, 1024) == 102
    assert O.budget(0.10, 8192) == 819
    assert O.budget(0.05, 41472) == 2073
    assert O.budget(0.20, 41472) == 8294
    assert O.budget(0.3, 10) == 3             # decimal ratio lands on the integer
    assert O.budget(0.7, 10) == 7
    with pytest.raises(ValueError):
        O.budget(-0.1, 10)
    with pytest.raises(ValueError):
        O.budget(1.5, 10)


# -------------------------------------------------- Lemma 1 brute force
def _brute_force_topk(s_hat, k):
    """argmin over |T| = k of sum_{t not in T} s_hat_t^2 (App. B.1, Lemma 1);
    among minimisers the lexicographically smallest index tuple."""
    n = len(s_hat)
    best, best_val = None, None
    for T in itertools.combinations(range(n), k):
        rest = [t for t in range(n) if t not in T]
        val = sum(s_hat[t] * s_hat[t] for t in rest)
        if best_val is None or val < best_val:
            best, best_val = T, val
    return list(best)


@pytest.mark.parametrize("seed", range(6))
def test_topk_is_lemma1_minimiser_with_ties(seed):
    rng = np.random.default_rng(seed)
    n = 10
    # small integers: exact squares and sums in fp64, many ties
    s_hat = rng.integers(0, 5, size=n).astype(np.float64)
    for k in range(n + 1):
        assert O.topk_select(s_hat, k).tolist() == _brute_force_topk(s_hat.tolist(), k)


@pytest.mark.parametrize("seed", range(4))
def test_topk_is_lemma1_minimiser_distinct(seed):
    rng = np.random.default_rng(100 + seed)
    n = 11
    s_hat = rng.random(n)
    for k in (0, 1, 3, 5, 10, 11):
        assert O.topk_select(s_hat, k).tolist() == _brute_force_topk(s_hat.tolist(), k)


def test_topk_matches_library_sort():
    rng = np.random.default_rng(7)
    s_hat = rng.random(500)
    k = 123
    want = np.sort(np.argsort(-s_hat, kind="stable")[:k])
    assert O.topk_select(s_hat, k).tolist() == want.tolist()
    t = torch.topk(torch.from_numpy(s_hat), k).indices.sort().values
    assert O.topk_select(s_hat, k).tolist() == t.tolist()


# ------------------------------------------------- library softmax / GQA map
def _rand_request(seed, L=2, Hq=6, Hkv=2, nq=5, N=37, d=8, spans=(0, 10, 25, 37)):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((L, Hq, nq, d))
    k = rng.standard_normal((L, Hkv, N, d)) * 1.5
    v = rng.standard_normal((L, Hkv, N, d)) * rng.lognormal(0, 0.5, size=(1, 1, N, 1))
    return q, k, v, list(spans)


def test_head_query_mean_matches_torch_softmax_with_gqa():
    q, k, v, _ = _rand_request(1)
    L, Hq, nq, d = q.shape
    Hkv = k.shape[1]
    for l in range(L):
        kk = torch.from_numpy(k[l]).repeat_interleave(Hq // Hkv, dim=0)      # head h -> kv h // G
        logits = torch.matmul(torch.from_numpy(q[l]), kk.transpose(-1, -2)) / math.sqrt(d)
        alpha = torch.softmax(logits, dim=-1)                                  # over visual keys
        want = alpha.mean(dim=(0, 1)).numpy()
        np.testing.assert_allclose(O.head_query_mean_attention(q[l], k[l]), want, rtol=1e-12, atol=1e-15)


def test_surrogate_special_case_eq5():
    """L = 1, H = 1, |Q| = 1: s_t = alpha_t ||V_t|| (Eq. 5), via scipy softmax and numpy norm."""
    scipy_special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(3)
    N, d = 50, 16
    q = rng.standard_normal((1, 1, 1, d))
    k = rng.standard_normal((1, 1, N, d)) * 2
    v = rng.standard_normal((1, 1, N, d))
    alpha = scipy_special.softmax(q[0, 0, 0] @ k[0, 0].T / math.sqrt(d))
    want = alpha * np.linalg.norm(v[0, 0], axis=1)
    sc = O.score_request(q, k, v, [0, N])
    np.testing.assert_allclose(sc["s"], want, rtol=1e-12, atol=0)


def test_value_norm_is_over_concatenated_heads():
    # heads carry 3 and 4 along one axis: the concatenated norm is 5
    v = np.zeros((2, 3, 4))
    v[0, :, 1] = 3.0
    v[1, :, 2] = -4.0
    np.testing.assert_array_equal(O.value_norms(v), [5.0, 5.0, 5.0])
    rng = np.random.default_rng(4)
    v = rng.standard_normal((4, 9, 8))
    want = np.linalg.norm(np.concatenate([v[g] for g in range(4)], axis=1), axis=1)
    np.testing.assert_allclose(O.value_norms(v), want, rtol=1e-14)


# ----------------------------------------------------- paper invariants
def test_softmax_identities():
    q, k, v, spans = _rand_request(5)
    sc = O.score_request(q, k, v, spans)
    np.testing.assert_allclose(sc["a"].sum(axis=1), 1.0, rtol=0, atol=1e-13)   # each a^(l) sums to 1
    np.testing.assert_allclose(sc["A"].sum(), q.shape[0], atol=1e-13)           # sum_t A_t = |L|
    n_j = np.diff(spans)
    np.testing.assert_allclose((n_j * sc["g"]).sum(), 1.0, atol=1e-13)          # sum_j n_j g_j = 1


def test_key_shift_invariance():
    q, k, v, spans = _rand_request(6)
    b = np.random.default_rng(60).standard_normal((q.shape[0], k.shape[1], 1, k.shape[3]))
    a1 = O.score_request(q, k, v, spans)
    a2 = O.score_request(q, k + b, v, spans)
    np.testing.assert_allclose(a2["a"], a1["a"], rtol=1e-10, atol=1e-15)
    np.testing.assert_allclose(a2["s"], a1["s"], rtol=1e-10, atol=1e-15)


def test_value_scale_equivariance():
    q, k, v, spans = _rand_request(7)
    r1 = O.refresh_mask(q, k, v, spans, k_budget=9)
    r2 = O.refresh_mask(q, k, 3.5 * v, spans, k_budget=9)
    np.testing.assert_allclose(r2["s"], 3.5 * r1["s"], rtol=1e-13)
    assert r2["idx"].tolist() == r1["idx"].tolist()


def test_zero_value_norm_gives_zero_score():
    q, k, v, spans = _rand_request(8)
    v[:, :, [3, 11, 30], :] = 0.0
    sc = O.score_request(q, k, v, spans)
    assert sc["s"][3] == 0.0 and sc["s"][11] == 0.0 and sc["s"][30] == 0.0
    assert (sc["s"][[0, 1, 2]] > 0).all()


def test_uniform_norm_reproduces_raw_attention_ranking():
    """Drop-||V|| ablation (Table 5): a uniform norm ranks by attention alone."""
    q, k, v, _ = _rand_request(9)
    N = k.shape[2]
    rng = np.random.default_rng(90)
    z = rng.standard_normal(v.shape)
    zc = np.transpose(z, (0, 2, 1, 3)).reshape(z.shape[0], N, -1)
    zc = zc / np.linalg.norm(zc, axis=-1, keepdims=True) * 2.0
    v_uni = np.transpose(zc.reshape(z.shape[0], N, z.shape[1], z.shape[3]), (0, 2, 1, 3))
    for kk in (1, 5, 20):
        sel = O.refresh_mask(q, k, v_uni, [0, N], k_budget=kk)["idx"]
        by_attention = O.topk_select(O.score_request(q, k, v_uni, [0, N])["A"], kk)
        assert sel.tolist() == by_attention.tolist()


def test_single_image_limit():
    """K = 1: c_1 = 1 for every lambda and selection is intra-image top-k of s (Sec. 3.5)."""
    q, k, v, _ = _rand_request(10)
    N = k.shape[2]
    for lam in (0.0, 0.25, 0.5, 1.0):
        assert O.image_coefficients(np.array([0.0123]), lam).tolist() == [1.0]
        out = O.refresh_mask(q, k, v, [0, N], lam=lam, k_budget=7)
        want = np.sort(np.argsort(-out["s"], kind="stable")[:7])
        assert out["idx"].tolist() == want.tolist()


def test_lambda_zero_is_plain_global_topk():
    q, k, v, spans = _rand_request(11)
    out = O.refresh_mask(q, k, v, spans, lam=0.0, k_budget=8)
    assert np.all(out["c"] == 1.0)
    want = np.sort(np.argsort(-out["s"], kind="stable")[:8])
    assert out["idx"].tolist() == want.tolist()


def test_mean_coefficient_is_one():
    rng = np.random.default_rng(12)
    for _ in range(20):
        g = rng.random(rng.integers(2, 40)) * 1e-3
        for lam in (0.0, 0.3, 1.0):
            assert abs(O.image_coefficients(g, lam).mean() - 1.0) < 1e-12


def test_relevant_image_is_amplified():
    """lambda = 1 raises tokens of an above-average image (Sec. 3.4)."""
    g = np.array([0.1, 0.3, 0.2])
    c = O.image_coefficients(g, 1.0)
    assert c[1] > 1.0 > c[0] and abs(c[2] - 1.0) < 1e-15


def test_budget_zero_and_full():
    q, k, v, spans = _rand_request(13)
    N = k.shape[2]
    out0 = O.refresh_mask(q, k, v, spans, r=0.0)
    assert out0["k"] == 0 and out0["idx"].size == 0 and out0["mask"].sum() == 0
    out1 = O.refresh_mask(q, k, v, spans, r=1.0)
    assert out1["idx"].tolist() == list(range(N)) and out1["mask"].sum() == N


def test_scored_layer_subset():
    q, k, v, spans = _rand_request(14, L=3)
    one = O.score_request(q, k, v, spans, layers=[1])
    alone = O.score_request(q[1:2], k[1:2], v[1:2], spans)
    np.testing.assert_allclose(one["s"], alone["s"], rtol=1e-15)
    np.testing.assert_allclose(one["g"], alone["g"], rtol=1e-15)


# ------------------------------------------------- value-norm side cache
def test_stored_norms_give_the_same_scores():
    """Sec. 4.3 / App. C.2: norms kept from cache construction leave the scores unchanged."""
    q, k, v, spans = _rand_request(16, L=3)
    stored = np.stack([np.linalg.norm(np.concatenate(list(v[l]), axis=1), axis=1) for l in range(3)])
    for layers in (None, [0, 2]):
        live = O.score_request(q, k, v, spans, layers=layers)
        kept = O.score_request(q, k, None, spans, layers=layers, vnorm=stored)
        for key in ("a", "vn", "s", "A", "g"):
            np.testing.assert_allclose(kept[key], live[key], rtol=1e-14, atol=0)


def test_stored_norms_are_read_per_scored_layer():
    """Norms constant per layer (c_l) give s = sum_l c_l a^(l) / |L| over the scored layers."""
    q, k, v, spans = _rand_request(17, L=4)
    N = k.shape[2]
    c = np.array([1.0, 10.0, 100.0, 1000.0])
    vnorm = np.repeat(c[:, None], N, axis=1)
    kept = O.score_request(q, k, None, spans, layers=[1, 3], vnorm=vnorm)
    a = [O.head_query_mean_attention(q[l], k[l]) for l in (1, 3)]
    np.testing.assert_allclose(kept["s"], (10.0 * a[0] + 1000.0 * a[1]) / 2, rtol=1e-13)
    # unit norms: s is the layer-mean attention A / |L|
    ones = O.score_request(q, k, None, spans, vnorm=np.ones((4, N)))
    np.testing.assert_allclose(ones["s"], ones["A"] / 4, rtol=1e-14)


# ------------------------------------------------ statistic variants
def _softmax_rows(x):
    """Library softmax of each row (scipy), for the pins below."""
    sp = pytest.importorskip("scipy.special")
    return sp.softmax(x, axis=-1)


def test_rms_statistic_brute_force_and_special_cases():
    """Eq. 4: abar_t = sqrt(mean over (q, h) of alpha^2), against scipy softmax;
    one query row and one head give abar = alpha exactly; abar >= a (power means)."""
    q, k, v, spans = _rand_request(18, L=2)
    L, hq, n_q, d = q.shape
    G = hq // k.shape[1]
    got = O.score_request(q, k, v, spans, statistic="rms")
    for l in range(L):
        alpha = np.stack([_softmax_rows(q[l, h] @ k[l, h // G].T / math.sqrt(d)) for h in range(hq)])
        want = np.sqrt((alpha ** 2).mean(axis=(0, 1)))
        np.testing.assert_allclose(got["stat"][l], want, rtol=1e-12)
    assert np.all(got["stat"] >= got["a"] * (1 - 1e-12))
    np.testing.assert_allclose(got["A"], O.score_request(q, k, v, spans)["A"], rtol=1e-15)
    one = O.score_request(q[:, :1, :1], k[:, :1], v, spans, statistic="rms")
    np.testing.assert_allclose(one["stat"], one["a"], rtol=1e-13)


def test_attention_alone_ablation():
    """Dropping the value norm (Sec. 4.4 factor ablation): s = A / |L| exactly."""
    q, k, v, spans = _rand_request(19, L=3)
    got = O.score_request(q, k, None, spans, use_value_norm=False)
    np.testing.assert_allclose(got["s"], got["A"] / 3, rtol=1e-14)


def test_full_context_softmax_matches_softmax_over_all_keys():
    """Outside keys entering through their log-sum-exp give the visual columns
    of a library softmax over visual + outside keys; without outside keys the
    visual-only softmax comes back."""
    sp = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(20)
    L, hq, hkv, n_q, N, n_text, d = 2, 4, 2, 3, 40, 25, 16
    q = rng.standard_normal((L, hq, n_q, d))
    k = rng.standard_normal((L, hkv, N, d)) * 1.5
    k_text = rng.standard_normal((L, hkv, n_text, d)) * 1.5
    v = rng.standard_normal((L, hkv, N, d))
    spans = [0, 15, N]
    G = hq // hkv
    extra = np.zeros((L, hq, n_q))
    want_a = np.zeros((L, N))
    for l in range(L):
        for h in range(hq):
            xt = q[l, h] @ k_text[l, h // G].T / math.sqrt(d)
            extra[l, h] = sp.logsumexp(xt, axis=1)
            x_all = np.concatenate([q[l, h] @ k[l, h // G].T / math.sqrt(d), xt], axis=1)
            want_a[l] += _softmax_rows(x_all)[:, :N].sum(axis=0)
    want_a /= n_q * hq
    got = O.score_request(q, k, v, spans, extra_lse=extra)
    np.testing.assert_allclose(got["a"], want_a, rtol=1e-12)
    assert np.all(got["a"].sum(axis=1) < 1.0)
    none = O.score_request(q, k, v, spans, extra_lse=np.full((L, hq, n_q), -np.inf))
    plain = O.score_request(q, k, v, spans)
    for key in ("a", "s", "A", "g"):
        np.testing.assert_allclose(none[key], plain[key], rtol=1e-14)


# ------------------------------------------- explicit per-image quotas
def test_quotas_textbook_largest_remainder():
    """Hamilton's rule on hand-checked cases: a remainder tie goes to the lower
    index; sizes 6, 6, 2 give 4, 4, 2 seats of 10 and 5, 5, 1 of 11 (the
    Alabama paradox, a known property of the largest-remainder rule)."""
    assert O.image_quotas(np.ones(3), [55, 30, 15], 10).tolist() == [6, 3, 1]
    assert O.image_quotas(np.ones(3), [6, 6, 2], 10).tolist() == [4, 4, 2]
    assert O.image_quotas(np.ones(3), [6, 6, 2], 11).tolist() == [5, 5, 1]
    # coefficients scale the sizes: c n = (20, 10, 10) of 8 -> 4, 2, 2
    assert O.image_quotas(np.array([2.0, 1.0, 0.5]), [10, 10, 20], 8).tolist() == [4, 2, 2]


def test_quotas_cap_and_degenerate_cases():
    # image 0 would take 8.3 of 50 but holds 2 tokens: capped, the rest re-shared
    assert O.image_quotas(np.array([10.0, 1.0]), [2, 100], 50).tolist() == [2, 48]
    assert O.image_quotas(np.array([3.0]), [17], 9).tolist() == [9]            # K = 1: k_1 = k
    assert O.image_quotas(np.zeros(3), [4, 8, 4], 8).tolist() == [2, 4, 2]     # all c = 0: sizes
    assert O.image_quotas(np.array([0.0, 1.0]), [5, 5], 3).tolist() == [0, 3]
    assert O.image_quotas(np.ones(2), [3, 4], 7).tolist() == [3, 4]            # k = sum n_j
    assert O.image_quotas(np.ones(2), [3, 4], 0).tolist() == [0, 0]


def test_quotas_minimise_deviation_brute_force():
    """Without caps, the largest-remainder quotas minimise sum |k_j - ideal_j|
    over every integer split of k (enumerated), and lie between floor and ceil."""
    rng = np.random.default_rng(21)
    for _ in range(200):
        K = int(rng.integers(1, 5))
        n = rng.integers(5, 12, size=K).tolist()
        c = rng.uniform(0.2, 2.0, size=K)
        k = int(rng.integers(0, min(n) + 1))  # small enough that no ideal exceeds n_j
        w = c * np.array(n, dtype=np.float64)
        ideal = k * w / w.sum()
        if np.any(ideal > np.array(n)):
            continue
        got = O.image_quotas(c, n, k)
        assert got.sum() == k and np.all(got >= np.floor(ideal)) and np.all(got <= np.ceil(ideal))
        best = min(sum(abs(x - q) for x, q in zip(split, ideal))
                   for split in itertools.product(*[range(k + 1)] * K) if sum(split) == k)
        assert abs(np.abs(got - ideal).sum() - best) < 1e-9


def test_quota_select_per_image_top():
    rng = np.random.default_rng(23)
    s = rng.uniform(size=40)
    s[[3, 7]] = s[5]                       # a three-way tie inside image 0
    spans = [0, 10, 25, 40]
    c = np.array([1.0, 2.0, 0.5])
    out = O.quota_select(s, c, spans, 12)
    q = out["quota"]
    assert q.tolist() == O.image_quotas(c, [10, 15, 15], 12).tolist() and q.sum() == 12
    for j in range(3):
        lo, hi = spans[j], spans[j + 1]
        mine = [t - lo for t in out["idx"] if lo <= t < hi]
        order = sorted(range(hi - lo), key=lambda t: (-s[lo + t], t))   # brute-force ranking
        assert sorted(mine) == sorted(order[:q[j]])
    one = O.quota_select(s, np.array([1.3]), [0, 40], 9)               # one image: the global top-k
    assert one["idx"].tolist() == O.topk_select(s, 9).tolist()


# ------------------------------------------- isotropic staleness (App. D)
def _stale_case(seed, L=2, hq=4, hkv=2, n_q=3, N=24, d=8, M=3):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((L, hq, n_q, d))
    k = rng.standard_normal((L, hkv, N, d))
    v = rng.standard_normal((L, hkv, N, d)) * rng.uniform(0.5, 2.0, size=(L, hkv, N, 1))
    z = rng.standard_normal((M, L, hkv, N, d))
    return q, k, v, z


def test_staleness_matches_its_expectation():
    """E[E_iso] = kappa^2 sum_{l,h,q} sum_{t not in T} alpha^2 ||V_t||^2 (the draws are
    independent, zero-mean, E||xi||^2 = kappa^2 ||V||^2): a large M lands within the
    Monte Carlo error of that closed form (scipy softmax for alpha)."""
    q, k, v, _ = _stale_case(30, M=1)
    L, hq, n_q, d = q.shape
    hkv, N = k.shape[1], k.shape[2]
    T = np.zeros(N)
    T[[1, 5, 9, 20]] = 1
    M = 4000
    z = np.random.default_rng(31).standard_normal((M, L, hkv, N, d))
    got = O.staleness_iso(q, k, v, T, z, 0.7)
    want = 0.0
    for l in range(L):
        for h in range(hq):
            g = h // (hq // hkv)
            alpha = _softmax_rows(q[l, h] @ k[l, g].T / math.sqrt(d))
            vn2 = (v[l, g] ** 2).sum(axis=1)
            want += 0.49 * ((alpha ** 2) * (vn2 * (1 - T))[None, :]).sum()
    assert abs(got - want) < 0.05 * want   # MC standard error ~ sqrt(2 / M) ~ 2 %


def test_staleness_special_cases():
    q, k, v, z = _stale_case(32)
    N = k.shape[2]
    assert O.staleness_iso(q, k, v, np.ones(N), z, 1.0) == 0.0          # everything refreshed
    e1 = O.staleness_iso(q, k, v, np.zeros(N), z, 1.0)
    np.testing.assert_allclose(O.staleness_iso(q, k, v, np.zeros(N), z, 3.0), 9.0 * e1, rtol=1e-13)
    # one key, one head, one row: alpha = 1, so E = kappa^2 ||V||^2 / d * mean_m ||z_m||^2
    q1, k1, v1 = q[:1, :1, :1], k[:1, :1, :1], v[:1, :1, :1]
    z1 = z[:, :1, :1, :1]
    d = q.shape[-1]
    want = 4.0 * (v1[0, 0, 0] ** 2).sum() / d * (z1[:, 0, 0, 0] ** 2).sum(axis=1).mean()
    np.testing.assert_allclose(O.staleness_iso(q1, k1, v1, np.zeros(1), z1, 2.0), want, rtol=1e-13)
    # refreshing more tokens never raises the error for the same draws when the
    # displacement directions are orthogonal across tokens (one-hot z)
    hkv, Nn, dd = k.shape[1], k.shape[2], k.shape[3]
    zo = np.zeros((1, q.shape[0], hkv, Nn, Nn))
    for t in range(Nn):
        zo[0, :, :, t, t] = 1.0
    qo = np.random.default_rng(33).standard_normal(q.shape[:3] + (Nn,))
    ko = np.random.default_rng(34).standard_normal(k.shape[:3] + (Nn,))
    vo = np.random.default_rng(35).standard_normal(k.shape[:3] + (Nn,))
    T1 = np.zeros(Nn); T1[[2, 3]] = 1
    T2 = T1.copy(); T2[[10, 11, 12]] = 1
    assert O.staleness_iso(qo, ko, vo, T2, zo, 1.0) <= O.staleness_iso(qo, ko, vo, T1, zo, 1.0)


# --------------------------------------------------------- refresh step
def test_gather_scatter_roundtrip():
    rng = np.random.default_rng(15)
    cache = rng.standard_normal((2, 3, 20, 4))
    idx = [1, 5, 19]
    rows = rng.standard_normal((2, 3, 3, 4))
    patched = O.kv_scatter(cache, idx, rows)
    np.testing.assert_array_equal(O.kv_gather(patched, idx), rows)
    keep = [t for t in range(20) if t not in idx]
    np.testing.assert_array_equal(patched[:, :, keep], cache[:, :, keep])
    np.testing.assert_array_equal(O.kv_gather(cache, idx)[:, 1, 2], cache[:, 2, 5])


def test_refresh_attention_full_budget_is_causal_sdpa():
    """k = N with no patch is ordinary causal self-attention: torch SDPA with GQA."""
    rng = np.random.default_rng(16)
    L, Hq, Hkv, N, d = 2, 4, 2, 13, 8
    k = rng.standard_normal((L, Hkv, N, d))
    v = rng.standard_normal((L, Hkv, N, d))
    q_rows = rng.standard_normal((L, N, Hq, d))
    out = O.refresh_attention(q_rows, k, v, list(range(N)))
    for l in range(L):
        qt = torch.from_numpy(q_rows[l]).transpose(0, 1)                      # [Hq, N, d]
        kt = torch.from_numpy(k[l]).repeat_interleave(Hq // Hkv, dim=0)
        vt = torch.from_numpy(v[l]).repeat_interleave(Hq // Hkv, dim=0)
        want = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
        np.testing.assert_allclose(out[l], want.transpose(0, 1).numpy(), rtol=1e-12, atol=1e-13)


def test_refresh_attention_sparse_rows_match_sdpa_rows():
    rng = np.random.default_rng(17)
    L, Hq, Hkv, N, d = 1, 4, 1, 30, 16
    k = rng.standard_normal((L, Hkv, N, d))
    v = rng.standard_normal((L, Hkv, N, d))
    idx = [2, 9, 10, 29]
    q_all = rng.standard_normal((L, N, Hq, d))
    out = O.refresh_attention(q_all[:, idx], k, v, idx)
    qt = torch.from_numpy(q_all[0]).transpose(0, 1)
    kt = torch.from_numpy(k[0]).repeat_interleave(Hq, dim=0)
    vt = torch.from_numpy(v[0]).repeat_interleave(Hq, dim=0)
    full = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True).transpose(0, 1).numpy()
    np.testing.assert_allclose(out[0], full[idx], rtol=1e-12, atol=1e-13)


def test_refresh_attention_first_position_returns_its_value():
    rng = np.random.default_rng(18)
    k = rng.standard_normal((1, 2, 6, 4))
    v = rng.standard_normal((1, 2, 6, 4))
    q = rng.standard_normal((1, 1, 4, 4)) * 10
    out = O.refresh_attention(q, k, v, [0])
    for h in range(4):
        np.testing.assert_array_equal(out[0, 0, h], v[0, h // 2, 0])
