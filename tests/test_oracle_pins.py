"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every check compares the oracle with something other than itself: a closed
form, an invariant, a library routine (scipy / torch), brute force on tiny
inputs, or constants printed in the paper (tests/golden/paper_constants.json).
A plausible slip in the oracle (a dropped text term in a normaliser, tau
applied to the importance score, a wrong GQA head index, a reversed tie
rule, a floor instead of a ceiling) fails at least one of them.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import expit, softmax

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_case(seed, H=4, Hkv=2, D=8, n_v=12, text=5, vis_start=0, scale_q=1.0):
    rng = np.random.default_rng(seed)
    T = n_v + text
    q = scale_q * rng.standard_normal((H, D))
    k = rng.standard_normal((Hkv, T, D))
    v = rng.standard_normal((Hkv, T, D))
    return q, k, v, vis_start, n_v, text


# ---------------------------------------------------------------- softmax / mass

def test_softmax_matches_scipy_and_sums_to_one():
    rng = np.random.default_rng(0)
    z = 4 * rng.standard_normal((3, 50))
    for tau in (1.0, 0.4, 0.1):
        a = O.softmax_tau(z, tau)
        np.testing.assert_allclose(a.sum(axis=1), 1.0, rtol=0, atol=1e-12)
        np.testing.assert_allclose(a, softmax(z / tau, axis=1), rtol=1e-12, atol=1e-15)


def test_mass_in_unit_interval_and_headmax_dominates_mean():
    for seed in range(10):
        q, k, v, vs, nv, tl = _rand_case(seed, scale_q=3.0)
        r = O.decode_step(q, k, v, vs, nv, tl, tau=0.1)
        assert np.all(r["mass"] >= 0) and np.all(r["mass"] <= 1 + 1e-12)
        m_mean, m_max, m_mean1, _ = r["mass_stats"]
        assert m_max >= m_mean - 1e-15
        assert 0 <= m_mean1 <= 1 + 1e-12


def test_tau_one_mass_is_library_softmax_visual_sum():
    """tau = 1: Eq. 5 on the plain attention (torch.softmax over all tokens)."""
    q, k, v, vs, nv, tl = _rand_case(3, H=6, Hkv=3, D=16, n_v=20, text=9, vis_start=4)
    r = O.decode_step(q, k, v, vs, nv, tl, tau=1.0)
    G = 2
    kk = torch.tensor(k).repeat_interleave(G, dim=0)                 # [H, T, D]
    z = torch.einsum("hd,htd->ht", torch.tensor(q), kk) / math.sqrt(16)
    a = torch.softmax(z, dim=-1).numpy()
    expect = a[:, vs:vs + nv].sum(axis=1)
    np.testing.assert_allclose(r["mass"], expect, rtol=1e-12)
    np.testing.assert_allclose(r["mass_stats"][2], expect.mean(), rtol=1e-12)


def test_small_tau_mass_tends_to_argmax_indicator():
    """tau -> 0+: each head's mass tends to 1 if its largest logit is visual, else 0."""
    for seed in range(6):
        q, k, v, vs, nv, tl = _rand_case(seed, H=4, Hkv=4, n_v=10, text=10, vis_start=3)
        r = O.decode_step(q, k, v, vs, nv, tl, tau=1e-4)
        z = r["z"]
        top = z.argmax(axis=1)
        gap = np.sort(z, axis=1)[:, -1] - np.sort(z, axis=1)[:, -2]
        for h in range(4):
            if gap[h] > 0.05:                       # no near-tie at the top
                want = 1.0 if vs <= top[h] < vs + nv else 0.0
                assert abs(r["mass"][h] - want) < 1e-6


def test_two_token_closed_form():
    """One visual and one text token: mass_h = sigmoid((z_v - z_t) / tau)."""
    rng = np.random.default_rng(5)
    H, D = 3, 4
    q = rng.standard_normal((H, D))
    k = rng.standard_normal((1, 2, D))
    v = rng.standard_normal((1, 2, D))
    tau = 0.4
    r = O.decode_step(q, k, v, 0, 1, 1, tau=tau, r_lo_ppm=0, r_hi_ppm=1_000_000)
    zv = q @ k[0, 0] / 2.0
    zt = q @ k[0, 1] / 2.0
    np.testing.assert_allclose(r["mass"], expit((zv - zt) / tau), rtol=1e-12)
    np.testing.assert_allclose(r["s"], [expit(zv - zt).mean()], rtol=1e-12)
    # K_t = ceil(max mass * 1) = 1 whenever the mass is positive: keep both tokens.
    assert r["k_t"] == 1
    w = expit(zv - zt)
    np.testing.assert_allclose(r["out"], w[:, None] * v[0, 0] + (1 - w)[:, None] * v[0, 1], rtol=1e-12)
    # K_t = 0 leaves the text token alone: out is exactly its value row.
    r0 = O.decode_step(q, k, v, 0, 1, 1, mode=O.FIXED_K, fixed_k=0)
    np.testing.assert_array_equal(r0["out"], np.broadcast_to(v[0, 1], (H, D)))


# ------------------------------------------------------------------ closed form q = 0

@pytest.mark.parametrize("tau", [1.0, 0.4, 0.1])
def test_zero_query_closed_form(tau):
    """q = 0: every logit is 0, so mass_h = N_v / T for any tau, S_i = 1 / T,
    the kept set is the first K visual indices (ties to the lower index) and
    the output is the plain mean of the kept visual and the text value rows."""
    H, Hkv, D, n_v, text, vs = 6, 2, 8, 40, 13, 5
    rng = np.random.default_rng(1)
    k = rng.standard_normal((Hkv, n_v + text, D))
    v = rng.standard_normal((Hkv, n_v + text, D))
    q = np.zeros((H, D))
    r = O.decode_step(q, k, v, vs, n_v, text, tau=tau, r_lo_ppm=0, r_hi_ppm=1_000_000)
    T = n_v + text
    np.testing.assert_allclose(r["mass"], n_v / T, rtol=1e-13)
    np.testing.assert_allclose(r["s"], 1.0 / T, rtol=1e-13)
    k_t = math.ceil(np.float32(n_v / T) * np.float32(n_v))       # Eq. 7, no clamp
    assert r["k_t"] == k_t
    np.testing.assert_array_equal(r["kept"][0], np.arange(k_t))
    rows = np.r_[np.arange(vs), vs + np.arange(k_t), np.arange(vs + n_v, T)]
    for h in range(H):
        np.testing.assert_allclose(r["out"][h], v[h // 3][rows].mean(axis=0), rtol=1e-12, atol=1e-14)


# --------------------------------------------------------- full budget = dense SDPA

@pytest.mark.parametrize("mode,extra", [(O.DENSE, {}), (O.FIXED_RATIO, dict(ratio_ppm=1_000_000)),
                                        (O.FIXED_K, dict(fixed_k=10**6))])
def test_full_budget_is_dense_attention(mode, extra):
    """Keeping every visual token reproduces textbook attention (torch SDPA)."""
    q, k, v, vs, nv, tl = _rand_case(11, H=8, Hkv=2, D=16, n_v=30, text=7, vis_start=2, scale_q=2.0)
    r = O.decode_step(q, k, v, vs, nv, tl, mode=mode, **extra)
    assert r["k_t"] == nv
    G = 4
    qt = torch.tensor(q)[:, None, :]                                  # [H, 1, D]
    kt = torch.tensor(k).repeat_interleave(G, dim=0)
    vt = torch.tensor(v).repeat_interleave(G, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)[:, 0].numpy()
    np.testing.assert_allclose(r["out"], ref, rtol=1e-10, atol=1e-12)


def test_gqa_head_mapping_against_sdpa():
    """Distinct kv-heads: query head h must read kv-head h // G (not h % Hkv)."""
    q, k, v, vs, nv, tl = _rand_case(12, H=6, Hkv=3, D=8, n_v=9, text=4, scale_q=2.0)
    k[1] *= 3.0
    v[2] += 5.0
    r = O.decode_step(q, k, v, vs, nv, tl, mode=O.DENSE)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[:, None], torch.tensor(k).repeat_interleave(2, 0),
        torch.tensor(v).repeat_interleave(2, 0))[:, 0].numpy()
    np.testing.assert_allclose(r["out"], ref, rtol=1e-10, atol=1e-12)


def test_explicit_scale_equals_default():
    q, k, v, vs, nv, tl = _rand_case(13, D=16)
    a = O.decode_step(q, k, v, vs, nv, tl)
    b = O.decode_step(q, k, v, vs, nv, tl, scale=0.25)
    np.testing.assert_allclose(a["out"], b["out"], rtol=1e-14)
    c = O.decode_step(q, k, v, vs, nv, tl, scale=0.5)
    assert not np.allclose(a["mass"], c["mass"])


# --------------------------------------------------------------- top-k brute force

def _brute_topk(s32, k):
    """Exhaustive: the K-subset with the largest float32 score sum; among equal
    sums, the lexicographically smallest sorted index tuple (lower index wins)."""
    best = None
    for comb in itertools.combinations(range(len(s32)), k):
        tot = sum(float(s32[i]) for i in comb)
        key = (-tot, comb)
        if best is None or key < best:
            best = key
    return np.array(best[1] if best else (), dtype=np.int64)


@pytest.mark.parametrize("seed", range(8))
def test_topk_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 10))
    s = rng.random(n)
    if seed % 2:                        # plant exact ties
        s[rng.integers(0, n, size=n // 2)] = s[0]
    for k in range(n + 1):
        np.testing.assert_array_equal(O.select_topk(s, k), _brute_topk(s.astype(np.float32), k))


def test_topk_tie_rule_lower_index():
    s = np.array([0.5, 0.2, 0.5, 0.5, 0.1])
    np.testing.assert_array_equal(O.select_topk(s, 2), [0, 2])
    np.testing.assert_array_equal(O.select_topk(s, 4), [0, 1, 2, 3])


def test_importance_uses_plain_softmax_over_all_heads():
    """Eq. 2: S = mean over all H heads of the tau = 1 probabilities (scipy)."""
    q, k, v, vs, nv, tl = _rand_case(21, H=4, Hkv=2, D=8, n_v=11, text=6, vis_start=3, scale_q=2.0)
    r = O.decode_step(q, k, v, vs, nv, tl, tau=0.1)
    z = np.stack([k[h // 2] @ q[h] for h in range(4)]) / math.sqrt(8)
    a = softmax(z, axis=1)
    np.testing.assert_allclose(r["s"], a[:, vs:vs + nv].mean(axis=0), rtol=1e-12)


def test_per_kv_head_granularity_with_one_query_head_per_group():
    """G = 1: the per-kv-head score is that head's own attention row."""
    q, k, v, vs, nv, tl = _rand_case(22, H=3, Hkv=3, D=8, n_v=15, text=4, scale_q=2.0)
    r = O.decode_step(q, k, v, vs, nv, tl, granularity=1, mode=O.FIXED_K, fixed_k=4)
    z = np.stack([k[h] @ q[h] for h in range(3)]) / math.sqrt(8)
    a = softmax(z, axis=1)
    for h in range(3):
        want = np.sort(np.argsort(-a[h, :nv], kind="stable")[:4])
        np.testing.assert_array_equal(r["kept"][h], want)


# ------------------------------------------------------------------------ budget

def test_budget_table_by_hand():
    """Eq. 7 with the Sec. 5.2 clamp (1%..5%), worked by hand."""
    B = O.budget
    # N_v = 576: K_lo = ceil(5.76) = 6, K_hi = floor(28.8) = 28.
    assert O.budget_bounds(576, 10_000, 50_000) == (6, 28)
    assert B(0.0, 576) == 6                 # raw 0 -> K_lo
    assert B(1e-9, 576) == 6                # raw ceil(5.76e-7) = 1 -> K_lo
    assert B(0.03, 576) == 18               # raw ceil(17.28) = 18 inside the clamp
    assert B(0.05, 576) == 28               # raw ceil(28.8) = 29 -> K_hi
    assert B(1.0, 576) == 28
    # N_v = 1296: K_lo = ceil(12.96) = 13, K_hi = floor(64.8) = 64.
    assert B(0.02, 1296) == 26              # ceil(25.92)
    assert B(0.04, 1296) == 52              # ceil(51.84)
    # N_v = 2304: K_lo = ceil(23.04) = 24, K_hi = floor(115.2) = 115.
    assert O.budget_bounds(2304, 10_000, 50_000) == (24, 115)
    assert B(0.025, 2304) == 58             # ceil(57.6)
    # N_v = 1: K_lo = 1, K_hi = max(1, 0) = 1.
    assert B(0.0, 1) == 1 and B(1.0, 1) == 1
    # Exact integers are not bumped: 0.5 * 64 = 32 exactly in float32.
    assert B(0.5, 64, r_lo_ppm=0, r_hi_ppm=1_000_000) == 32
    # No clamp: pure Eq. 7 and its ceiling.
    assert B(0.0, 576, r_lo_ppm=0, r_hi_ppm=1_000_000) == 0
    assert B(0.0101, 100, r_lo_ppm=0, r_hi_ppm=1_000_000) == 2
    # 10% setting: N_v = 1296 -> [ceil(64.8), floor(129.6)] = [65, 129].
    assert O.budget_bounds(1296, 50_000, 100_000) == (65, 129)
    # Other modes.
    assert B(0.9, 576, mode=O.FIXED_RATIO, ratio_ppm=10_000) == 6     # ceil(5.76)
    assert B(0.9, 576, mode=O.FIXED_RATIO, ratio_ppm=500_000) == 288
    assert B(0.9, 10, mode=O.FIXED_RATIO, ratio_ppm=1) == 1          # at least one
    assert B(0.9, 576, mode=O.FIXED_K, fixed_k=256) == 256
    assert B(0.9, 100, mode=O.FIXED_K, fixed_k=256) == 100
    assert B(0.9, 576, mode=O.DENSE) == 576
    for mode in (O.ADAPTIVE, O.FIXED_RATIO, O.FIXED_K, O.DENSE):
        assert B(0.5, 0, mode=mode, ratio_ppm=10_000, fixed_k=5) == 0


def test_budget_presets_follow_the_paper():
    with open(os.path.join(GOLDEN, "paper_constants.json")) as f:
        c = json.load(f)
    for preset, key in ((W.ADAPTIVE_5PCT, "setting_5pct"), (W.ADAPTIVE_10PCT, "setting_10pct")):
        assert preset["tau"] == c[key]["tau"]
        assert preset["r_lo_ppm"] == round(c[key]["clamp_lo"] * O.PPM)
        assert preset["r_hi_ppm"] == round(c[key]["clamp_hi"] * O.PPM)
    ratios = {b["ratio_ppm"] for b in W.SWEEP_BUDGETS if b["mode"] == O.FIXED_RATIO}
    assert {round(x * O.PPM) for x in c["fix_ratio"]["ratios"]} <= ratios


# ------------------------------------------------------------------- invariances

def test_visual_span_position_does_not_matter():
    """Softmax is invariant to token order: moving the prompt prefix behind the
    visual span leaves masses, kept (visual-relative) indices and outputs."""
    q, k, v, _, nv, tl = _rand_case(31, H=4, Hkv=2, D=8, n_v=16, text=9, scale_q=2.0)
    vs = 4
    r1 = O.decode_step(q, k, v, vs, nv, tl, mode=O.FIXED_K, fixed_k=5)
    order = np.r_[np.arange(vs, vs + nv), np.arange(vs), np.arange(vs + nv, nv + tl)]
    r2 = O.decode_step(q, k[:, order], v[:, order], 0, nv, tl, mode=O.FIXED_K, fixed_k=5)
    np.testing.assert_allclose(r1["mass"], r2["mass"], rtol=1e-12)
    np.testing.assert_array_equal(r1["kept"][0], r2["kept"][0])
    np.testing.assert_allclose(r1["out"], r2["out"], rtol=1e-12)


def test_permutation_equivariance_of_visual_rows():
    q, k, v, vs, nv, tl = _rand_case(32, H=4, Hkv=2, D=8, n_v=20, text=6, scale_q=2.0)
    perm = np.random.default_rng(0).permutation(nv)
    k2, v2 = k.copy(), v.copy()
    k2[:, :nv] = k[:, perm]
    v2[:, :nv] = v[:, perm]
    r1 = O.decode_step(q, k, v, 0, nv, tl, mode=O.FIXED_K, fixed_k=6)
    r2 = O.decode_step(q, k2, v2, 0, nv, tl, mode=O.FIXED_K, fixed_k=6)
    np.testing.assert_array_equal(np.sort(perm[r2["kept"][0]]), r1["kept"][0])
    np.testing.assert_allclose(r1["out"], r2["out"], rtol=1e-12)


def test_pruned_tokens_are_excluded_not_zero_weighted():
    """Dropping visual tokens renormalises over kept + text: the output equals
    dense attention over the surviving rows only (torch SDPA on that subset)."""
    q, k, v, vs, nv, tl = _rand_case(33, H=4, Hkv=1, D=8, n_v=20, text=6, scale_q=2.0)
    r = O.decode_step(q, k, v, vs, nv, tl, mode=O.FIXED_K, fixed_k=3)
    rows = np.r_[r["kept"][0], np.arange(nv, nv + tl)]
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[:, None], torch.tensor(k[:, rows]).expand(4, -1, -1),
        torch.tensor(v[:, rows]).expand(4, -1, -1))[:, 0].numpy()
    np.testing.assert_allclose(r["out"], ref, rtol=1e-10, atol=1e-12)


def test_planted_keys_are_recovered():
    """Keys planted along the query focus (cosine 0.8) carry the largest
    scores: with K_t >= #planted every planted key is kept (tiny workload)."""
    r = W.TINY
    li = W.make_layer(r, 0)
    q = W.make_queries(r, 0, li, steps=4)
    planted = set(li.planted[0][0].tolist())
    for s in range(4):
        res = O.decode_step(q[s, 0], li.k[0], li.v[0], 0, 576, 128 + s,
                            mode=O.FIXED_K, fixed_k=len(planted))
        assert set(res["kept"][0].tolist()) == planted
        res = O.decode_step(q[s, 0], li.k[0], li.v[0], 0, 576, 128 + s, **r.budget)
        assert res["k_t"] == 28                    # peaked visual mass -> K_hi (5%)
        assert set(res["kept"][0].tolist()) <= planted


def test_empty_visual_span():
    q, k, v, _, _, tl = _rand_case(40, n_v=0, text=7)
    r = O.decode_step(q, k, v, 0, 0, tl)
    assert r["k_t"] == 0 and len(r["kept"][0]) == 0
    np.testing.assert_array_equal(r["mass"], 0.0)
    ref = O.decode_step(q, k, v, 0, 0, tl, mode=O.DENSE)
    np.testing.assert_allclose(r["out"], ref["out"])


# ------------------------------------------------- layers after the anchor layer

def test_anchor_attention_with_every_visual_token_is_dense():
    """A kept set holding the whole visual span gives textbook attention."""
    q, k, v, vs, nv, tl = _rand_case(41, H=8, Hkv=2, D=16, n_v=25, text=9, vis_start=3, scale_q=2.0)
    out = O.anchor_attention(q, k, v, vs, nv, tl, [np.arange(nv)])
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[:, None], torch.tensor(k).repeat_interleave(4, 0),
        torch.tensor(v).repeat_interleave(4, 0))[:, 0].numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)


def test_anchor_attention_is_sdpa_over_text_and_kept_rows():
    """Any kept set: SDPA over exactly the text rows and the kept visual rows
    (pruned rows excluded, text rows before and after the span included)."""
    q, k, v, vs, nv, tl = _rand_case(42, H=6, Hkv=3, D=8, n_v=17, text=8, vis_start=4, scale_q=2.0)
    kept = np.array([0, 5, 6, 16])
    out = O.anchor_attention(q, k, v, vs, nv, tl, [kept])
    rows = np.r_[np.arange(vs), vs + kept, np.arange(vs + nv, nv + tl)]
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[:, None], torch.tensor(k[:, rows]).repeat_interleave(2, 0),
        torch.tensor(v[:, rows]).repeat_interleave(2, 0))[:, 0].numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)


def test_anchor_attention_at_the_anchor_layer_reproduces_the_decode_step():
    """Fed the anchor layer's own kept set, the layer-after-anchor attention
    equals the decode step's output at that layer (both granularities)."""
    q, k, v, vs, nv, tl = _rand_case(43, H=8, Hkv=2, D=16, n_v=40, text=10, vis_start=1, scale_q=3.0)
    for gran in (0, 1):
        r = O.decode_step(q, k, v, vs, nv, tl, mode=O.FIXED_K, fixed_k=6, granularity=gran)
        out = O.anchor_attention(q, k, v, vs, nv, tl, r["kept"])
        np.testing.assert_allclose(out, r["out"], rtol=1e-12, atol=1e-12)


def test_anchor_attention_per_kv_head_sets():
    """One kept set per kv-head: each query head attends over its own kv-head's
    set (SDPA per group), not over another group's."""
    q, k, v, vs, nv, tl = _rand_case(44, H=4, Hkv=2, D=8, n_v=12, text=5, scale_q=2.0)
    sets = [np.array([1, 2]), np.array([7, 11])]
    out = O.anchor_attention(q, k, v, vs, nv, tl, sets)
    for g in range(2):
        rows = np.r_[sets[g], np.arange(nv, nv + tl)]
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.tensor(q[2 * g:2 * g + 2])[:, None], torch.tensor(k[g:g + 1, rows]).expand(2, -1, -1),
            torch.tensor(v[g:g + 1, rows]).expand(2, -1, -1))[:, 0].numpy()
        np.testing.assert_allclose(out[2 * g:2 * g + 2], ref, rtol=1e-10, atol=1e-12)


# ------------------------------------------------------- active visual tokens

def test_active_count_zero_query_closed_form():
    """q = 0: every score is 1/T, so every visual token is active exactly when
    1/T exceeds delta."""
    q, k, v, vs, nv, tl = _rand_case(51, n_v=20, text=6)
    r = O.decode_step(np.zeros_like(q), k, v, vs, nv, tl)
    T = nv + tl
    n, act = O.active_count(r["s"], 0.9 / T)
    assert n == nv and act.all()
    n, act = O.active_count(r["s"], 1.1 / T)
    assert n == 0 and not act.any()


def test_active_count_brute_force_and_limits():
    """Count by hand on a random case; delta below every score counts all
    tokens, delta at the largest score counts none; monotone in delta."""
    q, k, v, vs, nv, tl = _rand_case(52, n_v=30, text=5, scale_q=3.0)
    s = O.decode_step(q, k, v, vs, nv, tl)["s"]
    for delta in (1e-4, 1e-3, 1e-2, 5e-2):
        n, act = O.active_count(s, delta)
        assert n == sum(1 for x in s if np.float32(x) > np.float32(delta))
        assert list(np.flatnonzero(act)) == [i for i in range(nv) if np.float32(s[i]) > np.float32(delta)]
    assert O.active_count(s, 0.0)[0] == nv
    assert O.active_count(s, float(np.float32(s.max())))[0] == 0
    counts = [O.active_count(s, d)[0] for d in np.geomspace(1e-6, 1.0, 25)]
    assert all(a >= b for a, b in zip(counts, counts[1:]))


def test_active_count_per_kv_head():
    q, k, v, vs, nv, tl = _rand_case(53, H=4, Hkv=2, n_v=16, text=4, scale_q=2.0)
    s = O.decode_step(q, k, v, vs, nv, tl, granularity=1)["s"]
    n, act = O.active_count(s, 0.02)
    assert n.shape == (2,) and act.shape == (2, nv)
    for g in range(2):
        assert n[g] == (s[g].astype(np.float32) > np.float32(0.02)).sum()


# ------------------------------------------------------------- top-p budget

def test_top_p_uniform_scores_closed_form():
    """q = 0: all scores equal, so the top-p set is ceil(p * N_v) tokens (p * N_v
    not an integer here), the first ones by the tie rule."""
    q, k, v, vs, nv, tl = _rand_case(61, n_v=20, text=6)
    for ppm, want in ((130_000, 3), (10_000, 1), (999_000, 20), (560_000, 12)):
        r = O.decode_step(np.zeros_like(q), k, v, vs, nv, tl, mode=O.TOP_P, ratio_ppm=ppm)
        assert r["k_t"] == want
        assert list(r["kept"][0]) == list(range(want))


def test_top_p_brute_force_over_subsets():
    """K is the smallest size of ANY subset of visual tokens whose scores reach a
    share p of the total (the best subset of a size is its top scores)."""
    for seed in range(6):
        q, k, v, vs, nv, tl = _rand_case(70 + seed, n_v=9, text=3, scale_q=3.0)
        s = O.decode_step(q, k, v, vs, nv, tl)["s"].astype(np.float32).astype(np.float64)
        for ppm in (50_000, 200_000, 500_000, 900_000):
            target = ppm / 1e6 * s.sum()
            want = min(kk for kk in range(1, nv + 1)
                       if any(sum(s[list(c)]) >= target for c in itertools.combinations(range(nv), kk)))
            assert O.top_p_budget(s, ppm) == want


def test_top_p_limits_and_monotonicity():
    q, k, v, vs, nv, tl = _rand_case(62, n_v=40, text=5, scale_q=2.0)
    s = O.decode_step(q, k, v, vs, nv, tl)["s"]
    assert O.top_p_budget(s, 0) == 0 and O.top_p_budget(s, 1_000_000) == nv
    ks = [O.top_p_budget(s, ppm) for ppm in range(0, 1_000_001, 50_000)]
    assert all(a <= b for a, b in zip(ks, ks[1:]))
    dominant = np.r_[np.full(9, 0.02), 0.5]               # one token holds 0.5 / 0.68 = 74% of the scores
    assert O.top_p_budget(dominant, 100_000) == 1 and O.top_p_budget(dominant, 730_000) == 1
    assert O.top_p_budget(dominant, 750_000) == 2


# ------------------------------------------------ FastV prefill pruning (appendix)

def test_fastv_zero_query_keeps_the_first_half():
    """q = 0: every visual token gets the same attention, so the tie rule keeps
    the lowest indices; ratio 0.5 keeps ceil(N_v / 2), at least one."""
    q, k, v, vs, nv, tl = _rand_case(80, n_v=13, text=4, vis_start=2)
    assert list(O.fastv_survivors(np.zeros_like(q), k, vs, nv, tl)) == list(range(7))
    assert list(O.fastv_survivors(np.zeros_like(q), k, vs, 1, tl)) == [0]


def test_fastv_brute_force_and_planted_recall():
    """Against explicit per-head loops on tiny inputs, and planted keys aligned
    with the last prompt token's query are always among the survivors."""
    for seed in range(5):
        q, k, v, vs, nv, tl = _rand_case(81 + seed, H=4, Hkv=2, D=8, n_v=10, text=5, vis_start=3)
        H, D = q.shape
        G = H // k.shape[0]
        T = nv + tl
        s = np.zeros(nv)
        for h in range(H):
            z = [float(np.dot(q[h], k[h // G, j])) / math.sqrt(D) for j in range(T)]
            m = max(z)
            den = sum(math.exp(x - m) for x in z)
            for i in range(nv):
                s[i] += math.exp(z[vs + i] - m) / den / H
        order = sorted(range(nv), key=lambda i: (-float(np.float32(s[i])), i))
        assert list(O.fastv_survivors(q, k, vs, nv, tl)) == sorted(order[:5])
    q, k, v, vs, nv, tl = _rand_case(90, H=4, Hkv=2, D=16, n_v=40, text=6)
    for i in (3, 17, 31):
        for g in range(2):
            k[g, vs + i] = 4.0 * q[2 * g:2 * g + 2].mean(0) / np.linalg.norm(q[2 * g:2 * g + 2].mean(0)) * math.sqrt(16)
    assert {3, 17, 31} <= set(O.fastv_survivors(q, k, vs, nv, tl, ratio_ppm=100_000).tolist())


def test_compact_cache_rows():
    """Rows labelled with their own position map as the definition says; with
    every visual token kept the cache is unchanged."""
    Hkv, T, D = 2, 30, 4
    x = np.broadcast_to(np.arange(T, dtype=np.float64)[None, :, None], (Hkv, T, D)).copy()
    vs, nv, tl = 4, 15, 15
    kept = np.array([0, 2, 3, 9, 14])
    c = O.compact_cache(x, vs, nv, tl, kept)
    want = list(range(4)) + [4, 6, 7, 13, 18] + list(range(19, 30))
    assert c.shape == (Hkv, len(kept) + tl, D)
    assert c[0, :, 0].tolist() == want and c[1, :, 3].tolist() == want
    assert np.array_equal(O.compact_cache(x, vs, nv, tl, np.arange(nv)), x)


def test_compacted_decode_equals_attention_restricted_to_survivors():
    """Dense attention over the compacted cache is the attention of the full
    cache with the pruned visual tokens removed from the softmax set (the
    anchor-layer attention with the survivors as its kept set), and a
    VisionPulse step over the compacted cache keeps a subset of survivors."""
    q, k, v, vs, nv, tl = _rand_case(91, H=4, Hkv=2, D=8, n_v=16, text=6, vis_start=2)
    surv = O.fastv_survivors(q * 0.7, k, vs, nv, tl)
    kc, vc = O.compact_cache(k, vs, nv, tl, surv), O.compact_cache(v, vs, nv, tl, surv)
    dense = O.decode_step(q, kc, vc, vs, len(surv), tl, mode=O.DENSE)
    want = O.anchor_attention(q, k, v, vs, nv, tl, [surv])
    np.testing.assert_allclose(dense["out"], want, rtol=0, atol=1e-12)
    r = O.decode_step(q, kc, vc, vs, len(surv), tl, mode=O.FIXED_RATIO, ratio_ppm=250_000)
    assert set(surv[r["kept"][0]].tolist()) <= set(surv.tolist()) and len(r["kept"][0]) == 2
