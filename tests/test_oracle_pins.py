"""Pins of the fp64 oracle against facts the paper and mathematics fix.

Each pin compares the oracle with something other than itself: a value printed
in the paper, a hand-derived worked example, a library routine in a special
case (torch SDPA, avg_pool1d, numpy means), or a counting identity. The
planted-mistake tests at the end show that a plausible slip in the oracle makes
at least one pin fail.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import dmc_ref as R

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example_alpha_11010.json")


def _rng(seed):
    return np.random.default_rng(seed)


def _tokens(rng, n, d, G=1, k0=None, q0=None):
    k = rng.standard_normal((n, d))
    v = rng.standard_normal((n, d))
    q = rng.standard_normal((n, G, d))
    if k0 is not None:
        k[:, 0] = k0
    if q0 is not None:
        q[:, :, 0] = q0
    return k, v, q


def _away_from_zero(rng, n, p_append):
    mag = np.abs(rng.standard_normal(n)) + 0.1
    sign = np.where(rng.random(n) < p_append, -1.0, 1.0)
    return sign * mag


# ---------------------------------------------------------------- pin checks
# Each returns True when the oracle satisfies the pin; the planted-mistake test
# runs all of them against a broken oracle.

def check_worked_example():
    fx = json.load(open(GOLDEN))
    k, v, q = (np.array(fx[n], dtype=np.float64) for n in ("k", "v", "q"))
    tol = fx["tolerance"]
    cache = R.HeadCache(3)
    ok = True
    for t in range(6):
        R.update(cache, k[t], v[t], int(R.decision(k[t, 0])), float(R.importance(q[t, :1])))
        ok &= len(cache) == fx["expected_lengths"][t]
        ok &= np.allclose(cache.z, fx["expected_z_after_each_token"][t], atol=tol, rtol=0)
        o = R.attend(cache, q[t])
        ok &= np.allclose(o, fx["expected_out"][t], atol=tol, rtol=0)
    K, V, z = cache.arrays()
    ok &= np.allclose(K, fx["expected_final_K"], atol=tol, rtol=0)
    ok &= np.allclose(V, fx["expected_final_V"], atol=tol, rtol=0)
    ok &= np.allclose(z, fx["expected_final_z"], atol=tol, rtol=0)
    ok &= list(R.decision(k[1:, 0])) == fx["expected_alpha_1_to_5"]
    return bool(ok)


def _sdpa_reference(k, v, q):
    """Vanilla causal attention via torch SDPA, q[0] and k[0] removed."""
    kt = torch.tensor(k, dtype=torch.float64).clone()
    vt = torch.tensor(v, dtype=torch.float64)
    qt = torch.tensor(q, dtype=torch.float64).clone()
    kt[:, 0] = 0
    qt[:, :, 0] = 0
    n, G, d = qt.shape
    out = torch.nn.functional.scaled_dot_product_attention(
        qt.permute(1, 0, 2), kt.expand(G, n, d), vt.expand(G, n, d), is_causal=True)
    return out.permute(1, 0, 2).numpy()


def check_all_append_is_vanilla(seed=1, n=11, d=8, G=2):
    rng = _rng(seed)
    k, v, q = _tokens(rng, n, d, G, k0=-(np.abs(rng.standard_normal(n)) + 0.1))
    r = R.run_head(np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, G)), k, v, q)
    ok = np.allclose(r["out"], _sdpa_reference(k, v, q), atol=1e-12, rtol=0)
    ok &= list(r["lens"]) == list(range(1, n + 1))
    return bool(ok)


def check_running_mean(seed=2, n=13, d=6):
    rng = _rng(seed)
    c = 0.3
    k, v, q = _tokens(rng, n, d, 1, k0=np.abs(rng.standard_normal(n)) + 0.1, q0=c)
    r = R.run_head(k, v, np.full((n, 1), c), np.zeros((0, d)), np.zeros((0, d)),
                   np.zeros((0, 1, d)))
    kk = k.copy()
    kk[:, 0] = 0
    w = 1.0 / (1.0 + math.exp(-c))
    ok = r["prompt_len"] == 1
    ok &= np.allclose(r["prompt_K"][0], kk.mean(axis=0), atol=1e-12, rtol=0)
    ok &= np.allclose(r["prompt_V"][0], v.mean(axis=0), atol=1e-12, rtol=0)
    ok &= abs(r["prompt_z"][0] - n * w) < 1e-12
    return bool(ok)


def check_avg_pool(seed=3, cr=4, blocks=6, d=5):
    """Fixed Memory Pooling ablation (DMC ablations appendix): append every CR
    tokens with constant omega gives average pooling with window CR."""
    rng = _rng(seed)
    n = cr * blocks
    k0 = np.where(np.arange(n) % cr == 0, -1.0, 1.0) * (np.abs(rng.standard_normal(n)) + 0.1)
    k, v, _ = _tokens(rng, n, d, 1, k0=k0)
    r = R.run_head(k, v, np.full((n, 1), -0.7), np.zeros((0, d)), np.zeros((0, d)),
                   np.zeros((0, 1, d)))
    kk = torch.tensor(k).clone()
    kk[:, 0] = 0
    pk = torch.nn.functional.avg_pool1d(kk.T[None], cr, cr)[0].T.numpy()
    pv = torch.nn.functional.avg_pool1d(torch.tensor(v).T[None], cr, cr)[0].T.numpy()
    ok = r["prompt_len"] == blocks
    ok &= np.allclose(r["prompt_K"], pk, atol=1e-12, rtol=0)
    ok &= np.allclose(r["prompt_V"], pv, atol=1e-12, rtol=0)
    return bool(ok)


def check_slot_count(seed=4, trials=20):
    rng = _rng(seed)
    ok = True
    for _ in range(trials):
        n = int(rng.integers(1, 60))
        k0 = _away_from_zero(rng, n, rng.random())
        k, v, q = _tokens(rng, n, 4, 1, k0=k0)
        r = R.run_head(k, v, q[:, :, 0], np.zeros((0, 4)), np.zeros((0, 4)), np.zeros((0, 1, 4)))
        ok &= r["prompt_len"] == 1 + int(np.count_nonzero(k0[1:] < 0))
    return bool(ok)


PINS = [check_worked_example, check_all_append_is_vanilla, check_running_mean,
        check_avg_pool, check_slot_count]


# ---------------------------------------------------------------- the pins

def test_sigmoid_c5_printed_value():
    # Training hyperparameters: the offset c = 5 "results in alpha_t = 0.0067".
    assert round(float(R.sigmoid(-5.0)), 4) == 0.0067
    assert abs(float(R.sigmoid(0.0)) - 0.5) == 0.0


def test_decision_is_sign_of_k0():
    rng = _rng(0)
    x = rng.standard_normal(10000) * 3
    x = x[np.abs(x) > 1e-9]
    assert np.array_equal(R.decision(x), (x >= 0).astype(np.int64))
    assert R.decision(0.0) == 1 and R.decision(-0.0) == 1  # tie rounds up
    assert R.decision(np.nan) == 0
    assert R.decision(0.05) == 1 and R.decision(-0.05) == 0


def test_worked_example_golden():
    assert check_worked_example()


def test_worked_example_closed_form_and_mask():
    fx = json.load(open(GOLDEN))
    k, v, q = (np.array(fx[n]) for n in ("k", "v", "q"))
    K, V, z = R.segment_slots(k, v, q[:, :1])
    assert np.allclose(K, fx["expected_final_K"], atol=1e-12)
    assert np.allclose(V, fx["expected_final_V"], atol=1e-12)
    assert np.allclose(z, fx["expected_final_z"], atol=1e-12)
    out = R.masked_attention(k, v, q[:, None, :])
    assert np.allclose(out[:, 0], fx["expected_out"], atol=1e-12)


def test_all_append_is_vanilla_attention():
    assert check_all_append_is_vanilla()
    assert check_all_append_is_vanilla(seed=7, n=30, d=16, G=1)


def test_all_append_with_prompt_is_vanilla_attention():
    rng = _rng(5)
    T, S, d, G = 9, 6, 8, 3
    k, v, q = _tokens(rng, T + S, d, G, k0=-(np.abs(rng.standard_normal(T + S)) + 0.1))
    r = R.run_head(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    ref = _sdpa_reference(k, v, q)[T:]
    assert np.allclose(r["out"], ref, atol=1e-12, rtol=0)


def test_running_mean_constant_omega():
    assert check_running_mean()


def test_fixed_memory_pooling_is_avg_pool():
    assert check_avg_pool()
    assert check_avg_pool(seed=9, cr=8, blocks=3, d=7)


def test_uniform_weighting_gives_plain_segment_means():
    # Importance-score ablation: constant omega -> unweighted mean per segment.
    rng = _rng(6)
    n, d = 40, 5
    k0 = _away_from_zero(rng, n, 0.3)
    k, v, _ = _tokens(rng, n, d, 1, k0=k0)
    r = R.run_head(k, v, np.full((n, 1), 1.3), np.zeros((0, d)), np.zeros((0, d)),
                   np.zeros((0, 1, d)))
    starts = [0] + [t for t in range(1, n) if k0[t] < 0]
    ends = starts[1:] + [n]
    kk = k.copy()
    kk[:, 0] = 0
    for j, (a, b) in enumerate(zip(starts, ends)):
        assert np.allclose(r["prompt_K"][j], kk[a:b].mean(axis=0), atol=1e-12)
        assert np.allclose(r["prompt_V"][j], v[a:b].mean(axis=0), atol=1e-12)


def test_slot_count_is_one_plus_zero_alphas():
    assert check_slot_count()


def test_decode_lengths_match_run():
    rng = _rng(8)
    n, d = 50, 4
    k0 = _away_from_zero(rng, n, 0.4)
    k, v, q = _tokens(rng, n, d, 1, k0=k0)
    r = R.run_head(k[:20], v[:20], q[:20, :, 0], k[20:], v[20:], q[20:])
    lens = R.decode_lengths(k0)
    assert lens[19] == r["prompt_len"]
    assert np.array_equal(lens[20:], r["lens"])


def test_z_is_sum_of_omega_per_slot():
    rng = _rng(10)
    n, d = 64, 4
    k0 = _away_from_zero(rng, n, 0.25)
    k, v, q = _tokens(rng, n, d, 1, k0=k0)
    r = R.run_head(k, v, q[:, :, 0], np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, 1, d)))
    w = 1.0 / (1.0 + np.exp(-q[:, 0, 0]))
    starts = [0] + [t for t in range(1, n) if k0[t] < 0]
    ends = starts[1:] + [n]
    expect = [w[a:b].sum() for a, b in zip(starts, ends)]
    assert np.allclose(r["prompt_z"], expect, atol=1e-12)


@pytest.mark.parametrize("seed", range(5))
def test_sequential_equals_closed_form(seed):
    rng = _rng(100 + seed)
    n, d, G = 70, 12, 2
    k, v, q = _tokens(rng, n, d, G, k0=_away_from_zero(rng, n, 0.3))
    r = R.run_head(k, v, q[:, :, 0], np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, G, d)))
    K, V, z = R.segment_slots(k, v, q[:, :, 0])
    assert np.allclose(r["prompt_K"], K, atol=1e-12)
    assert np.allclose(r["prompt_V"], V, atol=1e-12)
    assert np.allclose(r["prompt_z"], z, atol=1e-12)


@pytest.mark.parametrize("seed", range(5))
def test_sequential_equals_training_mask(seed):
    # Sec. 3.2: with binary alpha the additive mask reproduces inference exactly.
    rng = _rng(200 + seed)
    n, d, G = 25, 8, 3
    k, v, q = _tokens(rng, n, d, G, k0=_away_from_zero(rng, n, 0.4))
    r = R.run_head(np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, G)), k, v, q)
    assert np.allclose(r["out"], R.masked_attention(k, v, q), atol=1e-12)


@pytest.mark.parametrize("seed", [3, 4])
def test_prompt_attention_equals_training_mask(seed):
    """Prompt outputs token by token (inference) = the masked attention over all
    unrolled states (training formulation), for a group of 2 queries."""
    rng = np.random.default_rng(seed)
    n, d = 23, 6
    k, v = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    q = rng.normal(size=(n, 2, d))
    assert np.allclose(R.prompt_attention(k, v, q), R.masked_attention(k, v, q), atol=1e-12)


def test_prompt_attention_all_accumulate_is_running_mean():
    """k[0] >= 0 everywhere: one segment, every token sees only the running
    omega-weighted mean of the values so far."""
    rng = np.random.default_rng(5)
    n, d = 17, 5
    k, v = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    k[:, 0] = np.abs(k[:, 0]) + 0.1
    q = rng.normal(size=(n, 1, d))
    w = 1.0 / (1.0 + np.exp(-q[:, 0, 0]))
    want = np.cumsum(w[:, None] * v, axis=0) / np.cumsum(w)[:, None]
    assert np.allclose(R.prompt_attention(k, v, q)[:, 0], want, atol=1e-12)


@pytest.mark.parametrize("window", [1, 2, 5, 12])
def test_window_grouping_sequential_equals_training_mask(window):
    """Window grouping (Sec. 3.3): token-by-token updates over the last w
    tokens of a segment give the same outputs as the training formulation,
    where each token's state is the recurrence re-run over its last w tokens."""
    rng = np.random.default_rng(11 + window)
    n, d = 40, 6
    k, v = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    k[:, 0] = np.where(rng.random(n) < 0.2, -1.0, 1.0) * (np.abs(k[:, 0]) + 0.1)  # long segments
    q = rng.normal(size=(n, 2, d))
    got = R.prompt_attention(k, v, q, window=window)
    assert np.allclose(got, R.masked_attention(k, v, q, window=window), atol=1e-12)


@pytest.mark.parametrize("window", [1, 3, 7])
def test_window_grouping_slots_are_means_of_the_last_w_tokens(window):
    rng = np.random.default_rng(21 + window)
    n, d = 50, 5
    k, v = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    k[:, 0] = np.where(rng.random(n) < 0.15, -1.0, 1.0) * (np.abs(k[:, 0]) + 0.1)
    q0 = rng.normal(size=(n, 1))
    r = R.run_head(k, v, q0, np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, 1, d)), window=window)
    K, V, z = R.segment_slots(k, v, q0, window=window)
    assert np.allclose(r["prompt_K"], K) and np.allclose(r["prompt_V"], V) and np.allclose(r["prompt_z"], z)
    # brute force for every slot: the last min(len, w) tokens of its segment
    seg = R.segment_ids(k[:, 0])
    om = R.importance(q0)
    kk = k.copy()
    kk[:, 0] = 0.0
    for j in range(int(seg[-1]) + 1):
        idx = np.nonzero(seg == j)[0][-window:]
        assert np.allclose(K[j], (om[idx, None] * kk[idx]).sum(0) / om[idx].sum())
        assert np.isclose(z[j], om[idx].sum())


def test_window_grouping_wide_window_is_exact_dmc():
    rng = np.random.default_rng(31)
    n, d = 30, 4
    k, v, q = rng.normal(size=(n, d)), rng.normal(size=(n, d)), rng.normal(size=(n, 1, d))
    assert np.allclose(R.prompt_attention(k, v, q, window=n), R.prompt_attention(k, v, q), atol=1e-12)


def test_window_one_keeps_only_the_last_token():
    """w = 1: each slot is its segment's last token, z its omega."""
    rng = np.random.default_rng(41)
    n, d = 20, 4
    k, v = rng.normal(size=(n, d)), rng.normal(size=(n, d))
    q0 = rng.normal(size=(n, 1))
    K, V, z = R.segment_slots(k, v, q0, window=1)
    seg = R.segment_ids(k[:, 0])
    last = [int(np.nonzero(seg == j)[0][-1]) for j in range(int(seg[-1]) + 1)]
    assert np.allclose(V, v[last]) and np.allclose(z, R.importance(q0)[last])


def test_gqa_equal_group_q0_reduces_to_mha_omega():
    rng = _rng(11)
    n, d, G = 20, 6, 4
    k, v, q = _tokens(rng, n, d, G, k0=_away_from_zero(rng, n, 0.5))
    q[:, :, 0] = q[:, :1, 0]
    r = R.run_head(k, v, q[:, :, 0], np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, G, d)))
    r1 = R.run_head(k, v, q[:, :1, 0], np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, 1, d)))
    assert np.allclose(r["prompt_K"], r1["prompt_K"], atol=1e-15)
    assert np.allclose(r["prompt_z"], r1["prompt_z"], atol=1e-15)
    assert float(R.importance([0.2, -0.4, 1.0, 0.0])) == pytest.approx(1 / (1 + math.exp(-0.2)))


def test_prompt_then_decode_equals_token_stream():
    rng = _rng(12)
    n, d, G, T = 40, 8, 2, 25
    k, v, q = _tokens(rng, n, d, G, k0=_away_from_zero(rng, n, 0.3))
    r = R.run_head(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    full = R.run_head(np.zeros((0, d)), np.zeros((0, d)), np.zeros((0, G)), k, v, q)
    assert np.allclose(r["out"], full["out"][T:], atol=1e-12)


# ---------------------------------------------------------------- planted mistakes

def _bad_decision_flipped(k0):
    return (R.sigmoid(k0) < 0.5).astype(np.int64)


def _bad_importance_uniform(q0):
    return R.sigmoid(np.zeros_like(R.omega_logit(q0)))


def _make_bad_update(kind):
    good = R.update

    def bad(cache, k_t, v_t, alpha_t, omega_t):
        if kind == "keep_k0":
            k = np.array(k_t, dtype=np.float64)
            if alpha_t == 1 and len(cache):
                zp = cache.z[-1]
                zt = zp + omega_t
                cache.K[-1] = (cache.K[-1] * zp + k * omega_t) / zt
                cache.V[-1] = (cache.V[-1] * zp + np.asarray(v_t) * omega_t) / zt
                cache.z[-1] = zt
            else:
                cache.K.append(k)
                cache.V.append(np.array(v_t, dtype=np.float64))
                cache.z.append(float(omega_t))
            return
        if kind == "forget_z":
            if alpha_t == 1 and len(cache):
                cache.z[-1] = 0.0 * cache.z[-1]
            return good(cache, k_t, v_t, alpha_t, omega_t)
        if kind == "drop_first":
            if alpha_t == 1 and len(cache) == 0:
                return
            return good(cache, k_t, v_t, alpha_t, omega_t)
        if kind == "z_not_updated":
            zp = cache.z[-1] if (alpha_t == 1 and len(cache)) else None
            good(cache, k_t, v_t, alpha_t, omega_t)
            if zp is not None:
                cache.z[-1] = zp
            return
        raise ValueError(kind)
    return bad


def _make_bad_attend(kind):
    def bad(cache, q_t):
        q = np.array(q_t, dtype=np.float64)
        K, V, _ = cache.arrays()
        if kind == "keep_q0_and_k0":
            K = K.copy()
        else:
            q[0] = 0.0
        d = cache.d
        scale = {"scale_d_minus_1": 1 / math.sqrt(d - 1), "no_scale": 1.0}.get(kind, 1 / math.sqrt(d))
        s = (K @ q) * scale
        if kind == "drop_last_slot" and len(s) > 1:
            s[-1] = -np.inf
        p = np.exp(s - s.max())
        p /= p.sum()
        return p @ (K if kind == "keys_as_values" else V)
    return bad


def _bad_run_head_attend_before_update(k_prompt, v_prompt, q0_prompt, k_dec, v_dec, q_dec, cache=None):
    d = np.asarray(k_dec).shape[1]
    cache = R.HeadCache(d)
    for t in range(len(k_prompt)):
        R.update(cache, k_prompt[t], v_prompt[t], int(R.decision(k_prompt[t][0])),
                 float(R.importance(q0_prompt[t])))
    S, G = np.asarray(q_dec).shape[:2]
    out = np.zeros((S, G, d))
    lens = np.zeros(S, dtype=np.int64)
    for s in range(S):
        for g in range(G):
            out[s, g] = R.attend(cache, q_dec[s][g]) if len(cache) else 0.0
        R.update(cache, k_dec[s], v_dec[s], int(R.decision(k_dec[s][0])),
                 float(R.importance(np.asarray(q_dec[s])[:, 0])))
        lens[s] = len(cache)
    K, V, z = cache.arrays()
    return {"prompt_K": K, "prompt_V": V, "prompt_z": z, "prompt_len": len(cache),
            "out": out, "lens": lens, "cache": cache}


MUTATIONS = {
    "decision_flipped": ("decision", _bad_decision_flipped),
    "omega_uniform": ("importance", _bad_importance_uniform),
    "k0_not_cleared": ("update", _make_bad_update("keep_k0")),
    "z_prev_dropped": ("update", _make_bad_update("forget_z")),
    "first_token_dropped": ("update", _make_bad_update("drop_first")),
    "z_not_accumulated": ("update", _make_bad_update("z_not_updated")),
    "scale_sqrt_d_minus_1": ("attend", _make_bad_attend("scale_d_minus_1")),
    "no_scale": ("attend", _make_bad_attend("no_scale")),
    "keys_as_values": ("attend", _make_bad_attend("keys_as_values")),
    "current_slot_excluded": ("attend", _make_bad_attend("drop_last_slot")),
    "attend_before_update": ("run_head", _bad_run_head_attend_before_update),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, monkeypatch):
    attr, bad = MUTATIONS[name]
    monkeypatch.setattr(R, attr, bad)
    results = {}
    for pin in PINS:
        try:
            results[pin.__name__] = pin()
        except Exception:  # a crash also counts as the pin catching it
            results[pin.__name__] = False
    assert not all(results.values()), f"no pin caught the planted mistake {name}"


def test_pins_pass_on_the_real_oracle():
    assert all(pin() for pin in PINS)
