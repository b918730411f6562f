"""The plain-C oracle (oracle/dmc_ref.c) against the hand-derived worked example,
vanilla attention (torch SDPA) and the numpy oracle, on the CPU."""
import json
import os

import numpy as np
import pytest
import torch

from oracle import cref
from oracle import dmc_ref as R

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example_alpha_11010.json")


def _head(rng, T, S, d, G, p_append):
    n = T + S
    k = rng.standard_normal((n, d)).astype(np.float32)
    v = rng.standard_normal((n, d)).astype(np.float32)
    q = rng.standard_normal((n, G, d)).astype(np.float32)
    sign = np.where(rng.random(n) < p_append, -1.0, 1.0)
    k[:, 0] = (sign * (np.abs(rng.standard_normal(n)) + 0.1)).astype(np.float32)
    return {"k_prompt": k[:T], "v_prompt": v[:T], "q0_prompt": q[:T, :, 0],
            "k_dec": k[T:], "v_dec": v[T:], "q_dec": q[T:]}


def test_c_oracle_worked_example():
    fx = json.load(open(GOLDEN))
    k, v, q = (np.array(fx[n], dtype=np.float64) for n in ("k", "v", "q"))
    # the golden's q values are irrational: check in fp64 through float32 inputs
    # only where exact (k, v are small integers and halves), so feed the
    # prompt path (omega only needs q[0]) and compare slots.
    h = {"k_prompt": k, "v_prompt": v, "q0_prompt": q[:, :1], "k_dec": np.zeros((0, 3)),
         "v_dec": np.zeros((0, 3)), "q_dec": np.zeros((0, 1, 3))}
    r = cref.run_heads([h])[0]
    assert r["prompt_len"] == 3
    tol = 1e-6  # q[0] = +-ln 3 rounded to float32 moves omega by ~1e-8
    assert np.allclose(r["prompt_K"], fx["expected_final_K"], atol=tol)
    assert np.allclose(r["prompt_V"], fx["expected_final_V"], atol=tol)
    assert np.allclose(r["prompt_z"], fx["expected_final_z"], atol=tol)


def test_c_oracle_all_append_is_vanilla_attention():
    rng = np.random.default_rng(3)
    n, d, G = 17, 16, 2
    h = _head(rng, 0, n, d, G, 1.0)
    r = cref.run_heads([h])[0]
    k = torch.tensor(h["k_dec"], dtype=torch.float64).clone()
    v = torch.tensor(h["v_dec"], dtype=torch.float64)
    q = torch.tensor(h["q_dec"], dtype=torch.float64).clone()
    k[:, 0] = 0
    q[:, :, 0] = 0
    ref = torch.nn.functional.scaled_dot_product_attention(
        q.permute(1, 0, 2), k.expand(G, n, d), v.expand(G, n, d), is_causal=True).permute(1, 0, 2)
    assert np.allclose(r["out"], ref.numpy(), atol=1e-12)
    assert list(r["lens"]) == list(range(1, n + 1))


@pytest.mark.parametrize("G", [1, 4])
def test_c_oracle_matches_numpy_oracle(G):
    rng = np.random.default_rng(10 + G)
    heads = [_head(rng, int(rng.integers(0, 60)), int(rng.integers(1, 20)), 32, G, p)
             for p in (0.1, 0.3, 0.5, 0.9, 1.0, 0.0)]
    rc = cref.run_heads(heads, threads=3)
    for h, c in zip(heads, rc):
        r = R.run_head(h["k_prompt"], h["v_prompt"], h["q0_prompt"], h["k_dec"], h["v_dec"],
                       h["q_dec"])
        assert c["prompt_len"] == r["prompt_len"]
        assert np.array_equal(c["lens"], r["lens"])
        assert np.allclose(c["prompt_K"], r["prompt_K"], atol=1e-12)
        assert np.allclose(c["prompt_V"], r["prompt_V"], atol=1e-12)
        assert np.allclose(c["prompt_z"], r["prompt_z"], atol=1e-12)
        assert np.allclose(c["out"], r["out"], atol=1e-12)
        K, V, z = r["cache"].arrays()
        assert np.allclose(c["K"], K, atol=1e-12) and np.allclose(c["z"], z, atol=1e-12)


@pytest.mark.parametrize("window", [1, 4, 12])
def test_c_oracle_window_grouping_matches_numpy(window):
    """The C oracle's window grouping against the numpy oracle (prompt then
    decode with outputs), grouped queries."""
    rng = np.random.default_rng(90 + window)
    d, G, T, S_ = 8, 2, 60, 25
    kp, vp = rng.normal(size=(T, d)), rng.normal(size=(T, d))
    kp[:, 0] = np.where(rng.random(T) < 0.2, -1.0, 1.0) * (np.abs(kp[:, 0]) + 0.1)
    q0p = rng.normal(size=(T, G))
    kd, vd = rng.normal(size=(S_, d)), rng.normal(size=(S_, d))
    kd[:, 0] = np.where(rng.random(S_) < 0.2, -1.0, 1.0) * (np.abs(kd[:, 0]) + 0.1)
    qd = rng.normal(size=(S_, G, d))
    f = lambda a: a.astype(np.float32).astype(np.float64)
    kp, vp, q0p, kd, vd, qd = map(f, (kp, vp, q0p, kd, vd, qd))
    ref = R.run_head(kp, vp, q0p, kd, vd, qd, window=window)
    got = cref.run_heads([{"k_prompt": kp, "v_prompt": vp, "q0_prompt": q0p,
                           "k_dec": kd, "v_dec": vd, "q_dec": qd}], window=window)[0]
    assert got["prompt_len"] == ref["prompt_len"] and np.allclose(got["prompt_K"], ref["prompt_K"])
    K, V, z = ref["cache"].arrays()
    assert np.allclose(got["K"], K) and np.allclose(got["V"], V) and np.allclose(got["z"], z)
    assert np.allclose(got["out"], ref["out"], atol=1e-10)
