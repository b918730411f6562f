"""The seeded input generator follows its stated recipe (CPU): decision signs
at the per-head append probability, |k[0]| away from the tie after the cast,
reproducible per-sequence streams, DMC-HardC's shared decisions."""
import numpy as np
import pytest
import torch

from paper_2403_09636_gb300 import synthetic as S


def test_derive_seed_is_deterministic_and_spreads():
    assert S.derive_seed(1, 2, 3) == S.derive_seed(1, 2, 3)
    seeds = {S.derive_seed(0, 1, l, b) for l in range(32) for b in range(32)}
    assert len(seeds) == 32 * 32
    assert all(0 <= x < 2 ** 63 for x in seeds)


@pytest.mark.parametrize("name", ["llama2_7b_4x", "llama2_7b_mixed", "long_ragged", "llama2_70b_gqa_2x"])
def test_append_probability_is_one_over_cr(name):
    wl = S.WORKLOADS[name]
    p = S.append_prob(wl)
    assert p.shape == (wl.num_layers, wl.num_kv_heads)
    kind = wl.cr[0]
    if kind == "fixed":
        assert np.allclose(p, 1.0 / wl.cr[1])
    elif kind == "choice":
        assert set(np.round(1.0 / p, 9).ravel().tolist()) <= set(float(c) for c in wl.cr[1])
    else:
        assert (1.0 / p >= wl.cr[1] - 1e-9).all() and (1.0 / p <= wl.cr[2] + 1e-9).all()


def test_prompt_shapes_lengths_and_decision_rate():
    wl = S.shrink(S.WORKLOADS["llama2_7b_4x"], batch=4, num_layers=1)
    pr = S.gen_prompt(wl, 0, "cpu")
    T = int(pr["lens"].sum())
    assert pr["k"].shape == (T, wl.num_kv_heads, wl.head_dim) and pr["k"].dtype == torch.bfloat16
    assert pr["q0"].shape == (T, wl.num_q_heads)
    assert pr["cu_seqlens"].tolist() == [0] + np.cumsum(pr["lens"]).tolist()
    assert (pr["lens"] == 2048).all()
    k0 = pr["k"][:, :, 0].float()
    # no decision at the tie: |k[0]| >= 0.1 * scale before the cast, >= 0.05 after it
    assert (k0.abs() >= 0.049).all()
    # appends (k[0] < 0) at rate 1 / CR = 0.25 per head: 8192 tokens, 5 sigma ~ 0.024
    rate = (k0 < 0).float().mean(0)
    assert torch.all((rate - 0.25).abs() < 0.03), rate


def test_sequence_streams_are_independent_of_the_subset():
    wl = S.shrink(S.WORKLOADS["llama2_7b_mixed"], batch=3, num_layers=2, prompt=(50, 90))
    full = S.gen_prompt(wl, 1, "cpu")
    part = S.gen_prompt(wl, 1, "cpu", seqs=[2])
    a = int(full["cu_seqlens"][2])
    assert torch.equal(full["k"][a:], part["k"])
    assert torch.equal(full["q0"][a:], part["q0"])
    again = S.gen_prompt(wl, 1, "cpu")
    assert torch.equal(full["v"], again["v"])
    dec = S.gen_decode(wl, 1, 5, "cpu")
    assert dec["q"].shape == (wl.batch, wl.num_q_heads, wl.head_dim)
    assert torch.equal(dec["k"], S.gen_decode(wl, 1, 5, "cpu")["k"])


def test_hardc_shares_decisions_and_importance_across_heads():
    wl = S.shrink(S.WORKLOADS["llama2_7b_4x_hardc"], batch=2, num_layers=1, prompt=(64, 64))
    pr = S.gen_prompt(wl, 0, "cpu")
    k0 = pr["k"][:, :, 0]
    assert torch.equal(k0, k0[:, :1].expand_as(k0))            # one decision value per token
    assert torch.equal(pr["q0"], pr["q0"][:, :1].expand_as(pr["q0"]))  # one omega per token
    dec = S.gen_decode(wl, 0, 0, "cpu")
    assert torch.equal(dec["k"][:, :, 0], dec["k"][:, :1, 0].expand_as(dec["k"][:, :, 0]))
    assert torch.equal(dec["q"][:, :, 0], dec["q"][:, :1, 0].expand_as(dec["q"][:, :, 0]))
