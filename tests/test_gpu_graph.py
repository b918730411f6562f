"""Decode steps captured in a CUDA graph and replayed (GPU).

One decode step of every layer is captured once with static input and output
buffers; each replay after copying in a new step's q, k, v must give exactly
the outputs and slot counts of the same steps launched eagerly on a second
cache with the same history (the launches are deterministic), and the eager
outputs are checked against the oracle by the parity tests. Covers the MHA
kernel, the tensor-core kernel for grouped queries and the per-query path with
its pending-row buffer (fp32 groups).
"""
import pytest
import torch

from paper_2403_09636_gb300 import synthetic as S
from tests import dmc_harness as H

pytestmark = pytest.mark.gpu

CASES = [
    S.Workload("graph_mha_bf16", 3, 4, 8, 8, 128, "bf16", (150, 300), 12, ("choice", (1.0, 2.0, 4.0)), 0.5, seed=21),
    S.Workload("graph_gqa_bf16", 2, 3, 8, 2, 128, "bf16", (100, 400), 12, ("fixed", 2.0), 0.5, seed=22),
    S.Workload("graph_gqa_f32", 2, 2, 4, 2, 64, "f32", (60, 90), 12, ("fixed", 3.0), 1.0, seed=23),
]


@pytest.mark.parametrize("wl", CASES, ids=lambda w: w.name)
def test_graph_replay_matches_eager(cuda_dev, wl):
    p = S.append_prob(wl)
    eager, graphed = H.cache_for(wl, cuda_dev), H.cache_for(wl, cuda_dev)
    for layer in range(wl.num_layers):
        pr = S.gen_prompt(wl, layer, cuda_dev, p=p)
        for c in (eager, graphed):
            c.prefill(layer, pr["q0"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"])
    torch.cuda.synchronize()

    first = [S.gen_decode(wl, layer, 0, cuda_dev, p=p) for layer in range(wl.num_layers)]
    q_s = [x["q"].clone() for x in first]
    k_s = [x["k"].clone() for x in first]
    v_s = [x["v"].clone() for x in first]
    o_s = [torch.empty_like(x["q"]) for x in first]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for layer in range(wl.num_layers):
            graphed.decode(layer, q_s[layer], k_s[layer], v_s[layer], o_s[layer])

    for step in range(wl.decode_steps):
        xs = [S.gen_decode(wl, layer, step, cuda_dev, p=p) for layer in range(wl.num_layers)]
        ref = []
        for layer, x in enumerate(xs):
            out = torch.empty_like(x["q"])
            eager.decode(layer, x["q"], x["k"], x["v"], out)
            ref.append(out)
            q_s[layer].copy_(x["q"])
            k_s[layer].copy_(x["k"])
            v_s[layer].copy_(x["v"])
        g.replay()
        torch.cuda.synchronize()
        for layer in range(wl.num_layers):
            assert torch.equal(o_s[layer], ref[layer]), (step, layer)
    for layer in range(wl.num_layers):
        assert torch.equal(graphed.lengths(layer), eager.lengths(layer))
    assert graphed.status()[:2] == (0, 0)
    assert eager.status()[:2] == (0, 0)


@pytest.mark.parametrize("wl", CASES[:2], ids=lambda w: w.name)
def test_graph_prompt_and_decode_replay_matches_eager(cuda_dev, wl):
    """A whole step in one graph: reset, prompt attention (plan, the scan
    launched as a programmatic dependent, the attention kernel) for every
    layer, then one decode step of every layer. Each replay must give exactly
    the eager step's attention outputs and slot counts (page ids may differ:
    heads take pages from the pool in a racy order)."""
    p = S.append_prob(wl)
    eager, graphed = H.cache_for(wl, cuda_dev), H.cache_for(wl, cuda_dev)
    prompts = [S.gen_prompt(wl, layer, cuda_dev, p=p, full_q=True) for layer in range(wl.num_layers)]
    dec = [S.gen_decode(wl, layer, 0, cuda_dev, p=p) for layer in range(wl.num_layers)]
    pa_g = [torch.empty_like(pr["q"]) for pr in prompts]
    o_g = [torch.empty_like(x["q"]) for x in dec]

    def step(cache, pa_out, dec_out):
        cache.reset()
        for layer, pr in enumerate(prompts):
            cache.prefill_attention(layer, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"],
                                    pa_out[layer])
        for layer, x in enumerate(dec):
            cache.decode(layer, x["q"], x["k"], x["v"], dec_out[layer])

    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step(graphed, pa_g, o_g)
    for rep in range(2):
        pa_e = [torch.empty_like(pr["q"]) for pr in prompts]
        o_e = [torch.empty_like(x["q"]) for x in dec]
        step(eager, pa_e, o_e)
        g.replay()
        torch.cuda.synchronize()
        for layer in range(wl.num_layers):
            assert torch.equal(pa_g[layer], pa_e[layer]), (rep, layer)
            assert torch.equal(o_g[layer], o_e[layer]), (rep, layer)
            assert torch.equal(graphed.lengths(layer), eager.lengths(layer)), (rep, layer)
        assert graphed.status()[:2] == (0, 0)
        assert eager.status()[:2] == (0, 0)
