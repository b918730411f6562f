"""Prompt-phase attention on the tensor cores (GPU) against the fp64 oracle.

dmc_prefill_attention compresses a prompt (as dmc_prefill_compress) and returns
the output of every prompt token over the cache as it stands right after that
token's own update; the oracle runs the prompt token by token through
Algorithm 1 and attends after each update (oracle.dmc_ref.prompt_attention).
Checked: every output row and the cache contents (max-abs 2e-2, bf16), every
slot count (exact), grouped queries, prompts split over two calls, the
all-append and all-accumulate extremes, and decode continuing afterwards.
"""
import numpy as np
import pytest
import torch

from oracle import cref
from paper_2403_09636_gb300 import DmcCache, synthetic as S
from tests import dmc_harness as H

pytestmark = pytest.mark.gpu
TOL = 2e-2


def _wl(name, B, Hq, Hkv, prompt, cr, seed, layers=1):
    return S.Workload(name, layers, B, Hq, Hkv, 128, "bf16", prompt, 0, cr, 0.5, seed=seed)


def _cache(wl, extra_tokens=0, extra_steps=0):
    lens = S.prompt_lengths(wl)
    max_slots = int(lens.max()) + extra_tokens + extra_steps + 1
    NH = wl.batch * wl.num_kv_heads
    pages = wl.num_layers * NH * ((max_slots + 31) // 32) + 8
    return DmcCache(wl.num_layers, wl.batch, wl.num_q_heads, wl.num_kv_heads, 128, torch.bfloat16,
                    max_slots, pages, int(lens.sum()) + extra_tokens, device="cuda")


def _f(t):
    return t.float().cpu().numpy()


def _check_layer(wl, cache, layer, pr, out, parts=None):
    """Outputs, slot counts and slots of every head against the oracle. `parts`:
    per sequence, the prompt split [(k, v, q) before, (k, v, q) after] when the
    outputs cover only the second part."""
    G = wl.group
    cu = pr["cu_seqlens"].cpu().numpy()
    heads, where = [], []
    for b in range(wl.batch):
        sl = slice(int(cu[b]), int(cu[b + 1]))
        for h in range(wl.num_kv_heads):
            k, v = _f(pr["k"][sl, h]), _f(pr["v"][sl, h])
            q = _f(pr["q"][sl, h * G:(h + 1) * G])
            if parts is None:
                kp, vp, q0p = np.zeros((0, 128)), np.zeros((0, 128)), np.zeros((0, G))
            else:
                (kp, vp, qp) = parts[b][h]
                q0p = qp[:, :, 0]
            heads.append({"k_prompt": kp, "v_prompt": vp, "q0_prompt": q0p,
                          "k_dec": k, "v_dec": v, "q_dec": q})
            where.append((b, h, sl))
    ref = cref.run_heads(heads, threads=8)
    got_len = cache.lengths(layer).cpu().numpy()
    bad = []
    for (b, h, sl), r in zip(where, ref):
        if got_len[b, h] != r["len"]:
            bad.append(f"len b{b} h{h}: {got_len[b, h]} != {r['len']}")
            continue
        o = _f(out[sl, h * G:(h + 1) * G])
        err = float(np.max(np.abs(o - r["out"]))) if o.size else 0.0
        if not err <= TOL:
            bad.append(f"out b{b} h{h}: {err}")
        K, V, z, n = cache.export_heads(layer, [b * wl.num_kv_heads + h], int(r["len"]) + 1)
        for nm, x, y in (("K", _f(K[0, :r["len"]]), r["K"]), ("V", _f(V[0, :r["len"]]), r["V"]),
                         ("z", z[0, :r["len"]].cpu().numpy(), r["z"])):
            e = float(np.max(np.abs(x - y))) if x.size else 0.0
            if not e <= TOL:
                bad.append(f"{nm} b{b} h{h}: {e}")
    return bad


@pytest.mark.parametrize("G", [1, 2, 4, 8])
def test_prompt_attention_matches_oracle(cuda_dev, G):
    wl = _wl(f"pa_g{G}", 3, 2 * G, 2, (1, 700), ("choice", (1.0, 2.0, 4.0, 8.0)), seed=40 + G)
    cache = _cache(wl)
    pr = S.gen_prompt(wl, 0, cuda_dev, full_q=True)
    out = torch.full_like(pr["q"], float("nan"))
    cache.prefill_attention(0, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"], out)
    bad = _check_layer(wl, cache, 0, pr, out)
    assert not bad, bad[:8]
    assert cache.status()[:2] == (0, 0)


@pytest.mark.parametrize("cr", [1.0, 2.0])
def test_long_prompts_many_slot_tiles(cuda_dev, cr):
    """Prompts up to 2600 tokens: up to ~20 tiles of 128 slots per query row."""
    wl = _wl(f"pa_long{cr}", 2, 4, 4, (1900, 2600), ("fixed", cr), seed=50)
    cache = _cache(wl)
    pr = S.gen_prompt(wl, 0, cuda_dev, full_q=True)
    out = torch.empty_like(pr["q"])
    cache.prefill_attention(0, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"], out)
    bad = _check_layer(wl, cache, 0, pr, out)
    assert not bad, bad[:8]


def test_all_accumulate_one_segment(cuda_dev):
    """CR huge: essentially one segment per head; rows see almost only their
    running state (the diagonal term) across many chunk boundaries."""
    wl = _wl("pa_acc", 2, 2, 2, (300, 900), ("fixed", 1e6), seed=51)
    cache = _cache(wl)
    pr = S.gen_prompt(wl, 0, cuda_dev, full_q=True)
    out = torch.empty_like(pr["q"])
    cache.prefill_attention(0, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"], out)
    bad = _check_layer(wl, cache, 0, pr, out)
    assert not bad, bad[:8]


@pytest.mark.parametrize("G", [1, 4])
def test_prompt_split_over_two_calls(cuda_dev, G):
    """The second call continues every head's last segment (carry from the old
    last slot) and sees the first call's slots."""
    wl = _wl(f"pa_split{G}", 3, 2 * G, 2, (200, 600), ("choice", (1.0, 3.0, 6.0)), seed=60 + G)
    cache = _cache(wl)
    pr = S.gen_prompt(wl, 0, cuda_dev, full_q=True)
    cu = pr["cu_seqlens"].cpu().numpy()
    rng = np.random.default_rng(7)
    cuts = [int(rng.integers(1, int(cu[b + 1] - cu[b]))) for b in range(wl.batch)]
    idx1 = np.concatenate([np.arange(cu[b], cu[b] + cuts[b]) for b in range(wl.batch)])
    idx2 = np.concatenate([np.arange(cu[b] + cuts[b], cu[b + 1]) for b in range(wl.batch)])
    cu1 = torch.tensor(np.concatenate([[0], np.cumsum(cuts)]), dtype=torch.int32, device=cuda_dev)
    n2 = [int(cu[b + 1] - cu[b]) - cuts[b] for b in range(wl.batch)]
    cu2 = torch.tensor(np.concatenate([[0], np.cumsum(n2)]), dtype=torch.int32, device=cuda_dev)
    i1 = torch.as_tensor(idx1, device=cuda_dev)
    i2 = torch.as_tensor(idx2, device=cuda_dev)
    p1 = {k: pr[k][i1].contiguous() for k in ("q", "k", "v")}
    p2 = {k: pr[k][i2].contiguous() for k in ("q", "k", "v")}
    o1 = torch.empty_like(p1["q"])
    o2 = torch.empty_like(p2["q"])
    cache.prefill_attention(0, p1["q"], p1["k"], p1["v"], cu1, max(cuts), o1)
    cache.prefill_attention(0, p2["q"], p2["k"], p2["v"], cu2, max(n2), o2)
    pr2 = dict(p2, cu_seqlens=cu2)
    parts = [[(_f(p1["k"][cu1[b]:cu1[b + 1], h]), _f(p1["v"][cu1[b]:cu1[b + 1], h]),
               _f(p1["q"][cu1[b]:cu1[b + 1], h * G:(h + 1) * G])) for h in range(wl.num_kv_heads)]
             for b in range(wl.batch)]
    bad = _check_layer(wl, cache, 0, pr2, o2, parts=parts)
    assert not bad, bad[:8]


def test_decode_after_prompt_attention(cuda_dev):
    """The cache a prompt-attention call leaves is the one decode continues."""
    wl = _wl("pa_dec", 2, 4, 4, (100, 500), ("fixed", 3.0), seed=70, layers=2)
    steps = 6
    cache = _cache(wl, extra_steps=steps)
    prompts = [S.gen_prompt(wl, l, cuda_dev, full_q=True) for l in range(2)]
    for l, pr in enumerate(prompts):
        out = torch.empty_like(pr["q"])
        cache.prefill_attention(l, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"], out)
    decs = [[S.gen_decode(wl, l, t, cuda_dev) for l in range(2)] for t in range(steps)]
    outs = [[None, None] for _ in range(steps)]
    for t in range(steps):
        for l in range(2):
            o = torch.empty_like(decs[t][l]["q"])
            cache.decode(l, decs[t][l]["q"], decs[t][l]["k"], decs[t][l]["v"], o)
            outs[t][l] = o
    for l, pr in enumerate(prompts):
        cu = pr["cu_seqlens"].cpu().numpy()
        for b in range(wl.batch):
            sl = slice(int(cu[b]), int(cu[b + 1]))
            for h in range(wl.num_kv_heads):
                r = cref.run_heads([{
                    "k_prompt": _f(pr["k"][sl, h]), "v_prompt": _f(pr["v"][sl, h]),
                    "q0_prompt": _f(pr["q"][sl, h:h + 1, 0]),
                    "k_dec": np.stack([_f(decs[t][l]["k"][b, h]) for t in range(steps)]),
                    "v_dec": np.stack([_f(decs[t][l]["v"][b, h]) for t in range(steps)]),
                    "q_dec": np.stack([_f(decs[t][l]["q"][b, h:h + 1]) for t in range(steps)])}])[0]
                got = np.stack([_f(outs[t][l][b, h:h + 1]) for t in range(steps)])
                assert np.max(np.abs(got - r["out"])) <= TOL, (l, b, h)
    assert cache.status()[:2] == (0, 0)


def test_unsupported_caches_are_rejected(cuda_dev):
    from paper_2403_09636_gb300 import DmcError
    c = DmcCache(1, 1, 2, 2, 64, torch.bfloat16, 64, 8, 16, device="cuda")
    x = torch.zeros((4, 2, 64), dtype=torch.bfloat16, device=cuda_dev)
    cu = torch.tensor([0, 4], dtype=torch.int32, device=cuda_dev)
    with pytest.raises(DmcError):
        c.prefill_attention(0, x, x, x, cu, 4, torch.empty_like(x))
