"""Edge cases of the CUDA path (GPU): empty caches, page boundaries, prompts
split across calls, sub-batches, faults reported through the sticky status
bits, and run-to-run determinism."""
import numpy as np
import pytest
import torch

from oracle import cref
from paper_2403_09636_gb300 import (DMC_ERR_DEVICE_FAULT, DMC_ERR_PAGES_EXHAUSTED,
                                    DMC_FAULT_BAD_SEQLENS, DMC_FAULT_NAN_GATE,
                                    DMC_FAULT_PAGES_EXHAUSTED, DMC_FAULT_SLOT_CAPACITY, DmcCache,
                                    DmcError)

pytestmark = pytest.mark.gpu


def _tokens(gen, n, H, d, k0_sign, scale=0.5, dtype=torch.bfloat16, G=1, dev="cuda"):
    """n tokens; k0_sign [n, H] of +-1 decides accumulate/append."""
    k = torch.randn((n, H, d), generator=gen, device=dev) * scale
    v = torch.randn((n, H, d), generator=gen, device=dev) * scale
    q = torch.randn((n, H * G, d), generator=gen, device=dev) * scale
    mag = torch.randn((n, H), generator=gen, device=dev).abs() + 0.1
    k[:, :, 0] = torch.as_tensor(k0_sign, dtype=torch.float32, device=dev) * scale * mag
    return q.to(dtype), k.to(dtype), v.to(dtype)


def _oracle_head(kp, vp, q0p, kd, vd, qd):
    f = lambda t: t.float().cpu().numpy()
    return cref.run_heads([{"k_prompt": f(kp), "v_prompt": f(vp), "q0_prompt": f(q0p),
                            "k_dec": f(kd), "v_dec": f(vd), "q_dec": f(qd)}])[0]


def _gen(seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return g


@pytest.mark.parametrize("n_prompt", [0, 1, 31, 32, 33, 64, 65])
def test_page_boundaries_all_append(cuda_dev, n_prompt):
    """Every token appends: the cache is the plain KV cache, crossing pages."""
    H, d, steps = 2, 128, 40
    g = _gen(n_prompt)
    n = n_prompt + steps
    q, k, v = _tokens(g, n, H, d, -np.ones((n, H)))
    c = DmcCache(1, 1, H, H, d, torch.bfloat16, n + 1, 2 * ((n + 31) // 32) + 2, max(n_prompt, 1))
    if n_prompt:
        cu = torch.tensor([0, n_prompt], dtype=torch.int32, device=cuda_dev)
        c.prefill(0, q[:n_prompt, :, 0], k[:n_prompt], v[:n_prompt], cu, n_prompt)
    outs = []
    for t in range(n_prompt, n):
        out = torch.empty_like(q[t:t + 1])
        c.decode(0, q[t:t + 1], k[t:t + 1], v[t:t + 1], out)
        outs.append(out)
    outs = torch.cat(outs)
    assert c.lengths(0).cpu().tolist() == [[n, n]]
    for h in range(H):
        r = _oracle_head(k[:n_prompt, h], v[:n_prompt, h], q[:n_prompt, h:h + 1, 0],
                         k[n_prompt:, h], v[n_prompt:, h], q[n_prompt:, h:h + 1])
        assert np.max(np.abs(outs[:, h].float().cpu().numpy() - r["out"][:, 0])) <= 2e-2
    st, bits, used = c.status()
    assert st == 0 and bits == 0 and used == H * ((n + 31) // 32)


def test_all_accumulate_single_slot(cuda_dev):
    """Every token after the first accumulates: one slot holding the
    omega-weighted mean of the whole stream."""
    H, d, n_prompt, steps = 3, 64, 500, 20
    g = _gen(5)
    n = n_prompt + steps
    q, k, v = _tokens(g, n, H, d, np.ones((n, H)), dtype=torch.float32, scale=1.0)
    c = DmcCache(1, 1, H, H, d, torch.float32, 4, 8, n_prompt)
    cu = torch.tensor([0, n_prompt], dtype=torch.int32, device=cuda_dev)
    c.prefill(0, q[:n_prompt, :, 0], k[:n_prompt], v[:n_prompt], cu, n_prompt)
    outs = []
    for t in range(n_prompt, n):
        out = torch.empty_like(q[t:t + 1])
        c.decode(0, q[t:t + 1], k[t:t + 1], v[t:t + 1], out)
        outs.append(out)
    outs = torch.cat(outs)
    assert c.lengths(0).cpu().tolist() == [[1, 1, 1]]
    kk, vv, zz, ln = c.export_heads(0, list(range(H)), 2)
    for h in range(H):
        r = _oracle_head(k[:n_prompt, h], v[:n_prompt, h], q[:n_prompt, h:h + 1, 0],
                         k[n_prompt:, h], v[n_prompt:, h], q[n_prompt:, h:h + 1])
        assert np.max(np.abs(outs[:, h].cpu().numpy() - r["out"][:, 0])) <= 1e-4
        assert np.max(np.abs(kk[h, 0].cpu().numpy() - r["K"][0])) <= 1e-4
        assert abs(float(zz[h, 0]) - r["z"][0]) <= 1e-3


def test_prompt_split_across_calls_and_sub_batches(cuda_dev):
    """Prefill in two token chunks and two sequence groups equals the oracle
    run over the whole stream."""
    B, H, d = 3, 4, 128
    lens = [170, 61, 300]
    g = _gen(9)
    data = [_tokens(g, n, H, d, np.where(np.random.default_rng(b).random((n, H)) < 0.3, -1, 1))
            for b, n in enumerate(lens)]
    c = DmcCache(1, B, H, H, d, torch.bfloat16, 400, 64, 600)
    cut = [100, 61, 37]  # first part of each prompt
    # call 1: sequences 0..1, first parts; call 2: sequence 2 first part; call 3: all second parts
    def pack(parts):
        q0 = torch.cat([p[0][:, :, 0] for p in parts])
        k = torch.cat([p[1] for p in parts])
        v = torch.cat([p[2] for p in parts])
        cu = torch.tensor(np.concatenate([[0], np.cumsum([p[1].shape[0] for p in parts])]),
                          dtype=torch.int32, device=cuda_dev)
        return q0, k, v, cu, max(p[1].shape[0] for p in parts)
    first = [tuple(t[:cut[b]] for t in data[b]) for b in range(B)]
    second = [tuple(t[cut[b]:] for t in data[b]) for b in range(B)]
    q0, k, v, cu, mx = pack(first[:2])
    c.prefill(0, q0, k, v, cu, mx, first_seq=0)
    q0, k, v, cu, mx = pack(first[2:])
    c.prefill(0, q0, k, v, cu, mx, first_seq=2)
    q0, k, v, cu, mx = pack(second)
    c.prefill(0, q0, k, v, cu, mx, first_seq=0)
    kk, vv, zz, ln = c.export_heads(0, list(range(B * H)), 400)
    for b in range(B):
        q, kb, vb = data[b]
        for h in range(H):
            r = _oracle_head(kb[:, h], vb[:, h], q[:, h:h + 1, 0], kb[:0, h], vb[:0, h], q[:0, h:h + 1])
            i = b * H + h
            n = int(ln[i])
            assert n == r["prompt_len"]
            assert np.max(np.abs(kk[i, :n].float().cpu().numpy() - r["prompt_K"])) <= 2e-2
            assert np.max(np.abs(vv[i, :n].float().cpu().numpy() - r["prompt_V"])) <= 2e-2
            assert np.max(np.abs(zz[i, :n].cpu().numpy() - r["prompt_z"])) <= 2e-2
    assert c.status()[0] == 0


def test_decode_is_deterministic(cuda_dev):
    """Split heads are merged in a fixed block order, so two identical runs
    give bit-identical outputs."""
    B, H, d, n_prompt = 4, 8, 128, 1500
    g = _gen(11)
    q, k, v = _tokens(g, B * n_prompt, H, d, np.where(np.random.default_rng(0).random((B * n_prompt, H)) < 0.25, -1, 1))
    cu = torch.arange(0, B * n_prompt + 1, n_prompt, dtype=torch.int32, device=cuda_dev)
    qd, kd, vd = _tokens(g, B, H, d, np.ones((B, H)))
    outs = []
    for _ in range(2):
        c = DmcCache(1, B, H, H, d, torch.bfloat16, n_prompt + 4, 4096, B * n_prompt)
        c.prefill(0, q[:, :, 0], k, v, cu, n_prompt)
        out = torch.empty_like(qd)
        c.decode(0, qd, kd, vd, out)
        outs.append(out)
        assert c.status()[0] == 0
    assert torch.equal(outs[0], outs[1])


def test_pool_exhausted_is_reported(cuda_dev):
    H, d, n = 4, 64, 200
    g = _gen(12)
    q, k, v = _tokens(g, n, H, d, -np.ones((n, H)))
    c = DmcCache(1, 1, H, H, d, torch.bfloat16, 1024, 10, n)  # needs 4 * 7 pages
    cu = torch.tensor([0, n], dtype=torch.int32, device=cuda_dev)
    c.prefill(0, q[:, :, 0], k, v, cu, n)
    st, bits, _ = c.status()
    assert st == DMC_ERR_PAGES_EXHAUSTED and bits & DMC_FAULT_PAGES_EXHAUSTED
    c.reset()
    assert c.status()[0] == 0


def test_slot_capacity_is_reported(cuda_dev):
    H, d, n = 2, 64, 100
    g = _gen(13)
    q, k, v = _tokens(g, n, H, d, -np.ones((n, H)))
    c = DmcCache(1, 1, H, H, d, torch.bfloat16, 64, 64, n)
    cu = torch.tensor([0, n], dtype=torch.int32, device=cuda_dev)
    c.prefill(0, q[:, :, 0], k, v, cu, n)
    st, bits, _ = c.status()
    assert st == DMC_ERR_DEVICE_FAULT and bits & DMC_FAULT_SLOT_CAPACITY
    assert c.lengths(0).cpu().tolist() == [[0, 0]]  # the faulty heads were left untouched
    # decode appends into a full head
    c.reset()
    c.prefill(0, q[:64, :, 0], k[:64], v[:64], torch.tensor([0, 64], dtype=torch.int32, device=cuda_dev), 64)
    assert c.status()[0] == 0
    out = torch.empty_like(q[64:65])
    c.decode(0, q[64:65], k[64:65], v[64:65], out)
    st, bits, _ = c.status()
    assert bits & DMC_FAULT_SLOT_CAPACITY
    assert c.lengths(0).cpu().tolist() == [[64, 64]]


def test_bad_seqlens_and_nan_gate_are_reported(cuda_dev):
    H, d, n = 2, 64, 40
    g = _gen(14)
    q, k, v = _tokens(g, n, H, d, np.ones((n, H)))
    c = DmcCache(1, 2, H, H, d, torch.bfloat16, 128, 64, n)
    bad = torch.tensor([0, 30, 20], dtype=torch.int32, device=cuda_dev)  # not monotone
    c.prefill(0, q[:, :, 0], k, v, bad, 30)
    st, bits, _ = c.status()
    assert bits & DMC_FAULT_BAD_SEQLENS
    c.reset()
    k2 = k.clone()
    k2[5, 1, 0] = float("nan")
    c.prefill(0, q[:20, :, 0], k2[:20], v[:20], torch.tensor([0, 10, 20], dtype=torch.int32, device=cuda_dev), 10)
    st, bits, _ = c.status()
    assert bits & DMC_FAULT_NAN_GATE
    # a NaN decision counts as append: head (0, 1) has 2 slots, head (0, 0) one
    assert c.lengths(0).cpu().tolist() == [[1, 2], [1, 1]]


def test_invalid_arguments_raise(cuda_dev):
    c = DmcCache(2, 1, 4, 4, 64, torch.float32, 64, 16, 32)
    x = torch.zeros((1, 4, 64), device=cuda_dev)
    with pytest.raises(DmcError):
        c.decode(2, x, x, x, x)  # layer out of range
    with pytest.raises(DmcError):
        c.prefill(0, x[:, :, 0], x, x, torch.tensor([0, 1], dtype=torch.int32, device=cuda_dev), 1,
                  first_seq=1)  # sequence out of range
    with pytest.raises(DmcError):
        big = torch.zeros((33, 4, 64), device=cuda_dev)
        c.prefill(0, big[:, :, 0], big, big, torch.tensor([0, 33], dtype=torch.int32, device=cuda_dev), 33)
