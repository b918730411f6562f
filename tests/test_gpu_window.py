"""The window-grouping approximation (Sec. 3.3) on the GPU against the fp64
oracle: a slot is the omega-weighted mean of the last min(segment length, w)
tokens of its segment, the window cache holding each open segment's last
tokens across prefill and decode calls. Lengths exact; slots, z and outputs
within 2e-2 (bf16) / 1e-4 (fp32)."""
import numpy as np
import pytest
import torch

from oracle import cref
from paper_2403_09636_gb300 import DmcError, synthetic as S
from tests import dmc_harness as H

pytestmark = pytest.mark.gpu


def _check(run):
    assert run.len_ok, run.len_msgs[:5]
    bad = run.compare()
    assert not bad, bad[:10]


@pytest.mark.parametrize("window", [1, 4, 12])
def test_window_mha_bf16(cuda_dev, window):
    # CR up to 20: segments much longer than the window
    wl = S.Workload(f"win_mha_{window}", 2, 3, 4, 4, 128, "bf16", (60, 400), 30,
                    ("choice", (1.0, 3.0, 20.0)), 0.5, seed=100 + window)
    _check(H.Run(wl, cuda_dev, H.all_samples(wl), window=window))


@pytest.mark.parametrize("window", [3, 12])
def test_window_gqa_tensor_core(cuda_dev, window):
    wl = S.Workload(f"win_gqa_{window}", 2, 3, 8, 2, 128, "bf16", (80, 500), 30,
                    ("choice", (2.0, 16.0)), 0.5, seed=110 + window)
    _check(H.Run(wl, cuda_dev, H.all_samples(wl), window=window))


def test_window_fp32_grouped_virtual_heads(cuda_dev):
    """fp32 groups run every query head as its own unit list entry: one writer
    updates the window cache while the group's other queries read it."""
    wl = S.Workload("win_f32_g2", 1, 2, 4, 2, 128, "f32", (90, 200), 30, ("fixed", 8.0), 1.0, seed=120)
    for _ in range(3):
        r = H.Run(wl, cuda_dev, H.all_samples(wl), window=5)
        assert r.len_ok, r.len_msgs[:5]
        bad = r.compare(tol=1e-4)
        assert not bad, bad[:10]


def test_window_prompt_split_over_calls(cuda_dev):
    """The second call continues open segments whose last tokens come from the
    window cache; decode follows."""
    W, G = 6, 1
    wl = S.Workload("win_split", 1, 3, 2, 2, 128, "bf16", (100, 300), 0, ("fixed", 10.0), 0.5, seed=130)
    cache = H.cache_for(wl, cuda_dev, max_slots=400, num_pages=64, window=W)
    pr = S.gen_prompt(wl, 0, cuda_dev)
    cu = pr["cu_seqlens"].cpu().numpy()
    rng = np.random.default_rng(3)
    cuts = [int(rng.integers(1, int(cu[b + 1] - cu[b]))) for b in range(wl.batch)]
    lo = [int(cu[b]) for b in range(wl.batch)]
    mid = [int(cu[b]) + cuts[b] for b in range(wl.batch)]
    hi = [int(cu[b + 1]) for b in range(wl.batch)]
    for first, last in ((lo, mid), (mid, hi)):
        idx = torch.as_tensor(np.concatenate([np.arange(first[b], last[b]) for b in range(wl.batch)]),
                              device=cuda_dev)
        n = [last[b] - first[b] for b in range(wl.batch)]
        cuu = torch.tensor(np.concatenate([[0], np.cumsum(n)]), dtype=torch.int32, device=cuda_dev)
        cache.prefill(0, pr["q0"][idx].contiguous(), pr["k"][idx].contiguous(), pr["v"][idx].contiguous(),
                      cuu, max(n))
    steps = 8
    decs = [S.gen_decode(wl, 0, t, cuda_dev) for t in range(steps)]
    outs = []
    for d in decs:
        o = torch.empty_like(d["q"])
        cache.decode(0, d["q"], d["k"], d["v"], o)
        outs.append(o)
    f = lambda t: t.float().cpu().numpy()
    for b in range(wl.batch):
        sl = slice(int(cu[b]), int(cu[b + 1]))
        for h in range(wl.num_kv_heads):
            r = cref.run_heads([{"k_prompt": f(pr["k"][sl, h]), "v_prompt": f(pr["v"][sl, h]),
                                 "q0_prompt": f(pr["q0"][sl, h:h + 1]),
                                 "k_dec": np.stack([f(d["k"][b, h]) for d in decs]),
                                 "v_dec": np.stack([f(d["v"][b, h]) for d in decs]),
                                 "q_dec": np.stack([f(d["q"][b, h:h + 1]) for d in decs])}], window=W)[0]
            got = np.stack([f(o[b, h:h + 1]) for o in outs])
            assert np.max(np.abs(got - r["out"])) <= 2e-2, (b, h)
            K, V, z, n = cache.export_heads(0, [b * wl.num_kv_heads + h], r["len"] + 1)
            assert int(n[0]) == r["len"]
            assert np.max(np.abs(f(K[0, :r["len"]]) - r["K"])) <= 2e-2
            assert np.max(np.abs(z[0, :r["len"]].cpu().numpy() - r["z"])) <= 2e-2
    assert cache.status()[:2] == (0, 0)


def test_prompt_attention_rejects_window(cuda_dev):
    wl = S.Workload("win_pa", 1, 1, 2, 2, 128, "bf16", (50, 50), 0, ("fixed", 2.0), 0.5, seed=140)
    cache = H.cache_for(wl, cuda_dev, window=4)
    pr = S.gen_prompt(wl, 0, cuda_dev, full_q=True)
    with pytest.raises(DmcError):
        cache.prefill_attention(0, pr["q"], pr["k"], pr["v"], pr["cu_seqlens"], pr["max_seqlen"],
                                torch.empty_like(pr["q"]))
