"""Decode steps in one launch over several layers (dmc_decode_step_layers) and
replayed from a CUDA graph, each checked against the fp64 oracle (GPU).

Every decode step of every layer is compared with the oracle's Algorithm 1 and
Eq. attn-softmax on the same inputs: slot counts of every head after every
step (exact), and slots, z and every output of every head (max-abs 2e-2 for
bf16, 1e-4 for fp32 caches). bf16 cases use the high-signal inputs of
test_gpu_signal.py and must also stay farther than the tolerance from each
mutant oracle. The multi-layer launch splits the layers over two calls, so a
first layer other than 0 is covered. Covered: MHA bf16 (several layers, the
owner warp's pages and splits), fp32 grouped queries on the CUDA-core kernel
(per-query virtual heads and their pending row), window grouping (MHA and
grouped queries), grouped bf16 queries on the tensor-core kernel (groups of 4
at d 128 and 8 at d 64, its own walk over the layers), and the tiny fp32
workload. A second test requires the multi-layer launch to give exactly the
outputs of per-layer launches (the same work split per layer).
"""
import numpy as np
import pytest

from paper_2403_09636_gb300 import synthetic as S
from tests import dmc_harness as H
from tests import mutants as M

pytestmark = pytest.mark.gpu


def _sig(name, layers, B, Hq, Hkv, d, prompt, steps, cr, seed):
    return S.Workload(name, layers, B, Hq, Hkv, d, "bf16", prompt, steps, cr, 0.5, seed=seed,
                      q_scale=6.0, v_block_offset=0.5)


CASES = [
    (_sig("modes_mha_bf16", 4, 3, 8, 8, 128, (40, 900), 10, ("choice", (1.0, 2.0, 4.0)), 401), 0),
    (S.Workload("modes_f32_g2", 3, 2, 4, 2, 64, "f32", (60, 200), 10, ("fixed", 3.0), 1.0, seed=402), 0),
    (_sig("modes_window", 3, 2, 4, 4, 128, (60, 400), 10, ("choice", (2.0, 16.0)), 403), 12),
    (_sig("modes_gqa4", 2, 2, 8, 2, 128, (100, 600), 10, ("fixed", 2.0), 404), 0),
    (_sig("modes_gqa8_d64", 3, 2, 16, 2, 64, (80, 500), 10, ("choice", (1.0, 4.0)), 405), 0),
    (_sig("modes_gqa2_window", 3, 2, 4, 2, 128, (60, 400), 10, ("choice", (2.0, 16.0)), 406), 12),
    (S.WORKLOADS["tiny_f32"], 0),
]


@pytest.mark.parametrize("launch", ["layers", "graph"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0].name)
def test_launch_mode_matches_oracle(cuda_dev, case, launch):
    wl, window = case
    run = H.Run(wl, cuda_dev, H.all_samples(wl), window=window, launch=launch)
    assert run.len_ok, run.len_msgs[:5]
    bad = run.compare()
    if wl.dtype == "bf16":
        worst, fails = M.decode_separation(run, H.TOL["bf16"])
        print(f"\n{wl.name} {launch}: min |gpu - mutant| " +
              ", ".join(f"{m} {worst[m]:.4f}" for m in M.MODES))
        bad += fails
    assert not bad, bad[:10]


@pytest.mark.parametrize("case", CASES[:6], ids=lambda c: c[0].name)
def test_multi_layer_launch_equals_per_layer_launches(cuda_dev, case):
    wl, window = case
    samples = H.all_samples(wl)
    a = H.Run(wl, cuda_dev, samples, window=window, launch="stream")
    b = H.Run(wl, cuda_dev, samples, window=window, launch="layers")
    for s in samples:
        assert np.array_equal(np.array(a.inst[s]["out"]), np.array(b.inst[s]["out"])), s
        for x, y in zip(a.final_export[s], b.final_export[s]):
            assert np.array_equal(np.asarray(x), np.asarray(y)), s
