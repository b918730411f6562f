"""The CUDA path at the full sizes of the large workloads (GPU).

Each case runs the whole workload through the C ABI in the launch
configuration the benchmark uses (one cache, one launch per layer per decode
step, all decode steps) and checks, against the fp64 oracle:
  - the slot count of every head of every layer after the prompt and after
    every decode step (bit-exact);
  - slots, z and every decode output of 64 sampled (layer, sequence, KV head)
    instances (max-abs 2e-2, bf16 caches).
The page pool is sized exactly from the decisions. The 13B workload needs
~230 GB of cache: on a device with less free memory it keeps the leading
layers that fit, with the same per-layer shape and seeds.
"""
import pytest

from paper_2403_09636_gb300 import synthetic as S
from tests import dmc_harness as H

pytestmark = pytest.mark.gpu

CASES = ["llama2_7b_4x", "llama2_7b_mixed", "llama2_13b_4x", "llama2_70b_gqa_2x", "long_ragged",
         "llama2_7b_4x_hardc"]


@pytest.mark.parametrize("name", CASES)
def test_full_size_sampled(cuda_dev, name):
    wl = S.WORKLOADS[name]
    wl, cache = H.full_size_cache(wl, cuda_dev, wl.decode_steps)
    covered = f"{name}: {wl.num_layers} of {S.WORKLOADS[name].num_layers} layers checked"
    print(f"\n{covered}")
    run = H.Run(wl, cuda_dev, H.random_samples(wl, 64, seed=17), cache=cache)
    assert run.len_ok, (covered, run.len_msgs[:5])
    if wl.hardc:
        # DMC-HardC: every head of a sequence holds the same number of slots
        for layer in range(wl.num_layers):
            ln = cache.lengths(layer)
            assert bool((ln == ln[:, :1]).all()), (covered, layer)
    bad = run.compare()
    assert not bad, (covered, bad[:10])
    del run, cache
    import torch
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["llama2_7b_4x", "llama2_70b_gqa_2x"])
def test_full_size_multi_layer_launch(cuda_dev, name):
    """The bench workload (MHA, CUDA-core kernel) and the 70B GQA workload
    (tensor-core kernel) at full size with every decode step as
    dmc_decode_step_layers launches (two calls per step, each over half the
    layers): every slot count every step, and slots, z and every output of 64
    sampled heads against the oracle."""
    wl = S.WORKLOADS[name]
    wl, cache = H.full_size_cache(wl, cuda_dev, wl.decode_steps)
    covered = f"{name}: {wl.num_layers} of {S.WORKLOADS[name].num_layers} layers checked"
    print(f"\n{covered}")
    run = H.Run(wl, cuda_dev, H.random_samples(wl, 64, seed=18), cache=cache, launch="layers")
    assert run.len_ok, (covered, run.len_msgs[:5])
    bad = run.compare()
    assert not bad, (covered, bad[:10])
    del run, cache
    import torch
    torch.cuda.empty_cache()
