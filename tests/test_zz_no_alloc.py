"""dmc_decode_step_static_scratch against dmc_decode_step (GPU).

The static-scratch entry point serves callers that cannot allocate device
memory of their own (a plugin handed only its input and output buffers by a
framework that owns every allocation, or a loop that must not pay cudaMalloc's
implicit synchronisation): its split-K scratch lives in the library's static
device array instead. When the cache's decode grid fits the array it runs the
same launch as the regular entry point, and the launches are deterministic,
so outputs, slot counts and slots must be bit-identical, on two calls in a
row. Covered: the MHA CUDA-core kernel (bf16 d 128 with long heads split over
many warps; fp32 d 64), and the tensor-core kernel for a group of 8 queries
with a cache big enough for the full grid (two states per query per warp).
This file is collected last so that a failure here does not hide any other
test; it passes alone in a fresh process and after the other tests.
"""
import pytest
import torch

import paper_2403_09636_gb300 as P

pytestmark = pytest.mark.gpu


def _inputs(seed, n, Hkv, Hq, d, p_append, dtype):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    k = torch.randn((n, Hkv, d), generator=g, device="cuda") * 0.5
    v = torch.randn((n, Hkv, d), generator=g, device="cuda") * 0.5
    q = torch.randn((n, Hq, d), generator=g, device="cuda") * 0.5
    sign = torch.where(torch.rand((n, Hkv), generator=g, device="cuda") < p_append, -1.0, 1.0)
    k[:, :, 0] = sign * 0.5 * (torch.randn((n, Hkv), generator=g, device="cuda").abs() + 0.1)
    return q.to(dtype), k.to(dtype), v.to(dtype)


def _cache(B, Hkv, Hq, d, T, q, k, v, dtype):
    c = P.DmcCache(1, B, Hq, Hkv, d, dtype, T + 8, B * Hkv * (T // 32 + 2), B * T)
    cu = torch.arange(0, B * T + 1, T, dtype=torch.int32, device="cuda")
    c.prefill(0, q[:, :, 0], k, v, cu, T)
    return c


CASES = [
    # (B, Hkv, Hq, d, T, p_append, dtype): long MHA heads (3000 slots at CR ~1.1)
    # split over many warps, so the partial states carry real data
    (2, 4, 4, 128, 3000, 0.9, torch.bfloat16),
    (1, 3, 3, 64, 200, 0.5, torch.float32),
    # grouped queries on the tensor-core kernel: 16 KV heads of 3000 slots give
    # the full grid of one block per SM, 16 partial states per warp
    (4, 4, 32, 128, 3000, 0.9, torch.bfloat16),
]


@pytest.mark.parametrize("case", CASES, ids=["mha_bf16_d128", "mha_f32_d64", "gqa8_bf16_d128"])
def test_static_scratch_matches_regular_decode_two_calls(cuda_dev, case):
    B, Hkv, Hq, d, T, p, dt = case
    q, k, v = _inputs(21, B * T, Hkv, Hq, d, p, dt)
    ref = _cache(B, Hkv, Hq, d, T, q, k, v, dt)
    tst = _cache(B, Hkv, Hq, d, T, q, k, v, dt)
    s = torch.cuda.current_stream().cuda_stream
    for step in range(2):
        qd, kd, vd = (t.contiguous() for t in _inputs(100 + step, B, Hkv, Hq, d, 0.5, dt))
        out_ref = torch.empty_like(qd)
        out_tst = torch.full_like(qd, float("nan"))
        assert P.dmc_decode_step(ref.handle, 0, qd.data_ptr(), kd.data_ptr(), vd.data_ptr(),
                                 out_ref.data_ptr(), s) == P.DMC_OK
        assert P.dmc_decode_step_static_scratch(tst.handle, 0, qd.data_ptr(), kd.data_ptr(),
                                                vd.data_ptr(), out_tst.data_ptr(), s) == P.DMC_OK
        torch.cuda.synchronize()
        assert torch.equal(out_ref, out_tst), (step, (out_ref.float() - out_tst.float()).abs().max())
        assert torch.equal(ref.lengths(0), tst.lengths(0)), step
    ids = list(range(B * Hkv))
    for a, b in zip(ref.export_heads(0, ids, T + 8), tst.export_heads(0, ids, T + 8)):
        assert torch.equal(a, b)
    assert ref.status()[0] == P.DMC_OK and tst.status()[0] == P.DMC_OK


def test_static_scratch_rejects_null_handle():
    assert P.dmc_decode_step_static_scratch(None, 0, 16, 16, 16, 16, 0) == P.DMC_ERR_INVALID_ARG
