"""Seeded synthetic inputs for the DMC hot path (no method arithmetic here).

The paper measures Llama 2 7B/13B/70B on English text (throughput section);
neither weights nor text are available, so seeded Gaussian q, k, v stand in for
them, with the decision neuron k[..., 0] drawn so that each KV head appends
with a chosen probability 1/CR (the paper reports decisions that do not depend
on position and CRs that differ per head). The same generator feeds the oracle
and the CUDA path; it only draws random numbers.

Recipe per workload (all tensors [tokens, heads, head_dim] row-major):
  q, k, v ~ N(0, 1) * scale                       (scale 0.5 bf16, 1.0 fp32)
  k[..., 0] = sign * scale * (|N(0, 1)| + 0.1)    sign = -1 with prob p_append
                                                  (k[0] < 0 -> alpha = 0 -> append)
  p_append[layer, kv_head] = 1 / CR, CR drawn per (layer, KV head)
  q[..., 0] ~ N(0, 1) * scale feeds omega
Values are drawn in fp32 and then cast, so |k[0]| >= 0.05 holds after the bf16
cast and no decision sits at the sigmoid tie.

High-signal variant (parity tests only; every workload above leaves it off):
  q ~ N(0, 1) * q_scale                           a larger query scale makes the
                                                  softmax peak over a few slots
  v += N(0, 1) * v_block_offset                   one offset vector per block of
                                                  16 prompt tokens (per decode
                                                  token), so slot values and
                                                  outputs are O(1), not O(1/sqrt n)
These draws come after the ones above, so a workload with both off draws
exactly the numbers it always did.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch

_MASK64 = (1 << 64) - 1


def derive_seed(*parts: int) -> int:
    """splitmix64 over the parts -> a 63-bit seed for torch.Generator."""
    x = 0x9E3779B97F4A7C15
    for p in parts:
        x = (x + (int(p) & _MASK64) + 0x9E3779B97F4A7C15) & _MASK64
        x ^= x >> 30
        x = (x * 0xBF58476D1CE4E5B9) & _MASK64
        x ^= x >> 27
        x = (x * 0x94D049BB133111EB) & _MASK64
        x ^= x >> 31
    return x & ((1 << 63) - 1)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    dtype: str                 # "f32" or "bf16"
    prompt: tuple              # (lo, hi) prompt tokens per sequence, uniform
    decode_steps: int
    cr: tuple                  # ("fixed", CR) | ("choice", (CRs...)) | ("loguniform", lo, hi)
    scale: float
    seed: int = 0
    # DMC-HardC (in-layer relaxation ablation): decisions and importance
    # shared by every head of a layer, so all heads of a sequence have the
    # same segments and lengths
    hardc: bool = False
    # high-signal parity inputs: query scale (0 = `scale`) and the std of a
    # per-block offset added to v (0 = none)
    q_scale: float = 0.0
    v_block_offset: float = 0.0

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def esize(self) -> int:
        return 4 if self.dtype == "f32" else 2


WORKLOADS = {
    # batch 1, 1 layer, 4 MHA heads, d 64, 256 prompt + 32 decode, p_append 0.5
    "tiny_f32": Workload("tiny_f32", 1, 1, 4, 4, 64, "f32", (256, 256), 32,
                         ("fixed", 2.0), 1.0),
    # Llama-2-7B attention shape, per-head CR drawn from {1, 2, 4, 8}
    "llama2_7b_mixed": Workload("llama2_7b_mixed", 32, 32, 32, 32, 128, "bf16",
                                (2048, 2048), 512, ("choice", (1.0, 2.0, 4.0, 8.0)), 0.5),
    # the same shape with a uniform 4x compression on every head
    "llama2_7b_4x": Workload("llama2_7b_4x", 32, 32, 32, 32, 128, "bf16",
                             (2048, 2048), 512, ("fixed", 4.0), 0.5),
    # Llama-2-13B shape, batch 256, 4096 prompt, uniform 4x
    "llama2_13b_4x": Workload("llama2_13b_4x", 40, 256, 40, 40, 128, "bf16",
                              (4096, 4096), 256, ("fixed", 4.0), 0.5),
    # Llama-2-70B shape: 64 query heads over 8 KV heads, DMC 2x per KV head
    "llama2_70b_gqa_2x": Workload("llama2_70b_gqa_2x", 80, 64, 64, 8, 128, "bf16",
                                  (4096, 4096), 256, ("fixed", 2.0), 0.5),
    # long ragged prompts U[1024, 32768], heavy-tailed CR log-uniform in [1, 32]
    "long_ragged": Workload("long_ragged", 32, 8, 32, 32, 128, "bf16",
                            (1024, 32768), 128, ("loguniform", 1.0, 32.0), 0.5),
    # the 7B 4x shape with DMC-HardC decisions: one alpha and omega per token
    # for all heads of a layer
    "llama2_7b_4x_hardc": Workload("llama2_7b_4x_hardc", 32, 32, 32, 32, 128, "bf16",
                                   (2048, 2048), 512, ("fixed", 4.0), 0.5, hardc=True),
}


def shrink(wl: Workload, **kw) -> Workload:
    """A copy of a workload with some fields replaced (smaller parity cases)."""
    return dataclasses.replace(wl, **kw)


def append_prob(wl: Workload) -> np.ndarray:
    """p_append [num_layers, num_kv_heads] (float64) = 1 / CR per KV head."""
    g = torch.Generator().manual_seed(derive_seed(wl.seed, 11))
    L, H = wl.num_layers, wl.num_kv_heads
    kind = wl.cr[0]
    if kind == "fixed":
        cr = torch.full((L, H), float(wl.cr[1]), dtype=torch.float64)
    elif kind == "choice":
        opts = torch.tensor(wl.cr[1], dtype=torch.float64)
        cr = opts[torch.randint(len(opts), (L, H), generator=g)]
    elif kind == "loguniform":
        lo, hi = math.log(wl.cr[1]), math.log(wl.cr[2])
        u = torch.rand((L, H), generator=g, dtype=torch.float64)
        cr = torch.exp(lo + (hi - lo) * u)
    else:
        raise ValueError(kind)
    return (1.0 / cr).numpy()


def prompt_lengths(wl: Workload) -> np.ndarray:
    """Prompt length of every sequence [batch] (int64)."""
    lo, hi = wl.prompt
    if lo == hi:
        return np.full(wl.batch, lo, dtype=np.int64)
    g = torch.Generator().manual_seed(derive_seed(wl.seed, 13))
    return torch.randint(lo, hi + 1, (wl.batch,), generator=g).numpy().astype(np.int64)


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _draw_tokens(n, wl: Workload, p_layer, g, device, want_full_q: bool, block: int = 1):
    """Draw n tokens of one layer in fp32: q (full or first neuron), k, v.
    `block`: tokens that share one v offset (high-signal variant only)."""
    H, Hq, d, s = wl.num_kv_heads, wl.num_q_heads, wl.head_dim, wl.scale
    qs = wl.q_scale if wl.q_scale > 0 else s
    k = torch.randn((n, H, d), generator=g, device=device) * s
    v = torch.randn((n, H, d), generator=g, device=device) * s
    if want_full_q:
        q = torch.randn((n, Hq, d), generator=g, device=device) * qs
    else:
        q = torch.randn((n, Hq), generator=g, device=device) * qs
    u = torch.rand((n, H), generator=g, device=device)
    mag = torch.randn((n, H), generator=g, device=device).abs() + 0.1
    p = torch.as_tensor(p_layer, dtype=torch.float32, device=device)
    if wl.hardc:
        # one decision and one importance per token for every head of the layer
        u, mag, p = u[:, :1].expand(n, H), mag[:, :1].expand(n, H), p[:1].expand(H)
        if want_full_q:
            q[:, :, 0] = q[:, :1, 0]
        else:
            q[:, :] = q[:, :1].clone()
    sign = torch.where(u < p[None, :], -1.0, 1.0)
    k[:, :, 0] = sign * s * mag
    if wl.v_block_offset > 0 and n > 0:
        nb = (n + block - 1) // block
        off = torch.randn((nb, H, d), generator=g, device=device) * wl.v_block_offset
        v = v + off.repeat_interleave(block, dim=0)[:n]
    return q, k, v


def gen_prompt(wl: Workload, layer: int, device, seqs=None, p=None, full_q: bool = False):
    """Prompt inputs of one layer for the sequences `seqs` (default: all).

    Returns dict q0 [sum T, Hq] (first neuron of every query), k, v
    [sum T, Hkv, d] in the workload dtype, cu_seqlens int32 [n+1] (on `device`)
    and the per-sequence lengths (numpy). Each sequence has its own generator
    stream, so any subset is reproducible. With full_q the whole queries are
    drawn too ("q" [sum T, Hq, d], q0 = its first neuron); that draws more
    numbers, so those prompts differ from the default ones."""
    if seqs is None:
        seqs = range(wl.batch)
    seqs = list(seqs)
    if p is None:
        p = append_prob(wl)
    lens = prompt_lengths(wl)[seqs]
    total = int(lens.sum())
    H, Hq, d = wl.num_kv_heads, wl.num_q_heads, wl.head_dim
    dt = wl.torch_dtype
    q0 = torch.empty((total, Hq), dtype=dt, device=device)
    qf = torch.empty((total, Hq, d), dtype=dt, device=device) if full_q else None
    k = torch.empty((total, H, d), dtype=dt, device=device)
    v = torch.empty((total, H, d), dtype=dt, device=device)
    off = 0
    for b, n in zip(seqs, lens):
        n = int(n)
        g = _gen(device, derive_seed(wl.seed, 1, layer, b))
        qb, kb, vb = _draw_tokens(n, wl, p[layer], g, device, want_full_q=full_q, block=16)
        if full_q:
            qf[off:off + n] = qb.to(dt)
            q0[off:off + n] = qb[:, :, 0].to(dt)
        else:
            q0[off:off + n] = qb.to(dt)
        k[off:off + n] = kb.to(dt)
        v[off:off + n] = vb.to(dt)
        off += n
    cu = np.zeros(len(seqs) + 1, dtype=np.int32)
    cu[1:] = np.cumsum(lens)
    return {"q0": q0, "q": qf, "k": k, "v": v,
            "cu_seqlens": torch.as_tensor(cu, device=device),
            "lens": lens, "max_seqlen": int(lens.max()) if len(lens) else 0}


def gen_decode(wl: Workload, layer: int, step: int, device, p=None):
    """Inputs of one decode step of one layer: q [B, Hq, d], k, v [B, Hkv, d]."""
    if p is None:
        p = append_prob(wl)
    g = _gen(device, derive_seed(wl.seed, 2, layer, step))
    q, k, v = _draw_tokens(wl.batch, wl, p[layer], g, device, want_full_q=True)
    dt = wl.torch_dtype
    return {"q": q.to(dt), "k": k.to(dt), "v": v.to(dt)}
