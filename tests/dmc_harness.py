"""Helpers for the GPU parity tests: drive the CUDA path through the C ABI and
the fp64 oracle on the same seeded inputs, and compare."""
from __future__ import annotations

import numpy as np
import torch

from oracle import cref
from oracle import dmc_ref as R
from paper_2403_09636_gb300 import DmcCache, synthetic as S

TOL = {"f32": 1e-4, "bf16": 2e-2}


def expected_prompt_lengths(k0_np, cu, start=None):
    """Slot count per (sequence, head) after a prompt, from the oracle's
    decision rule: an empty head's first token opens slot 0, and every later
    token with alpha = 0 opens another."""
    B = len(cu) - 1
    H = k0_np.shape[1]
    out = np.zeros((B, H), dtype=np.int64)
    for b in range(B):
        seg = k0_np[cu[b]:cu[b + 1]]
        alpha = R.decision(seg)
        opens = (alpha == 0).astype(np.int64)
        s0 = np.zeros(H, dtype=np.int64) if start is None else np.asarray(start[b], dtype=np.int64)
        if seg.shape[0]:
            opens[0] = np.where(s0 == 0, 1, opens[0])
        out[b] = s0 + opens.sum(axis=0)
    return out


def expected_step_lengths(prev, k0_np):
    """Lengths after one decode token per head (prev [B, H], k0 [B, H])."""
    alpha = R.decision(k0_np)
    return prev + np.where((prev == 0) | (alpha == 0), 1, 0)


def cache_for(wl: S.Workload, device, max_slots=None, num_pages=None, max_prefill_tokens=None,
              window=0):
    lens = S.prompt_lengths(wl)
    if max_slots is None:
        max_slots = int(lens.max()) + wl.decode_steps + 1
    NH = wl.batch * wl.num_kv_heads
    if num_pages is None:
        num_pages = wl.num_layers * NH * ((max_slots + 31) // 32)
    if max_prefill_tokens is None:
        max_prefill_tokens = int(lens.sum())
    return DmcCache(wl.num_layers, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                    wl.torch_dtype, max_slots, num_pages, max_prefill_tokens, device=device,
                    window=window)


def exact_final_lengths(wl: S.Workload, device, steps, p=None):
    """Slot count of every (layer, seq, kv head) after its prompt and `steps`
    decode tokens, from the signs of the generated decision neurons. Used only
    to size the page pool of the large workloads exactly; the parity checks
    take their lengths from the oracle's rule."""
    if p is None:
        p = S.append_prob(wl)
    out = torch.zeros((wl.num_layers, wl.batch, wl.num_kv_heads), dtype=torch.int64)
    for layer in range(wl.num_layers):
        pr = S.gen_prompt(wl, layer, device, p=p)
        cu = pr["cu_seqlens"].to(torch.int64)
        neg = (pr["k"][:, :, 0] < 0).to(torch.int64)
        csum = torch.cat([torch.zeros_like(neg[:1]), torch.cumsum(neg, 0)])
        n = csum[cu[1:]] - csum[cu[:-1]]
        nonempty = (cu[1:] > cu[:-1])[:, None]
        first_acc = (pr["k"][cu[:-1].clamp(max=max(int(cu[-1]) - 1, 0)), :, 0] >= 0) & nonempty
        lens = n + first_acc.to(torch.int64)
        del pr, neg, csum
        for step in range(steps):
            k0 = S.gen_decode(wl, layer, step, device, p=p)["k"][:, :, 0]
            lens = lens + ((lens == 0) | (k0 < 0)).to(torch.int64)
        out[layer] = lens.cpu()
    return out


def full_size_cache(wl: S.Workload, device, steps, margin_bytes=3 << 30):
    """A cache for a full-size workload with an exactly sized page pool. If the
    device cannot hold every layer next to one layer's prompt inputs, the
    workload keeps its leading layers that fit (same per-layer shape, same
    seeds); returns (workload, cache)."""
    final = exact_final_lengths(wl, device, steps)
    torch.cuda.empty_cache()
    pages = ((final + 31) // 32).sum(dim=(1, 2)).cumsum(0)          # pages of layers [0, l]
    lens = S.prompt_lengths(wl)
    max_slots = int(final.max()) + 1
    total = int(lens.sum())
    row = wl.head_dim * wl.esize
    # one layer's prompt in the cache dtype plus one sequence's fp32 draws
    peak = total * (2 * wl.num_kv_heads * row + wl.num_q_heads * wl.esize) + \
        int(lens.max()) * (3 * wl.num_kv_heads * wl.head_dim + wl.num_q_heads) * 4
    free = torch.cuda.mem_get_info(device)[0]
    from paper_2403_09636_gb300 import dmc_cache_config, dmc_cache_required_bytes, PAGE_SIZE
    dt = 0 if wl.dtype == "f32" else 1
    layers = wl.num_layers
    while layers > 1:
        cfg = dmc_cache_config(layers, wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, dt,
                               PAGE_SIZE, max_slots, int(pages[layers - 1]) + 64, total, 0)
        if dmc_cache_required_bytes(cfg) + peak + margin_bytes <= free:
            break
        layers -= 1
    if layers < wl.num_layers:
        wl = S.shrink(wl, num_layers=layers)
    cache = cache_for(wl, device, max_slots=max_slots, num_pages=int(pages[layers - 1]) + 64,
                      max_prefill_tokens=total)
    return wl, cache


class Run:
    """Prefill + decode of a workload on the GPU, keeping host copies of the
    inputs of sampled (layer, seq, kv_head) instances and the GPU results for
    them."""

    def __init__(self, wl: S.Workload, device, samples, decode_steps=None, cache=None,
                 check_all_lengths=True, window=0, launch="stream"):
        """launch: how each decode step runs: "stream" (one dmc_decode_step per
        layer), "layers" (dmc_decode_step_layers: the layers in two launches,
        [0, L // 2) and [L // 2, L), or one when L = 1) or "graph" (the
        per-layer launches of a step captured once in a CUDA graph and
        replayed with each step's inputs copied into its static buffers)."""
        self.wl = wl
        self.launch = launch
        self.window = window
        self.samples = list(samples)
        G, d = wl.group, wl.head_dim
        steps = wl.decode_steps if decode_steps is None else decode_steps
        self.cache = cache if cache is not None else cache_for(wl, device, window=window)
        p = S.append_prob(wl)
        self.inst = {s: {"k_prompt": None, "k_dec": [], "v_dec": [], "q_dec": [], "out": []}
                     for s in self.samples}
        self.len_ok = True
        self.len_msgs = []
        layers = sorted({l for (l, _, _) in self.samples}) if not check_all_lengths else \
            list(range(wl.num_layers))
        lens_now = {}
        for layer in range(wl.num_layers):
            pr = S.gen_prompt(wl, layer, device, p=p)
            self.cache.prefill(layer, pr["q0"], pr["k"], pr["v"], pr["cu_seqlens"],
                               pr["max_seqlen"])
            cu = pr["cu_seqlens"].cpu().numpy()
            if layer in layers:
                k0 = pr["k"][:, :, 0].float().cpu().numpy()
                exp = expected_prompt_lengths(k0, cu)
                got = self.cache.lengths(layer).cpu().numpy()
                if not np.array_equal(exp, got):
                    self.len_ok = False
                    self.len_msgs.append(f"prefill layer {layer}: {np.argwhere(exp != got)[:5]}")
                lens_now[layer] = exp
            for s in self.samples:
                if s[0] != layer:
                    continue
                _, b, h = s
                sl = slice(int(cu[b]), int(cu[b + 1]))
                self.inst[s]["k_prompt"] = pr["k"][sl, h].float().cpu().numpy()
                self.inst[s]["v_prompt"] = pr["v"][sl, h].float().cpu().numpy()
                self.inst[s]["q0_prompt"] = pr["q0"][sl, h * G:(h + 1) * G].float().cpu().numpy()
            del pr
        self.prompt_export = {}
        for s in self.samples:
            layer, b, h = s
            k, v, z, ln = self.cache.export_heads(layer, [b * wl.num_kv_heads + h],
                                                  int(S.prompt_lengths(wl)[b]) + 1)
            n = int(ln[0])
            self.prompt_export[s] = (k[0, :n].float().cpu().numpy(), v[0, :n].float().cpu().numpy(),
                                     z[0, :n].cpu().numpy(), n)
        by_layer = {}
        for s in self.samples:
            by_layer.setdefault(s[0], []).append(s)
        idx = {l: (torch.tensor([b for (_, b, _) in ss], device=device),
                   torch.tensor([h for (_, _, h) in ss], device=device)) for l, ss in by_layer.items()}
        B, Hkv = wl.batch, wl.num_kv_heads
        NL = wl.num_layers
        graph = None
        if launch == "graph" and steps:
            first = [S.gen_decode(wl, layer, 0, device, p=p) for layer in range(NL)]
            g_in = [{k_: first[layer][k_].clone() for k_ in ("q", "k", "v")} for layer in range(NL)]
            g_out = [torch.empty_like(first[layer]["q"]) for layer in range(NL)]
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                for layer in range(NL):
                    x = g_in[layer]
                    self.cache.decode(layer, x["q"], x["k"], x["v"], g_out[layer])
        for step in range(steps):
            dds = [S.gen_decode(wl, layer, step, device, p=p) for layer in range(NL)]
            outs = [torch.empty_like(dd["q"]) for dd in dds]
            if launch == "stream":
                for layer, dd in enumerate(dds):
                    self.cache.decode(layer, dd["q"], dd["k"], dd["v"], outs[layer])
            elif launch == "layers":
                q = torch.stack([dd["q"] for dd in dds])
                k = torch.stack([dd["k"] for dd in dds])
                v = torch.stack([dd["v"] for dd in dds])
                o = torch.empty_like(q)
                cut = NL // 2
                for lo, hi in ((0, cut), (cut, NL)):
                    if hi > lo:
                        self.cache.decode_layers(lo, q[lo:hi], k[lo:hi], v[lo:hi], o[lo:hi])
                outs = list(o.unbind(0))
            elif launch == "graph":
                for layer, dd in enumerate(dds):
                    for k_ in ("q", "k", "v"):
                        g_in[layer][k_].copy_(dd[k_])
                graph.replay()
                outs = [x.clone() for x in g_out]
            else:
                raise ValueError(launch)
            for layer in range(NL):
                dd, out = dds[layer], outs[layer]
                if layer in lens_now:
                    exp = expected_step_lengths(lens_now[layer], dd["k"][:, :, 0].float().cpu().numpy())
                    got = self.cache.lengths(layer).cpu().numpy()
                    if not np.array_equal(exp, got):
                        self.len_ok = False
                        self.len_msgs.append(f"step {step} layer {layer}: {np.argwhere(exp != got)[:5]}")
                    lens_now[layer] = exp
                if layer not in by_layer:
                    continue
                ib, ih = idx[layer]
                kk = dd["k"][ib, ih].float().cpu().numpy()
                vv = dd["v"][ib, ih].float().cpu().numpy()
                qq = dd["q"].view(B, Hkv, G, d)[ib, ih].float().cpu().numpy()
                oo = out.view(B, Hkv, G, d)[ib, ih].float().cpu().numpy()
                for i, s in enumerate(by_layer[layer]):
                    I = self.inst[s]
                    I["k_dec"].append(kk[i])
                    I["v_dec"].append(vv[i])
                    I["q_dec"].append(qq[i])
                    I["out"].append(oo[i])
        self.final_export = {}
        for s in self.samples:
            layer, b, h = s
            cap = int(S.prompt_lengths(wl)[b]) + steps + 1
            k, v, z, ln = self.cache.export_heads(layer, [b * wl.num_kv_heads + h], cap)
            n = int(ln[0])
            self.final_export[s] = (k[0, :n].float().cpu().numpy(), v[0, :n].float().cpu().numpy(),
                                    z[0, :n].cpu().numpy(), n)
        self.status = self.cache.status()
        self.steps = steps

    def oracle(self, threads=8):
        heads = []
        d, G = self.wl.head_dim, self.wl.group
        for s in self.samples:
            I = self.inst[s]
            heads.append({
                "k_prompt": I["k_prompt"], "v_prompt": I["v_prompt"], "q0_prompt": I["q0_prompt"],
                "k_dec": np.array(I["k_dec"]).reshape(-1, d), "v_dec": np.array(I["v_dec"]).reshape(-1, d),
                "q_dec": np.array(I["q_dec"]).reshape(-1, G, d)})
        return dict(zip(self.samples, cref.run_heads(heads, threads=threads, window=self.window)))

    def compare(self, tol=None):
        """Returns a list of failure strings (empty = parity)."""
        tol = TOL[self.wl.dtype] if tol is None else tol
        bad = list(self.len_msgs)
        if self.status[0] != 0:
            bad.append(f"device status {self.status}")
        ref = self.oracle()
        for s in self.samples:
            r = ref[s]
            k, v, z, n = self.prompt_export[s]
            if n != r["prompt_len"]:
                bad.append(f"{s} prompt len {n} != {r['prompt_len']}")
            else:
                for name, a, b in (("K", k, r["prompt_K"]), ("V", v, r["prompt_V"]), ("z", z, r["prompt_z"])):
                    err = float(np.max(np.abs(a - b))) if n else 0.0
                    if not err <= tol:
                        bad.append(f"{s} prompt {name} max err {err}")
            if self.steps:
                out = np.array(self.inst[s]["out"])
                err = float(np.max(np.abs(out - r["out"])))
                if not err <= tol:
                    bad.append(f"{s} decode out max err {err}")
            k, v, z, n = self.final_export[s]
            if n != r["len"]:
                bad.append(f"{s} final len {n} != {r['len']}")
            else:
                for name, a, b in (("K", k, r["K"]), ("V", v, r["V"]), ("z", z, r["z"])):
                    err = float(np.max(np.abs(a - b)))
                    if not err <= tol:
                        bad.append(f"{s} final {name} max err {err}")
        return bad


def all_samples(wl: S.Workload):
    return [(l, b, h) for l in range(wl.num_layers) for b in range(wl.batch)
            for h in range(wl.num_kv_heads)]


def random_samples(wl: S.Workload, n, seed=0):
    rng = np.random.default_rng(seed)
    got = set()
    while len(got) < n:
        got.add((int(rng.integers(wl.num_layers)), int(rng.integers(wl.batch)),
                 int(rng.integers(wl.num_kv_heads))))
    return sorted(got)
