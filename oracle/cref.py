"""ctypes front end of oracle/dmc_ref.c (Algorithm 1 + attention in plain C, fp64).

TEST INFRASTRUCTURE ONLY (see the package docstring). `build()` compiles the C
file with gcc into oracle/_build/; `run_heads()` runs many independent head
instances on POSIX threads and returns numpy arrays.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dmc_ref.c")
_OUT = os.path.join(_HERE, "_build", "libdmc_ref.so")
_lib = None


class Instance(C.Structure):
    _fields_ = [
        ("d", C.c_int32), ("G", C.c_int32), ("n_prompt", C.c_int32), ("n_decode", C.c_int32),
        ("pk", C.c_void_p), ("pv", C.c_void_p), ("pq0", C.c_void_p),
        ("dk", C.c_void_p), ("dv", C.c_void_p), ("dq", C.c_void_p),
        ("cap", C.c_int32),
        ("K", C.c_void_p), ("V", C.c_void_p), ("z", C.c_void_p),
        ("pK", C.c_void_p), ("pV", C.c_void_p), ("pz", C.c_void_p),
        ("len_prompt", C.c_void_p), ("len_final", C.c_void_p), ("lens", C.c_void_p),
        ("out", C.c_void_p), ("status", C.c_int32), ("window", C.c_int32),
    ]


def build(force: bool = False) -> str:
    """Compile dmc_ref.c (plain -O2, IEEE arithmetic) if it is missing or stale."""
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    if (not force and os.path.exists(_OUT)
            and os.path.getmtime(_OUT) >= os.path.getmtime(_SRC)):
        return _OUT
    tmp = _OUT + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC,
                           "-lm", "-lpthread"])
    os.replace(tmp, _OUT)
    return _OUT


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        _lib.dmc_ref_run.argtypes = [C.POINTER(Instance)]
        _lib.dmc_ref_run_many.argtypes = [C.POINTER(Instance), C.c_int, C.c_int]
        assert _lib.dmc_ref_instance_size() == C.sizeof(Instance)
    return _lib


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _ptr(a):
    return a.ctypes.data if a is not None else None


def run_heads(heads, threads: int = 1, want_out: bool = True, want_prompt_slots: bool = True,
              window: int = 0):
    """Run independent head instances.

    heads: list of dicts with k_prompt [T,d], v_prompt [T,d], q0_prompt [T,G],
    k_dec [S,d], v_dec [S,d], q_dec [S,G,d] (float arrays; bf16 values are
    exact in float32). Returns a list of dicts with prompt_K/V/z, K/V/z,
    prompt_len, len, lens [S], out [S,G,d]."""
    keep = []
    insts = (Instance * max(1, len(heads)))()
    results = []
    for i, h in enumerate(heads):
        pk, pv, pq0 = _f32(h["k_prompt"]), _f32(h["v_prompt"]), _f32(h["q0_prompt"])
        dk, dv, dq = _f32(h["k_dec"]), _f32(h["v_dec"]), _f32(h["q_dec"])
        T = pk.shape[0]
        S = dk.shape[0]
        d = pk.shape[1] if T else dk.shape[1]
        G = dq.shape[1] if S else (pq0.shape[1] if pq0.ndim == 2 else 1)
        cap = T + S + 1
        r = {
            "K": np.zeros((cap, d)), "V": np.zeros((cap, d)), "z": np.zeros(cap),
            "prompt_K": np.zeros((cap, d)) if want_prompt_slots else None,
            "prompt_V": np.zeros((cap, d)) if want_prompt_slots else None,
            "prompt_z": np.zeros(cap) if want_prompt_slots else None,
            "lp": np.zeros(1, np.int32), "lf": np.zeros(1, np.int32),
            "lens": np.zeros(max(S, 1), np.int32),
            "out": np.zeros((max(S, 1), max(G, 1), d)) if want_out else None,
        }
        keep.append((pk, pv, pq0, dk, dv, dq))
        inst = insts[i]
        inst.d, inst.G, inst.n_prompt, inst.n_decode = d, G, T, S
        inst.window = int(window)
        inst.pk, inst.pv, inst.pq0 = _ptr(pk), _ptr(pv), _ptr(pq0)
        inst.dk, inst.dv, inst.dq = _ptr(dk), _ptr(dv), _ptr(dq)
        inst.cap = cap
        inst.K, inst.V, inst.z = _ptr(r["K"]), _ptr(r["V"]), _ptr(r["z"])
        inst.pK, inst.pV, inst.pz = _ptr(r["prompt_K"]), _ptr(r["prompt_V"]), _ptr(r["prompt_z"])
        inst.len_prompt, inst.len_final = _ptr(r["lp"]), _ptr(r["lf"])
        inst.lens, inst.out = _ptr(r["lens"]), _ptr(r["out"])
        results.append(r)
    bad = lib().dmc_ref_run_many(insts, len(heads), int(threads))
    if bad:
        raise RuntimeError(f"{bad} oracle instances failed")
    outs = []
    for h, r in zip(heads, results):
        lp, lf = int(r["lp"][0]), int(r["lf"][0])
        S = np.asarray(h["k_dec"]).shape[0]
        o = {"prompt_len": lp, "len": lf, "K": r["K"][:lf], "V": r["V"][:lf], "z": r["z"][:lf],
             "lens": r["lens"][:S]}
        if want_prompt_slots:
            o.update(prompt_K=r["prompt_K"][:lp], prompt_V=r["prompt_V"][:lp],
                     prompt_z=r["prompt_z"][:lp])
        if want_out:
            o["out"] = r["out"][:S]
        outs.append(o)
    return outs
