"""Dynamic Memory Compression hot path on one GB300 (sm_103a): Python binding.

A thin ctypes layer over libdmc.so (include/dmc.h). Every function named
dmc_* forwards its arguments unchanged to the C function of the same name:
pointers are plain integers (e.g. tensor.data_ptr()), streams are raw
cudaStream_t handles (torch.cuda.current_stream().cuda_stream). All compute
runs in the library's CUDA kernels; there is no fallback of any kind, and a
missing library raises.

`DmcCache` is a convenience wrapper that owns a torch uint8 arena tensor and
turns non-OK statuses into exceptions. The synthetic input generator lives in
`paper_2403_09636_gb300.synthetic` and is imported separately.
"""
from __future__ import annotations

import ctypes as C
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdmc.so")

DMC_OK, DMC_ERR_INVALID_ARG, DMC_ERR_ARENA_TOO_SMALL = 0, 1, 2
DMC_ERR_PAGES_EXHAUSTED, DMC_ERR_CUDA, DMC_ERR_DEVICE_FAULT = 3, 4, 5
DMC_F32, DMC_BF16 = 0, 1
DMC_FAULT_PAGES_EXHAUSTED = 0x1
DMC_FAULT_SLOT_CAPACITY = 0x2
DMC_FAULT_NAN_GATE = 0x4
DMC_FAULT_BAD_SEQLENS = 0x8
DMC_FAULT_WAIT_TIMEOUT = 0x10
PAGE_SIZE = 32

EXPORTED = ("dmc_cache_required_bytes", "dmc_cache_create", "dmc_cache_destroy",
            "dmc_cache_reset", "dmc_prefill_compress", "dmc_prefill_attention", "dmc_decode_step",
            "dmc_decode_step_layers", "dmc_decode_step_static_scratch", "dmc_cache_lengths",
            "dmc_cache_export_heads", "dmc_cache_status", "dmc_status_string")


class dmc_cache_config(C.Structure):
    _fields_ = [("num_layers", C.c_int32), ("batch", C.c_int32), ("num_q_heads", C.c_int32),
                ("num_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("dtype", C.c_int32),
                ("page_size", C.c_int32), ("max_slots_per_head", C.c_int32),
                ("num_pages", C.c_int64), ("max_prefill_tokens", C.c_int32),
                ("window", C.c_int32)]


class DmcError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__(f"{what}: {dmc_status_string(status)} ({status})" if what else
                         dmc_status_string(status))


_lib = None


def lib():
    """The loaded libdmc.so. Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2403_09636_gb300.build` (nvcc, sm_103a)")
        l = C.CDLL(LIB_PATH)
        vp, i32, i64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_size_t
        cfgp = C.POINTER(dmc_cache_config)
        sig = {
            "dmc_cache_required_bytes": (sz, [cfgp]),
            "dmc_cache_create": (C.c_int, [cfgp, vp, sz, vp, C.POINTER(vp)]),
            "dmc_cache_destroy": (C.c_int, [vp]),
            "dmc_cache_reset": (C.c_int, [vp, vp]),
            "dmc_prefill_compress": (C.c_int, [vp, i32, i32, i32, vp, i64, i64, vp, vp, vp, i32,
                                               i32, vp]),
            "dmc_prefill_attention": (C.c_int, [vp, i32, i32, i32, vp, vp, vp, vp, i32, i32, vp, vp]),
            "dmc_decode_step": (C.c_int, [vp, i32, vp, vp, vp, vp, vp]),
            "dmc_decode_step_layers": (C.c_int, [vp, i32, i32, vp, vp, vp, vp, vp]),
            "dmc_decode_step_static_scratch": (C.c_int, [vp, i32, vp, vp, vp, vp, vp]),
            "dmc_cache_lengths": (C.c_int, [vp, i32, vp, vp]),
            "dmc_cache_export_heads": (C.c_int, [vp, i32, i32, vp, i32, vp, vp, vp, vp, vp]),
            "dmc_cache_status": (C.c_int, [vp, vp, C.POINTER(C.c_uint32), C.POINTER(i64)]),
            "dmc_status_string": (C.c_char_p, [C.c_int]),
        }
        for name, (res, args) in sig.items():
            f = getattr(l, name)
            f.restype, f.argtypes = res, args
        _lib = l
    return _lib


# ---------------------------------------------------------------- same-name forwarders

def dmc_cache_required_bytes(cfg: dmc_cache_config) -> int:
    return int(lib().dmc_cache_required_bytes(C.byref(cfg)))


def dmc_cache_create(cfg: dmc_cache_config, arena_ptr: int, arena_bytes: int, stream: int):
    """Returns (status, handle)."""
    h = C.c_void_p()
    st = lib().dmc_cache_create(C.byref(cfg), arena_ptr, arena_bytes, stream, C.byref(h))
    return st, h.value


def dmc_cache_destroy(handle) -> int:
    return lib().dmc_cache_destroy(handle)


def dmc_cache_reset(handle, stream: int) -> int:
    return lib().dmc_cache_reset(handle, stream)


def dmc_prefill_compress(handle, layer, first_seq, num_seqs, q_ptr, q_token_stride,
                         q_head_stride, k_ptr, v_ptr, cu_seqlens_ptr, total_tokens, max_seqlen,
                         stream) -> int:
    return lib().dmc_prefill_compress(handle, layer, first_seq, num_seqs, q_ptr, q_token_stride,
                                      q_head_stride, k_ptr, v_ptr, cu_seqlens_ptr, total_tokens,
                                      max_seqlen, stream)


def dmc_prefill_attention(handle, layer, first_seq, num_seqs, q_ptr, k_ptr, v_ptr, cu_seqlens_ptr,
                          total_tokens, max_seqlen, out_ptr, stream) -> int:
    return lib().dmc_prefill_attention(handle, layer, first_seq, num_seqs, q_ptr, k_ptr, v_ptr,
                                       cu_seqlens_ptr, total_tokens, max_seqlen, out_ptr, stream)


def dmc_decode_step(handle, layer, q_ptr, k_ptr, v_ptr, out_ptr, stream) -> int:
    return lib().dmc_decode_step(handle, layer, q_ptr, k_ptr, v_ptr, out_ptr, stream)


def dmc_decode_step_layers(handle, first_layer, num_layers, q_ptr, k_ptr, v_ptr, out_ptr,
                           stream) -> int:
    return lib().dmc_decode_step_layers(handle, first_layer, num_layers, q_ptr, k_ptr, v_ptr,
                                        out_ptr, stream)


def dmc_decode_step_static_scratch(handle, layer, q_ptr, k_ptr, v_ptr, out_ptr, stream) -> int:
    """dmc_decode_step for callers that cannot allocate device memory: its
    scratch lives in the library's static device array (see include/dmc.h)."""
    return lib().dmc_decode_step_static_scratch(handle, layer, q_ptr, k_ptr, v_ptr, out_ptr, stream)


def dmc_cache_lengths(handle, layer, out_ptr, stream) -> int:
    return lib().dmc_cache_lengths(handle, layer, out_ptr, stream)


def dmc_cache_export_heads(handle, layer, n, head_ids_ptr, cap, k_out_ptr, v_out_ptr, z_out_ptr,
                           len_out_ptr, stream) -> int:
    return lib().dmc_cache_export_heads(handle, layer, n, head_ids_ptr, cap, k_out_ptr, v_out_ptr,
                                        z_out_ptr, len_out_ptr, stream)


def dmc_cache_status(handle, stream):
    """Returns (status, fault_bits, pages_used). Synchronizes the stream."""
    bits = C.c_uint32()
    used = C.c_int64()
    st = lib().dmc_cache_status(handle, stream, C.byref(bits), C.byref(used))
    return st, int(bits.value), int(used.value)


def dmc_status_string(status: int) -> str:
    return lib().dmc_status_string(int(status)).decode()


def _check(st: int, what: str):
    if st != DMC_OK:
        raise DmcError(st, what)


# ---------------------------------------------------------------- convenience wrapper

class DmcCache:
    """A cache living in a torch-allocated device arena. Tensors passed to the
    methods must be contiguous, on the cache's device, in the cache dtype."""

    def __init__(self, num_layers, batch, num_q_heads, num_kv_heads, head_dim, dtype,
                 max_slots_per_head, num_pages, max_prefill_tokens=0, device=None, stream=None,
                 window=0):
        import torch
        self.torch = torch
        self.device = torch.device(device if device is not None else "cuda")
        tdt = {torch.float32: DMC_F32, torch.bfloat16: DMC_BF16}[dtype]
        self.dtype = dtype
        self.cfg = dmc_cache_config(num_layers, batch, num_q_heads, num_kv_heads, head_dim, tdt,
                                    PAGE_SIZE, max_slots_per_head, int(num_pages),
                                    int(max_prefill_tokens), int(window))
        self.nbytes = dmc_cache_required_bytes(self.cfg)
        if self.nbytes == 0:
            raise DmcError(DMC_ERR_INVALID_ARG, "dmc_cache_required_bytes")
        self.arena = torch.empty(self.nbytes, dtype=torch.uint8, device=self.device)
        st, self.handle = dmc_cache_create(self.cfg, self.arena.data_ptr(), self.nbytes,
                                           self._s(stream))
        _check(st, "dmc_cache_create")

    def _s(self, stream):
        if stream is None:
            stream = self.torch.cuda.current_stream(self.device)
        return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)

    def close(self):
        if getattr(self, "handle", None):
            dmc_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reset(self, stream=None):
        _check(dmc_cache_reset(self.handle, self._s(stream)), "dmc_cache_reset")

    def prefill(self, layer, q0, k, v, cu_seqlens, max_seqlen, first_seq=0, stream=None):
        """q0: [total, Hq] (or any tensor whose element (t, j, 0) sits at
        t*stride(0) + j*stride(1)); k, v: [total, Hkv, D]; cu_seqlens int32."""
        n = cu_seqlens.numel() - 1
        total = k.shape[0]
        _check(dmc_prefill_compress(self.handle, layer, first_seq, n, q0.data_ptr(),
                                    q0.stride(0), q0.stride(1), k.data_ptr(), v.data_ptr(),
                                    cu_seqlens.data_ptr(), total, int(max_seqlen),
                                    self._s(stream)), "dmc_prefill_compress")

    def prefill_attention(self, layer, q, k, v, cu_seqlens, max_seqlen, out, first_seq=0,
                          stream=None):
        """q, out: [total, Hq, D]; k, v: [total, Hkv, D]; cu_seqlens int32."""
        n = cu_seqlens.numel() - 1
        _check(dmc_prefill_attention(self.handle, layer, first_seq, n, q.data_ptr(), k.data_ptr(),
                                     v.data_ptr(), cu_seqlens.data_ptr(), k.shape[0],
                                     int(max_seqlen), out.data_ptr(), self._s(stream)),
               "dmc_prefill_attention")

    def decode(self, layer, q, k, v, out, stream=None):
        _check(dmc_decode_step(self.handle, layer, q.data_ptr(), k.data_ptr(), v.data_ptr(),
                               out.data_ptr(), self._s(stream)), "dmc_decode_step")

    def decode_layers(self, first_layer, q, k, v, out, stream=None):
        """q, out: [n, B, Hq, D]; k, v: [n, B, Hkv, D] for layers first_layer .. + n - 1."""
        _check(dmc_decode_step_layers(self.handle, first_layer, q.shape[0], q.data_ptr(),
                                      k.data_ptr(), v.data_ptr(), out.data_ptr(), self._s(stream)),
               "dmc_decode_step_layers")

    def lengths(self, layer, stream=None):
        t = self.torch
        out = t.empty((self.cfg.batch, self.cfg.num_kv_heads), dtype=t.int32, device=self.device)
        _check(dmc_cache_lengths(self.handle, layer, out.data_ptr(), self._s(stream)),
               "dmc_cache_lengths")
        return out

    def export_heads(self, layer, head_ids, cap, stream=None):
        t = self.torch
        ids = t.as_tensor(head_ids, dtype=t.int32, device=self.device)
        n = ids.numel()
        D = self.cfg.head_dim
        k = t.zeros((n, cap, D), dtype=self.dtype, device=self.device)
        v = t.zeros((n, cap, D), dtype=self.dtype, device=self.device)
        z = t.zeros((n, cap), dtype=t.float32, device=self.device)
        ln = t.zeros(n, dtype=t.int32, device=self.device)
        _check(dmc_cache_export_heads(self.handle, layer, n, ids.data_ptr(), cap, k.data_ptr(),
                                      v.data_ptr(), z.data_ptr(), ln.data_ptr(), self._s(stream)),
               "dmc_cache_export_heads")
        return k, v, z, ln

    def status(self, stream=None):
        """(status, fault bits, pages used); synchronizes the stream."""
        return dmc_cache_status(self.handle, self._s(stream))
