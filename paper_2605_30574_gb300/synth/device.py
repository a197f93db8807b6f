"""ctypes binding of the device twin of the input generator (``libsplice_synth.so``).

Fills whole device stores of a workload with the values ``host.SynthInputs``
regenerates on the CPU.  Tensors are torch uint16/int16/bfloat16 CUDA tensors
(bf16 bit patterns); fills run on torch's current stream.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import host as H
from . import workloads as W

_LIB = None


def _lib():
    global _LIB
    if _LIB is None:
        path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libsplice_synth.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is not built: run paper_2605_30574_gb300.build.build()")
        L = ctypes.CDLL(path)
        u64, i, l, f, vp = ctypes.c_uint64, ctypes.c_int, ctypes.c_long, ctypes.c_float, ctypes.c_void_p
        L.synth_normal.argtypes = [u64, i, u64, l, f, vp, vp]
        L.synth_fill_clean.argtypes = [u64, i, i, i, i, i, i, i, vp, vp, vp]
        L.synth_fill_donor.argtypes = [u64, i, i, i, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_uint32),
                                       i, i, i, i, i, i, vp, vp, vp]
        L.synth_fill_suffix.argtypes = [u64, l, i, i, i, i, i, vp, vp, vp]
        L.synth_fill_new_kv.argtypes = [u64, l, i, i, i, i, i, i, i, vp, vp, vp]
        L.synth_fill_q.argtypes = [u64, l, i, i, i, i, i, i, i, f, vp, vp]
        for fn in (L.synth_normal, L.synth_fill_clean, L.synth_fill_donor, L.synth_fill_suffix,
                   L.synth_fill_new_kv, L.synth_fill_q):
            fn.restype = ctypes.c_int
        _LIB = L
    return _LIB


def _stream():
    import torch
    return torch.cuda.current_stream().cuda_stream


def _ok(rc, what):
    if rc != 0:
        raise RuntimeError(f"{what} failed with CUDA error {rc}")


def normal(seed, stream, idx0, n, mult, out):
    _ok(_lib().synth_normal(seed, stream, idx0, n, float(np.float32(mult)), out.data_ptr(), _stream()), "synth_normal")


def fill_clean(wl: W.Workload, p0: int, k, v):
    """k, v: [Pl][N][Hkv][Tp][d] for prompts p0 .. p0 + Pl - 1."""
    Pl = k.shape[0]
    _ok(_lib().synth_fill_clean(wl.seed, p0, Pl, wl.num_prompts, wl.num_layers, wl.num_kv_heads,
                                wl.prompt_len, wl.head_dim, k.data_ptr(), v.data_ptr(), _stream()), "fill_clean")


def fill_donor(wl: W.Workload, p0: int, k, v):
    """k, v: [Pl][D_stored][N][Hkv][Tp][d] (stored = non-ZERO slots, in slot order)."""
    Pl = k.shape[0]
    n = wl.num_donor_slots
    kinds = (ctypes.c_int * n)(*wl.slot_kinds)
    thr = (ctypes.c_uint32 * n)(*[W.PERTURB_THRESHOLD_24.get(kd, 0) for kd in wl.slot_kinds])
    _ok(_lib().synth_fill_donor(wl.seed, p0, Pl, n, kinds, thr, wl.num_layers, wl.num_kv_heads, wl.prompt_len,
                                wl.head_dim, wl.scaffold_head, wl.scaffold_tail, k.data_ptr(), v.data_ptr(),
                                _stream()), "fill_donor")


def fill_suffix(wl: W.Workload, s0: int, k, v):
    """k, v: [Bl][N][Hkv][T][d] for sequences s0 .. s0 + Bl - 1 (every slot)."""
    Bl = k.shape[0]
    _ok(_lib().synth_fill_suffix(wl.seed, s0, Bl, wl.num_layers, wl.num_kv_heads, wl.max_steps, wl.head_dim,
                                 k.data_ptr(), v.data_ptr(), _stream()), "fill_suffix")


def fill_new_kv(wl: W.Workload, s0: int, layer: int, step: int, k, v):
    """k, v: [Bl][Hkv][d], the generated K/V of step ``step`` (slot step - 1)."""
    Bl = k.shape[0]
    _ok(_lib().synth_fill_new_kv(wl.seed, s0, Bl, wl.num_layers, wl.num_kv_heads, wl.max_steps, wl.head_dim,
                                 layer, step, k.data_ptr(), v.data_ptr(), _stream()), "fill_new_kv")


def fill_q(wl: W.Workload, s0: int, layer: int, step: int, q):
    """q: [Bl][Hq][d] queries of step ``step`` at ``layer``."""
    Bl = q.shape[0]
    _ok(_lib().synth_fill_q(wl.seed, s0, Bl, wl.num_layers, wl.num_q_heads, wl.max_steps, wl.head_dim, layer,
                            step, float(H.q_mult(wl.head_dim)), q.data_ptr(), _stream()), "fill_q")
