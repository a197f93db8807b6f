"""Thin ctypes binding of the C ABI in ``include/splice.h``.

Argument marshalling only: tensors (torch tensors or raw integer device
pointers) become pointers, the stream defaults to torch's current stream, and
a non-OK status raises :class:`SpliceError`.  Every step of the path runs in
``libsplice.so``; if the library is not built this module raises instead of
falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

_LIB = None
_PKG = os.path.dirname(os.path.abspath(__file__))

OK, EINVAL, ENOMEM, ECUDA, ESTATE, EDEVICE = range(6)
DONOR_ZERO, DONOR_BLANK, DONOR_SAME_ALGO, DONOR_DIFF_ALGO, DONOR_DIFF_FAMILY = range(5)
SRC_CLEAN, SRC_ZERO, SRC_DONOR0 = 0, 1, 2

# Every function the C ABI exports, with its ctypes signature.
_c_int, _c_size, _vp = ctypes.c_int, ctypes.c_size_t, ctypes.c_void_p


class SpliceError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: status {status}: {detail}")
        self.status = status


class ModelShape(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int), ("num_q_heads", ctypes.c_int),
                ("num_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("sliding_window", ctypes.c_int), ("global_every", ctypes.c_int),
                ("sm_scale", ctypes.c_float)]


class Seq(ctypes.Structure):
    _fields_ = [("prompt_id", ctypes.c_int), ("donor_slot", ctypes.c_int),
                ("L", ctypes.c_int), ("W", ctypes.c_int)]


SIGNATURES = {
    "splice_desc_create": (_c_int, [ctypes.POINTER(ModelShape), _c_int, _c_int, _c_int,
                                     ctypes.POINTER(ctypes.c_int), _c_int, ctypes.POINTER(Seq),
                                     _c_int, _vp, ctypes.POINTER(_vp)]),
    "splice_desc_create_host": (_c_int, [ctypes.POINTER(ModelShape), _c_int, _c_int, _c_int,
                                          ctypes.POINTER(ctypes.c_int), _c_int, ctypes.POINTER(Seq),
                                          _c_int, ctypes.POINTER(_vp)]),
    "splice_desc_destroy": (_c_int, [_vp]),
    "splice_workspace_bytes": (_c_size, [_vp]),
    "splice_num_stored_donor_slots": (_c_int, [_vp]),
    "suffix_kv_append": (_c_int, [_vp, _c_int, _c_int, _vp, _vp, _vp, _vp, _vp]),
    "spliced_decode_attn": (_c_int, [_vp, _c_int, _c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                     _vp, _c_size, _vp]),
    "spliced_decode_step": (_c_int, [_vp, _c_int, _c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                     _vp, _c_size, _vp]),
    "spliced_decode_attn_static": (_c_int, [_vp, _c_int, _c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                            _vp]),
    "splice_static_scratch_bytes": (_c_size, []),
    "splice_debug_source_map": (_c_int, [_vp, _c_int, _c_int, ctypes.POINTER(ctypes.c_uint8)]),
    "splice_plan_stats": (_c_int, [_vp, _c_int, _c_int, ctypes.POINTER(_c_int), ctypes.POINTER(_c_int),
                                   ctypes.POINTER(_c_int), ctypes.POINTER(_c_int)]),
    "splice_debug_pass_order": (_c_int, [_vp, _c_int]),
    "splice_delta_bytes": (ctypes.c_size_t, [_vp]),
    "splice_delta_build": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, ctypes.c_float,
                                    ctypes.POINTER(ctypes.c_float), _vp]),
    "splice_delta_clear": (_c_int, [_vp, _vp]),
    "splice_debug_plan_delta": (_c_int, [_vp, ctypes.POINTER(ctypes.c_uint8)]),
    "splice_debug_plan_rows": (_c_int, [_vp, _c_int, _c_int, ctypes.POINTER(ctypes.c_int32), _c_int,
                                        ctypes.POINTER(_c_int)]),
    "splice_check_device_error": (_c_int, [_vp]),
    "splice_debug_wait_timeout": (_c_int, [_vp, ctypes.c_uint, _vp]),
    "splice_debug_late_copy": (_c_int, [_vp, _vp, _c_size, ctypes.c_uint, _vp]),
    "splice_kernel_launches": (ctypes.c_longlong, [_vp]),
    "splice_profile_enable": (_c_int, [_vp, _c_int]),
    "splice_profile_read": (_c_int, [_vp, ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(ctypes.c_double)]),
    "splice_kernel_kind_name": (ctypes.c_char_p, [_c_int]),
    "splice_status_str": (ctypes.c_char_p, [_c_int]),
    "splice_last_error": (ctypes.c_char_p, []),
}


def lib_path() -> str:
    return os.path.join(_PKG, "libsplice.so")


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        path = lib_path()
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is not built: run paper_2605_30574_gb300.build.build() "
                               "(there is no fallback path)")
        L = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _LIB = L
    return _LIB


def _check(status: int, where: str):
    if status != OK:
        detail = lib().splice_last_error().decode(errors="replace")
        raise SpliceError(status, where, detail)


def _ptr(x):
    """Device pointer of a torch tensor (must be contiguous), an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        raise ValueError("tensors passed to the splice library must be contiguous")
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Desc:
    """Owns a ``splice_desc*``; destroyed on ``close()`` or garbage collection."""

    def __init__(self, handle: int, num_seqs: int, on_device: bool, slot_kinds=()):
        self.handle = handle
        self.num_seqs = num_seqs
        self.on_device = on_device
        self.slot_kinds = tuple(int(k) for k in slot_kinds)

    def close(self):
        if self.handle:
            h, self.handle = self.handle, None
            _check(lib().splice_desc_destroy(h), "splice_desc_destroy")

    def __del__(self):
        try:
            if self.handle:
                lib().splice_desc_destroy(self.handle)
        except Exception:
            pass


def _desc_slots(desc: Desc):
    return desc.slot_kinds


def _marshal(shape, slot_kinds, seqs):
    sh = ModelShape(**shape) if isinstance(shape, dict) else shape
    kinds = (ctypes.c_int * len(slot_kinds))(*[int(k) for k in slot_kinds])
    arr = (Seq * len(seqs))(*[Seq(int(s[0]), int(s[1]), int(s[2]), int(s[3])) for s in seqs])
    return sh, kinds, arr


def splice_desc_create(shape, num_prompts, prompt_len, slot_kinds, seqs, max_steps, stream=None) -> Desc:
    """``seqs``: iterable of (prompt_id, donor_slot, L, W)."""
    seqs = list(seqs)
    sh, kinds, arr = _marshal(shape, slot_kinds, seqs)
    out = _vp()
    _check(lib().splice_desc_create(ctypes.byref(sh), num_prompts, prompt_len, len(slot_kinds), kinds,
                                    len(seqs), arr, max_steps, _stream(stream), ctypes.byref(out)),
           "splice_desc_create")
    return Desc(out.value, len(seqs), True, slot_kinds)


def splice_desc_create_host(shape, num_prompts, prompt_len, slot_kinds, seqs, max_steps) -> Desc:
    seqs = list(seqs)
    sh, kinds, arr = _marshal(shape, slot_kinds, seqs)
    out = _vp()
    _check(lib().splice_desc_create_host(ctypes.byref(sh), num_prompts, prompt_len, len(slot_kinds), kinds,
                                         len(seqs), arr, max_steps, ctypes.byref(out)),
           "splice_desc_create_host")
    return Desc(out.value, len(seqs), False, slot_kinds)


def splice_workspace_bytes(desc: Desc) -> int:
    return int(lib().splice_workspace_bytes(desc.handle))


def splice_num_stored_donor_slots(desc: Desc) -> int:
    return int(lib().splice_num_stored_donor_slots(desc.handle))


def suffix_kv_append(desc: Desc, layer, step, k_new, v_new, k_suffix, v_suffix, stream=None):
    _check(lib().suffix_kv_append(desc.handle, layer, step, _ptr(k_new), _ptr(v_new), _ptr(k_suffix),
                                  _ptr(v_suffix), _stream(stream)), "suffix_kv_append")


def spliced_decode_attn(desc: Desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                        out, workspace, workspace_bytes=None, stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().spliced_decode_attn(desc.handle, layer, step, _ptr(q), _ptr(k_clean), _ptr(v_clean),
                                     _ptr(k_donor), _ptr(v_donor), _ptr(k_suffix), _ptr(v_suffix), _ptr(out),
                                     _ptr(workspace), workspace_bytes, _stream(stream)),
           "spliced_decode_attn")


def spliced_decode_step(desc: Desc, layer, step, q, k_new, v_new, k_clean, v_clean, k_donor, v_donor, k_suffix,
                        v_suffix, out, workspace, workspace_bytes=None, stream=None):
    """suffix_kv_append + spliced_decode_attn in one call (the append runs
    inside the generated-span pass)."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().spliced_decode_step(desc.handle, layer, step, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_clean),
                                     _ptr(v_clean), _ptr(k_donor), _ptr(v_donor), _ptr(k_suffix), _ptr(v_suffix),
                                     _ptr(out), _ptr(workspace), workspace_bytes, _stream(stream)),
           "spliced_decode_step")


def splice_static_scratch_bytes() -> int:
    """Size of the no-allocation entry point's static scratch, as the library was built."""
    return int(lib().splice_static_scratch_bytes())


def spliced_decode_attn_static(desc: Desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix,
                               v_suffix, out, stream=None):
    """spliced_decode_attn without a workspace: the library's static device
    scratch holds the partial states (for callers that cannot allocate)."""
    _check(lib().spliced_decode_attn_static(desc.handle, layer, step, _ptr(q), _ptr(k_clean), _ptr(v_clean),
                                            _ptr(k_donor), _ptr(v_donor), _ptr(k_suffix), _ptr(v_suffix),
                                            _ptr(out), _stream(stream)),
           "spliced_decode_attn_static")


def splice_debug_source_map(desc: Desc, layer, step) -> bytes:
    buf = (ctypes.c_uint8 * desc.num_seqs)()
    _check(lib().splice_debug_source_map(desc.handle, layer, step, buf), "splice_debug_source_map")
    return bytes(buf)


def splice_debug_pass_order(desc: Desc, order: int) -> None:
    """0: order of the two passes chosen per call; 1: prompt-span pass first;
    2: generated-span pass first."""
    _check(lib().splice_debug_pass_order(desc.handle, order), "splice_debug_pass_order")


def splice_plan_stats(desc: Desc, layer, step) -> dict:
    g, t, p, s = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(lib().splice_plan_stats(desc.handle, layer, step, ctypes.byref(g), ctypes.byref(t),
                                   ctypes.byref(p), ctypes.byref(s)), "splice_plan_stats")
    return {"num_groups": g.value, "num_tiles": t.value, "prompt_visible": p.value, "suffix_visible": s.value}


GROUP_DELTA = 0x100


def splice_delta_bytes(desc: Desc) -> int:
    return int(lib().splice_delta_bytes(desc.handle))


def splice_delta_build(desc: Desc, k_clean, v_clean, k_donor, v_donor, delta, max_fraction=1.0, delta_bytes=None,
                       stream=None) -> list:
    """Encodes the stored donor spans into ``delta`` (a device buffer of
    splice_delta_bytes bytes) and enters delta mode for the slots whose
    encoded fraction is at most ``max_fraction``; returns every slot's
    fraction (-1 for ZERO slots)."""
    if delta_bytes is None:
        delta_bytes = delta.numel() * delta.element_size()
    n = len(_desc_slots(desc))
    frac = (ctypes.c_float * n)()
    _check(lib().splice_delta_build(desc.handle, _ptr(k_clean), _ptr(v_clean), _ptr(k_donor), _ptr(v_donor),
                                    _ptr(delta), delta_bytes, float(max_fraction), frac, _stream(stream)),
           "splice_delta_build")
    return [float(f) for f in frac]


def splice_delta_clear(desc: Desc, stream=None):
    _check(lib().splice_delta_clear(desc.handle, _stream(stream)), "splice_delta_clear")


def splice_debug_plan_delta(desc: Desc, slot_delta):
    flags = (ctypes.c_uint8 * len(slot_delta))(*[1 if f else 0 for f in slot_delta])
    _check(lib().splice_debug_plan_delta(desc.handle, flags), "splice_debug_plan_delta")


def splice_debug_plan_rows(desc: Desc, layer, step) -> list:
    """[(tile, group source, sequence, row mask)] of the prompt-span tiles at (layer, step)."""
    n = _c_int()
    _check(lib().splice_debug_plan_rows(desc.handle, layer, step, None, 0, ctypes.byref(n)), "splice_debug_plan_rows")
    buf = (ctypes.c_int32 * (4 * max(1, n.value)))()
    _check(lib().splice_debug_plan_rows(desc.handle, layer, step, buf, n.value, ctypes.byref(n)),
           "splice_debug_plan_rows")
    return [tuple(buf[4 * i:4 * i + 4]) for i in range(n.value)]


def splice_debug_wait_timeout(desc: Desc, limit_us: int, stream=None):
    _check(lib().splice_debug_wait_timeout(desc.handle, limit_us, _stream(stream)), "splice_debug_wait_timeout")


def splice_debug_late_copy(dst, src, delay_us: int, stream=None):
    """dst <- src (same size) by a kernel that lets dependents launch at once and copies after delay_us."""
    nbytes = src.numel() * src.element_size()
    _check(lib().splice_debug_late_copy(_ptr(dst), _ptr(src), nbytes, int(delay_us), _stream(stream)),
           "splice_debug_late_copy")


def splice_check_device_error(desc: Desc):
    _check(lib().splice_check_device_error(desc.handle), "splice_check_device_error")


KERNEL_KINDS = 4


def splice_kernel_launches(desc: Desc) -> int:
    return int(lib().splice_kernel_launches(desc.handle))


def splice_profile_enable(desc: Desc, enable: bool = True):
    _check(lib().splice_profile_enable(desc.handle, 1 if enable else 0), "splice_profile_enable")


def splice_profile_read(desc: Desc) -> dict:
    """{kind name: (launches, total ms)} since the previous read."""
    n = (ctypes.c_longlong * KERNEL_KINDS)()
    ms = (ctypes.c_double * KERNEL_KINDS)()
    _check(lib().splice_profile_read(desc.handle, n, ms), "splice_profile_read")
    return {lib().splice_kernel_kind_name(k).decode(): (int(n[k]), float(ms[k])) for k in range(KERNEL_KINDS)}


def splice_status_str(status: int) -> str:
    return lib().splice_status_str(status).decode()
