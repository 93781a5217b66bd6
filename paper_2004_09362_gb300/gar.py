"""Python binding of libgar (include/gar.h): argument marshalling only.

Every function has the name of the C entry point it calls.  Device memory and streams
come from PyTorch; all Allreduce work runs in the library's CUDA kernels.  If libgar.so
is missing or fails to load, importing this module raises -- there is no fallback.
"""

from __future__ import annotations

import ctypes
import os
from typing import Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libgar.so")

GAR_F32, GAR_BF16, GAR_I32 = 0, 1, 2
GAR_SUM, GAR_MAX, GAR_MIN = 0, 1, 2
GAR_STEP_FAITHFUL, GAR_FUSED, GAR_STEP_PERSISTENT = 0, 1, 2
GAR_STEPS_BO, GAR_STEPS_LO, GAR_STEPS_RING = -1, -2, -3
GAR_GROUP_CYCLIC, GAR_GROUP_XOR = 0, 1
GAR_FORM_SINGLE, GAR_FORM_BREADTH, GAR_FORM_SPLIT = 0, 1, 2
GROUPS = {"cyclic": GAR_GROUP_CYCLIC, "xor": GAR_GROUP_XOR}
GAR_MAX_P = 1024
GAR_FUSED_MAX_OPS = 4096
GAR_OK = 0

DTYPES = {"f32": GAR_F32, "bf16": GAR_BF16, "i32": GAR_I32}
OPS = {"sum": GAR_SUM, "max": GAR_MAX, "min": GAR_MIN}
MODES = {"step": GAR_STEP_FAITHFUL, "step_faithful": GAR_STEP_FAITHFUL, "fused": GAR_FUSED,
         "persistent": GAR_STEP_PERSISTENT}
ELEM_SIZE = {GAR_F32: 4, GAR_BF16: 2, GAR_I32: 4}

# Every symbol include/gar.h declares (checked by the CPU tests).
EXPORTS = (
    "gar_plan_create", "gar_plan_destroy", "gar_plan_get_info", "gar_plan_bytes",
    "gar_plan_step", "gar_plan_origin", "gar_plan_fused_program", "gar_plan_step_ops",
    "gar_plan_set_workspace", "gar_plan_compile", "gar_plan_prepare", "gar_allreduce",
    "gar_allreduce_host", "gar_allreduce_batched", "gar_last_step_bytes", "gar_strerror",
    "gar_last_error", "gar_selftest_compile", "gar_allreduce_noalloc", "gar_plan_fused_source",
    "gar_cost_model", "gar_optimal_steps", "gar_plan_status", "gar_plan_debug_barrier",
    "gar_plan_create_group",
)


class GarError(RuntimeError):
    def __init__(self, code: int, where: str, detail: str):
        super().__init__(f"{where} failed: {gar_strerror(code)} ({code}): {detail}")
        self.code = code


class gar_plan_info(ctypes.Structure):
    _fields_ = [("P", ctypes.c_int32), ("L", ctypes.c_int32), ("S", ctypes.c_int32),
                ("r", ctypes.c_int32), ("K", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("op", ctypes.c_int32), ("n_launches", ctypes.c_int32), ("n", ctypes.c_uint64),
                ("fused_combines", ctypes.c_int32), ("fused_width", ctypes.c_int32),
                ("fused_regs", ctypes.c_int32), ("fused_local_bytes", ctypes.c_int32),
                ("group", ctypes.c_int32), ("ring", ctypes.c_int32), ("fused_form", ctypes.c_int32)]


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"libgar.so not built at {_LIB_PATH}; run __graft_entry__.build()")
    lib = ctypes.CDLL(_LIB_PATH)
    vp, i32, u64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_size_t
    P_ = ctypes.POINTER
    sig = {
        "gar_plan_create": (i32, [P_(vp), i32, u64, i32, i32, i32]),
        "gar_plan_create_group": (i32, [P_(vp), i32, u64, i32, i32, i32, i32]),
        "gar_plan_destroy": (None, [vp]),
        "gar_plan_get_info": (i32, [vp, P_(gar_plan_info)]),
        "gar_plan_bytes": (i32, [vp, P_(sz), P_(u64), P_(i32)]),
        "gar_plan_step": (i32, [vp, i32, P_(i32), P_(i32), P_(ctypes.c_int32), P_(i32)]),
        "gar_plan_origin": (i32, [vp, P_(ctypes.c_int32)]),
        "gar_plan_fused_program": (i32, [vp, P_(ctypes.c_int32), P_(i32), P_(ctypes.c_int32)]),
        "gar_plan_step_ops": (i32, [vp, P_(ctypes.c_int32), P_(i32), P_(ctypes.c_int32), P_(i32)]),
        "gar_plan_set_workspace": (i32, [vp, vp, sz]),
        "gar_plan_compile": (i32, [vp, i32]),
        "gar_plan_prepare": (i32, [vp, i32]),
        "gar_allreduce": (i32, [vp, P_(vp), i32, vp]),
        "gar_allreduce_host": (i32, [vp, P_(vp), P_(vp), P_(vp), i32, vp]),
        "gar_allreduce_batched": (i32, [P_(vp), i32, vp, i32, vp]),
        "gar_last_step_bytes": (i32, [vp, P_(u64)]),
        "gar_strerror": (ctypes.c_char_p, [i32]),
        "gar_last_error": (ctypes.c_char_p, []),
        "gar_selftest_compile": (i32, []),
        "gar_allreduce_noalloc": (i32, [vp, P_(vp), vp]),
        "gar_plan_fused_source": (i32, [vp, ctypes.c_char_p, P_(sz)]),
        "gar_cost_model": (i32, [i32, i32, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                 ctypes.c_double, P_(ctypes.c_double)]),
        "gar_optimal_steps": (i32, [i32, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                    ctypes.c_double, P_(i32)]),
        "gar_plan_status": (i32, [vp]),
        "gar_plan_debug_barrier": (i32, [vp, ctypes.c_uint, ctypes.c_uint]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


def lib_path() -> str:
    return _LIB_PATH


def gar_strerror(code: int) -> str:
    return _lib.gar_strerror(int(code)).decode()


def gar_last_error() -> str:
    return (_lib.gar_last_error() or b"").decode()


def _check(code: int, where: str):
    if code != GAR_OK:
        raise GarError(code, where, gar_last_error())


def _code(v, table, what):
    if isinstance(v, str):
        if v not in table:
            raise ValueError(f"unknown {what} {v!r}")
        return table[v]
    return int(v)


class Plan:
    """Owns a gar_plan* (destroyed with the object) and, for step-faithful mode, the
    torch tensor backing its workspace."""

    def __init__(self, handle: int):
        self._h = ctypes.c_void_p(handle)
        self.workspace = None
        self._info = None

    @property
    def handle(self) -> ctypes.c_void_p:
        if not self._h:
            raise ValueError("plan destroyed")
        return self._h

    def info(self) -> dict:
        if self._info is None or self._info["fused_width"] == 0 or self._info["fused_regs"] == 0:
            self._info = gar_plan_get_info(self)
        return self._info

    def __del__(self):
        try:
            if self._h:
                _lib.gar_plan_destroy(self._h)
                self._h = ctypes.c_void_p(None)
        except Exception:
            pass


def gar_plan_create(P: int, n: int, dtype="f32", op="sum", steps=GAR_STEPS_BO) -> Plan:
    h = ctypes.c_void_p()
    _check(_lib.gar_plan_create(ctypes.byref(h), int(P), int(n), _code(dtype, DTYPES, "dtype"),
                                _code(op, OPS, "op"), int(steps)), "gar_plan_create")
    return Plan(h.value)


def gar_plan_create_group(P: int, n: int, dtype="f32", op="sum", steps=GAR_STEPS_BO,
                          group="cyclic") -> Plan:
    h = ctypes.c_void_p()
    _check(_lib.gar_plan_create_group(ctypes.byref(h), int(P), int(n), _code(dtype, DTYPES, "dtype"),
                                      _code(op, OPS, "op"), int(steps), _code(group, GROUPS, "group")),
           "gar_plan_create_group")
    return Plan(h.value)


def gar_plan_destroy(plan: Plan) -> None:
    if plan._h:
        _lib.gar_plan_destroy(plan._h)
        plan._h = ctypes.c_void_p(None)


def gar_plan_get_info(plan: Plan) -> dict:
    info = gar_plan_info()
    _check(_lib.gar_plan_get_info(plan.handle, ctypes.byref(info)), "gar_plan_get_info")
    return {f: getattr(info, f) for (f, _t) in gar_plan_info._fields_}


def gar_plan_bytes(plan: Plan):
    S = ctypes.c_int()
    ws = ctypes.c_size_t()
    _check(_lib.gar_plan_bytes(plan.handle, ctypes.byref(ws), None, ctypes.byref(S)), "gar_plan_bytes")
    per = (ctypes.c_uint64 * max(1, S.value))()
    _check(_lib.gar_plan_bytes(plan.handle, None, per, None), "gar_plan_bytes")
    return ws.value, [int(per[t]) for t in range(S.value)], S.value


def gar_plan_step(plan: Plan, t: int):
    phase, partner, count = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    P = plan.info()["P"]
    pl = (ctypes.c_int32 * P)()
    _check(_lib.gar_plan_step(plan.handle, int(t), ctypes.byref(phase), ctypes.byref(partner), pl,
                              ctypes.byref(count)), "gar_plan_step")
    return phase.value, partner.value, [int(pl[k]) for k in range(count.value)]


def gar_plan_origin(plan: Plan):
    P = plan.info()["P"]
    o = (ctypes.c_int32 * P)()
    _check(_lib.gar_plan_origin(plan.handle, o), "gar_plan_origin")
    return [int(v) for v in o]


def gar_plan_fused_program(plan: Plan):
    nops = ctypes.c_int()
    _check(_lib.gar_plan_fused_program(plan.handle, None, ctypes.byref(nops), None),
           "gar_plan_fused_program")
    K = plan.info()["K"]
    ops = (ctypes.c_int32 * max(1, 2 * nops.value))()
    outs = (ctypes.c_int32 * K)()
    _check(_lib.gar_plan_fused_program(plan.handle, ops, ctypes.byref(nops), outs),
           "gar_plan_fused_program")
    pairs = [(int(ops[2 * k]), int(ops[2 * k + 1])) for k in range(nops.value)]
    return pairs, [int(v) for v in outs]


def gar_plan_step_ops(plan: Plan):
    nops, nl = ctypes.c_int(), ctypes.c_int()
    _check(_lib.gar_plan_step_ops(plan.handle, None, ctypes.byref(nops), None, ctypes.byref(nl)),
           "gar_plan_step_ops")
    ops = (ctypes.c_int32 * max(1, 8 * nops.value))()
    part = (ctypes.c_int32 * max(1, nl.value))()
    _check(_lib.gar_plan_step_ops(plan.handle, ops, ctypes.byref(nops), part, ctypes.byref(nl)),
           "gar_plan_step_ops")
    arr = np.frombuffer(ops, dtype=np.int32, count=8 * nops.value).reshape(nops.value, 8).copy()
    return arr, [int(part[k]) for k in range(nl.value)]


def gar_plan_fused_source(plan: Plan) -> str:
    n = ctypes.c_size_t(0)
    _check(_lib.gar_plan_fused_source(plan.handle, None, ctypes.byref(n)), "gar_plan_fused_source")
    buf = ctypes.create_string_buffer(n.value)
    _check(_lib.gar_plan_fused_source(plan.handle, buf, ctypes.byref(n)), "gar_plan_fused_source")
    return buf.value.decode()


def gar_plan_set_workspace(plan: Plan, ptr: int, nbytes: int) -> None:
    _check(_lib.gar_plan_set_workspace(plan.handle, ctypes.c_void_p(int(ptr) or None), int(nbytes)),
           "gar_plan_set_workspace")


def gar_plan_compile(plan: Plan, mode="fused") -> None:
    _check(_lib.gar_plan_compile(plan.handle, _code(mode, MODES, "mode")), "gar_plan_compile")


def gar_plan_prepare(plan: Plan, mode="fused") -> None:
    _check(_lib.gar_plan_prepare(plan.handle, _code(mode, MODES, "mode")), "gar_plan_prepare")


def _stream_handle(stream) -> ctypes.c_void_p:
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    if hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    return ctypes.c_void_p(int(stream) or None)


def rank_pointer_array(rank_buffers) -> ctypes.Array:
    """The P addresses as the C array of pointers the library's calls take: from a 2-D
    tensor (rows = ranks), a list of tensors or ints, or an array this function returned
    (passed through).  Build it once and pass it to every call to skip the per-call
    marshalling (a few microseconds at P = 127)."""
    if isinstance(rank_buffers, ctypes.Array):
        return rank_buffers
    if hasattr(rank_buffers, "dim") and rank_buffers.dim() == 2:
        t = rank_buffers
        if t.stride(1) != 1:
            raise ValueError("rows must be contiguous")
        P, base, step = t.shape[0], t.data_ptr(), t.stride(0) * t.element_size()
        if P < 24:      # below about 24 ranks plain Python is faster than numpy
            return (ctypes.c_void_p * P)(*[base + x * step for x in range(P)])
        a = np.arange(P, dtype=np.uint64) * np.uint64(step) + np.uint64(base)
    elif len(rank_buffers) and isinstance(rank_buffers[0], int):
        if len(rank_buffers) < 24:
            return (ctypes.c_void_p * len(rank_buffers))(*rank_buffers)
        a = np.array(rank_buffers, dtype=np.uint64)
    else:
        a = np.array([int(b) if isinstance(b, int) else b.data_ptr() for b in rank_buffers],
                     dtype=np.uint64)
    return (ctypes.c_void_p * len(a)).from_buffer(a)    # keeps `a` alive


def _ptr_array(ptrs) -> ctypes.Array:
    return rank_pointer_array(ptrs)


def rank_pointers(rank_buffers) -> list[int]:
    """Device addresses of P rank buffers given as a list of tensors, a list of ints, or a
    2-D tensor whose rows are the ranks' vectors."""
    if hasattr(rank_buffers, "dim") and rank_buffers.dim() == 2:
        t = rank_buffers
        if t.stride(1) != 1:
            raise ValueError("rows must be contiguous")
        base, step = t.data_ptr(), t.stride(0) * t.element_size()
        return [base + x * step for x in range(t.shape[0])]
    return [int(b) if isinstance(b, int) else b.data_ptr() for b in rank_buffers]


def ensure_workspace(plan: Plan, device=None):
    """Allocates (once) the step-faithful workspace as a torch uint8 tensor and attaches
    it to the plan."""
    import torch
    ws, _per, _S = gar_plan_bytes(plan)
    if ws == 0:
        return None
    if plan.workspace is None or plan.workspace.numel() < ws:
        plan.workspace = torch.empty(ws, dtype=torch.uint8, device=device or "cuda")
        gar_plan_set_workspace(plan, plan.workspace.data_ptr(), ws)
    return plan.workspace


def gar_plan_status(plan: Plan) -> int:
    """GAR_OK, or the status code of the last persistent Allreduce (raises on CUDA errors)."""
    rc = _lib.gar_plan_status(plan.handle)
    if rc not in (GAR_OK, -8):
        _check(rc, "gar_plan_status")
    return rc


def gar_plan_debug_barrier(plan: Plan, phantom: int = 0, spin_limit: int = 0) -> None:
    _check(_lib.gar_plan_debug_barrier(plan.handle, int(phantom), int(spin_limit)),
           "gar_plan_debug_barrier")


def gar_allreduce(plan: Plan, rank_buffers, mode="fused", stream=None) -> None:
    mode_c = _code(mode, MODES, "mode")
    if mode_c in (GAR_STEP_FAITHFUL, GAR_STEP_PERSISTENT) and plan.workspace is None:
        ensure_workspace(plan)
    ptrs = rank_pointer_array(rank_buffers)
    _check(_lib.gar_allreduce(plan.handle, ptrs, mode_c, _stream_handle(stream)), "gar_allreduce")


def gar_allreduce_host(plan: Plan, host_in, host_out, dev_bufs, mode="fused", stream=None) -> None:
    mode_c = _code(mode, MODES, "mode")
    if mode_c in (GAR_STEP_FAITHFUL, GAR_STEP_PERSISTENT) and plan.workspace is None:
        ensure_workspace(plan)
    hin = rank_pointer_array(host_in)
    hout = rank_pointer_array(host_out)
    dev = rank_pointer_array(dev_bufs)
    _check(_lib.gar_allreduce_host(plan.handle, hin, hout, dev, mode_c, _stream_handle(stream)),
           "gar_allreduce_host")


BATCH_DESC = np.dtype([("plan", np.int32), ("reserved", np.int32), ("in", np.uint64),
                       ("out", np.uint64)])


def make_batch_desc(plan_index, in_ptrs, out_ptrs, device="cuda"):
    """Packs gar_batch_desc records into a device uint8 tensor."""
    import torch
    rec = np.zeros(len(plan_index), dtype=BATCH_DESC)
    rec["plan"] = np.asarray(plan_index, dtype=np.int32)
    rec["in"] = np.asarray(in_ptrs, dtype=np.uint64)
    rec["out"] = np.asarray(out_ptrs, dtype=np.uint64)
    return torch.from_numpy(rec.view(np.uint8).copy()).to(device)


def gar_allreduce_batched(plans: Sequence[Plan], desc, count: int, stream=None) -> None:
    arr = (ctypes.c_void_p * len(plans))()
    for k, p in enumerate(plans):
        arr[k] = p.handle.value
    dptr = desc if isinstance(desc, int) else desc.data_ptr()
    _check(_lib.gar_allreduce_batched(arr, len(plans), ctypes.c_void_p(dptr), int(count),
                                      _stream_handle(stream)), "gar_allreduce_batched")


def gar_allreduce_noalloc(plan: Plan, rank_buffers, stream=None) -> None:
    ptrs = rank_pointer_array(rank_buffers)
    _check(_lib.gar_allreduce_noalloc(plan.handle, ptrs, _stream_handle(stream)),
           "gar_allreduce_noalloc")


def gar_last_step_bytes(plan: Plan) -> list[int]:
    S = plan.info()["S"]
    per = (ctypes.c_uint64 * max(1, S))()
    _check(_lib.gar_last_step_bytes(plan.handle, per), "gar_last_step_bytes")
    return [int(per[t]) for t in range(S)]


def gar_cost_model(P: int, steps: int, m_bytes: float, alpha: float, beta: float,
                   gamma: float) -> float:
    t = ctypes.c_double()
    _check(_lib.gar_cost_model(int(P), int(steps), float(m_bytes), float(alpha), float(beta),
                               float(gamma), ctypes.byref(t)), "gar_cost_model")
    return t.value


def gar_optimal_steps(P: int, m_bytes: float, alpha: float, beta: float, gamma: float) -> int:
    S = ctypes.c_int()
    _check(_lib.gar_optimal_steps(int(P), float(m_bytes), float(alpha), float(beta), float(gamma),
                                  ctypes.byref(S)), "gar_optimal_steps")
    return S.value


def gar_selftest_compile() -> None:
    _check(_lib.gar_selftest_compile(), "gar_selftest_compile")
