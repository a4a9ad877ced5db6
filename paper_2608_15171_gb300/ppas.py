"""ctypes binding of ``libppas.so`` (the C ABI declared in ``include/ppas.h``).

Argument marshalling only: every function here forwards to the C entry point
of the same name; all computation runs in the library's CUDA kernels and its
C++ planner.  Importing this module loads the library and raises
``ImportError`` when it has not been built (there is no fallback).

Tensors are passed as ``torch.Tensor`` (device pointers via ``data_ptr()``)
and streams default to torch's current CUDA stream.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libppas.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: run paper_2608_15171_gb300.build.build() first")
_lib = ctypes.CDLL(LIB_PATH)
try:
    # the per-layer calls through the CPython module (built beside the library
    # when this Python has headers): same C entry points, ~1 us of argument
    # parsing instead of ctypes' ~12 us
    from . import _ppasfast as _fast
except ImportError:
    _fast = None

PPAS_OK = 0
PPAS_ERR_INVALID_ARG = -1
PPAS_ERR_CAPACITY = -2
PPAS_ERR_OUT_OF_BLOCKS = -3
PPAS_ERR_UNSUPPORTED = -4
PPAS_ERR_CUDA = -5
PPAS_DEVERR_TIMEOUT = 1
PPAS_DEVERR_BAD_INDEX = 2
PPAS_PAGE_TOKENS = 16
PPAS_REQ_PENDING, PPAS_REQ_WAITING, PPAS_REQ_RUNNING, PPAS_REQ_FINISHED = 0, 1, 2, 3

EXPORTED = ("ppas_sched_create", "ppas_sched_destroy", "ppas_sched_free_blocks", "ppas_plan_step",
            "ppas_kv_append", "ppas_attention_workspace_size", "ppas_attention_step",
            "ppas_status_string", "ppas_abi_version", "ppas_attention_step_noalloc",
            "ppas_debug_wait_timeout", "ppas_attention_kernel_count", "ppas_gateup_pack",
            "ppas_gateup_swiglu")
PPAS_NOALLOC_SCRATCH_BYTES = 64 * 1024 * 1024


class ppas_request(ctypes.Structure):
    _fields_ = [("arrival_us", ctypes.c_int64), ("prompt_len", ctypes.c_int32),
                ("output_len", ctypes.c_int32), ("num_computed", ctypes.c_int32),
                ("num_generated", ctypes.c_int32), ("state", ctypes.c_int32),
                ("n_blocks", ctypes.c_int32)]


_P32 = ctypes.POINTER(ctypes.c_int32)


class ppas_step(ctypes.Structure):
    _fields_ = [("cap_rows", ctypes.c_int32), ("cap_blocks_per_seq", ctypes.c_int32),
                ("cap_tokens", ctypes.c_int32), ("n_rows", ctypes.c_int32),
                ("n_decode", ctypes.c_int32), ("n_prefill", ctypes.c_int32),
                ("b_prefill", ctypes.c_int32), ("pressure", ctypes.c_int32),
                ("n_p", ctypes.c_int32), ("n_d", ctypes.c_int32),
                ("prefill_tokens", ctypes.c_int32), ("total_tokens", ctypes.c_int32),
                ("req_idx", _P32), ("q_len", _P32), ("ctx_len", _P32),
                ("block_table", _P32), ("slot_mapping", _P32)]


_c = ctypes
_lib.ppas_sched_create.argtypes = [_c.c_int32, _P32, _c.POINTER(_c.c_void_p)]
_lib.ppas_sched_create.restype = _c.c_int32
_lib.ppas_sched_destroy.argtypes = [_c.c_void_p]
_lib.ppas_sched_destroy.restype = None
_lib.ppas_sched_free_blocks.argtypes = [_c.c_void_p]
_lib.ppas_sched_free_blocks.restype = _c.c_int32
_lib.ppas_plan_step.argtypes = [_c.c_void_p, _c.POINTER(ppas_request), _c.c_int32, _c.c_int64,
                                _c.c_int32, _c.c_int32, _c.c_int32, _c.POINTER(ppas_step)]
_lib.ppas_plan_step.restype = _c.c_int32
_lib.ppas_kv_append.argtypes = [_c.c_void_p, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_void_p, _c.c_void_p,
                                _c.c_int32, _c.c_int32, _c.c_int32, _c.c_void_p, _c.c_void_p]
_lib.ppas_kv_append.restype = _c.c_int32
_lib.ppas_attention_workspace_size.argtypes = [_c.c_int32, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32]
_lib.ppas_attention_workspace_size.restype = _c.c_size_t
_lib.ppas_attention_kernel_count.argtypes = [_c.c_int32, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32,
                                              _c.c_size_t]
_lib.ppas_attention_kernel_count.restype = _c.c_int32
_lib.ppas_gateup_pack.argtypes = [_c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32, _c.c_void_p]
_lib.ppas_gateup_pack.restype = _c.c_int32
_lib.ppas_gateup_swiglu.argtypes = [_c.c_void_p, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32, _c.c_int32,
                                    _c.c_void_p, _c.c_void_p]
_lib.ppas_gateup_swiglu.restype = _c.c_int32
_lib.ppas_attention_step.argtypes = [_c.c_void_p, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_void_p,
                                     _c.c_int32, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32, _c.c_int32, _c.c_int32,
                                     _c.c_float, _c.c_void_p, _c.c_int32, _c.c_void_p, _c.c_size_t,
                                     _c.c_void_p, _c.c_void_p]
_lib.ppas_attention_step.restype = _c.c_int32
_lib.ppas_attention_step_noalloc.argtypes = [_c.c_void_p, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_void_p,
                                             _c.c_int32, _c.c_void_p, _c.c_void_p, _c.c_int32, _c.c_int32, _c.c_int32,
                                             _c.c_int32, _c.c_float, _c.c_void_p, _c.c_int32, _c.c_void_p,
                                             _c.c_void_p]
_lib.ppas_attention_step_noalloc.restype = _c.c_int32
_lib.ppas_debug_wait_timeout.argtypes = [_c.c_void_p, _c.c_uint32, _c.c_void_p]
_lib.ppas_debug_wait_timeout.restype = _c.c_int32
_lib.ppas_status_string.argtypes = [_c.c_int32]
_lib.ppas_status_string.restype = _c.c_char_p
_lib.ppas_abi_version.argtypes = []
_lib.ppas_abi_version.restype = _c.c_int32


class PpasError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {ppas_status_string(status)} ({status})")
        self.status = status


def _check(status: int, where: str) -> None:
    if status != PPAS_OK:
        raise PpasError(status, where)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _p32(a: np.ndarray):
    return a.ctypes.data_as(_P32)


def _addr(a: np.ndarray) -> int:
    """Address of an int32 array's data (the cheap route for a writable
    array; per-step calls pass small length arrays on every layer)."""
    try:
        return ctypes.addressof(ctypes.c_int32.from_buffer(a))
    except (TypeError, ValueError):  # read-only or empty
        return a.ctypes.data


def _ptr(t) -> int:
    if t is None:
        return 0
    return int(t.data_ptr()) if hasattr(t, "data_ptr") else int(t)


def _stream(stream) -> int:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    return int(getattr(stream, "cuda_stream", stream))


# ---------------------------------------------------------------- plain calls
def ppas_status_string(status: int) -> str:
    return _lib.ppas_status_string(int(status)).decode()


def ppas_abi_version() -> int:
    return int(_lib.ppas_abi_version())


def ppas_sched_create(num_blocks: int, initial_free_order=None) -> ctypes.c_void_p:
    handle = ctypes.c_void_p()
    order = None if initial_free_order is None else _i32(initial_free_order)
    if order is not None and order.size != num_blocks:
        raise PpasError(PPAS_ERR_INVALID_ARG, "ppas_sched_create")
    _check(_lib.ppas_sched_create(int(num_blocks), None if order is None else _p32(order),
                                  ctypes.byref(handle)), "ppas_sched_create")
    return handle


def ppas_sched_destroy(handle) -> None:
    _lib.ppas_sched_destroy(handle)


def ppas_sched_free_blocks(handle) -> int:
    return int(_lib.ppas_sched_free_blocks(handle))


def ppas_plan_step(handle, reqs, n_reqs: int, now_us: int, threshold: int, mbt_hi: int, mbt_lo: int,
                   step: ppas_step) -> int:
    """Raw call: ``reqs`` is a ctypes array of ``ppas_request``; returns the status."""
    return int(_lib.ppas_plan_step(handle, reqs, int(n_reqs), int(now_us), int(threshold), int(mbt_hi),
                                   int(mbt_lo), ctypes.byref(step)))


def ppas_kv_append(k_new, v_new, d_slot_mapping, n_tokens: int, k_cache, v_cache, num_blocks: int,
                   n_kv_heads: int, head_dim: int, d_err_flag=None, stream=None) -> None:
    if _fast is not None:
        _check(_fast.kv_append(_ptr(k_new), _ptr(v_new), _ptr(d_slot_mapping), int(n_tokens), _ptr(k_cache),
                               _ptr(v_cache), int(num_blocks), int(n_kv_heads), int(head_dim), _ptr(d_err_flag),
                               _stream(stream)), "ppas_kv_append")
        return
    _check(_lib.ppas_kv_append(_ptr(k_new), _ptr(v_new), _ptr(d_slot_mapping), int(n_tokens), _ptr(k_cache),
                               _ptr(v_cache), int(num_blocks), int(n_kv_heads), int(head_dim), _ptr(d_err_flag),
                               _stream(stream)), "ppas_kv_append")


def ppas_attention_workspace_size(q_lens, ctx_lens, n_q_heads: int, n_kv_heads: int) -> int:
    ql, cl = _i32(q_lens), _i32(ctx_lens)
    return int(_lib.ppas_attention_workspace_size(int(ql.size), _addr(ql), _addr(cl), int(n_q_heads),
                                                  int(n_kv_heads)))


def ppas_gateup_pack(w, w_packed, hidden: int, inter: int, stream=None) -> None:
    _check(_lib.ppas_gateup_pack(_ptr(w), _ptr(w_packed), int(hidden), int(inter), _stream(stream)),
           "ppas_gateup_pack")


def ppas_gateup_swiglu(x, w_packed, y, n_tokens: int, hidden: int, inter: int, d_err_flag=None,
                       stream=None) -> None:
    _check(_lib.ppas_gateup_swiglu(_ptr(x), _ptr(w_packed), _ptr(y), int(n_tokens), int(hidden), int(inter),
                                   _ptr(d_err_flag), _stream(stream)), "ppas_gateup_swiglu")


def ppas_attention_kernel_count(q_lens, ctx_lens, n_q_heads: int, n_kv_heads: int, workspace_bytes: int) -> int:
    ql, cl = _i32(q_lens), _i32(ctx_lens)
    n = int(_lib.ppas_attention_kernel_count(int(ql.size), _addr(ql), _addr(cl), int(n_q_heads), int(n_kv_heads),
                                             int(workspace_bytes)))
    if n < 0:
        raise PpasError(PPAS_ERR_INVALID_ARG, "ppas_attention_kernel_count")
    return n


def ppas_attention_step(q, k_cache, v_cache, num_blocks: int, d_block_tables, max_blocks_per_seq: int,
                        q_lens, ctx_lens, n_q_heads: int, n_kv_heads: int, head_dim: int, scale: float, out,
                        out_is_fp32: bool, workspace=None, workspace_bytes: int = 0, d_err_flag=None,
                        stream=None) -> None:
    ql, cl = _i32(q_lens), _i32(ctx_lens)
    if _fast is not None:
        _check(_fast.attention_step(_ptr(q), _ptr(k_cache), _ptr(v_cache), int(num_blocks), _ptr(d_block_tables),
                                    int(max_blocks_per_seq), ql, cl, int(n_q_heads), int(n_kv_heads),
                                    int(head_dim), float(scale), _ptr(out), 1 if out_is_fp32 else 0,
                                    _ptr(workspace), int(workspace_bytes), _ptr(d_err_flag), _stream(stream)),
               "ppas_attention_step")
        return
    _check(_lib.ppas_attention_step(_ptr(q), _ptr(k_cache), _ptr(v_cache), int(num_blocks),
                                    _ptr(d_block_tables), int(max_blocks_per_seq), _addr(ql), _addr(cl),
                                    int(ql.size), int(n_q_heads), int(n_kv_heads), int(head_dim),
                                    float(scale), _ptr(out), 1 if out_is_fp32 else 0, _ptr(workspace),
                                    int(workspace_bytes), _ptr(d_err_flag), _stream(stream)),
           "ppas_attention_step")


def ppas_attention_step_noalloc(q, k_cache, v_cache, num_blocks: int, d_block_tables, max_blocks_per_seq: int,
                                q_lens, ctx_lens, n_q_heads: int, n_kv_heads: int, head_dim: int, scale: float,
                                out, out_is_fp32: bool, d_err_flag=None, stream=None) -> None:
    """``ppas_attention_step`` for callers that cannot allocate device memory:
    the split-K scratch is the library's fixed array of
    ``PPAS_NOALLOC_SCRATCH_BYTES`` (shared by every call; serialise calls)."""
    ql, cl = _i32(q_lens), _i32(ctx_lens)
    _check(_lib.ppas_attention_step_noalloc(_ptr(q), _ptr(k_cache), _ptr(v_cache), int(num_blocks),
                                            _ptr(d_block_tables), int(max_blocks_per_seq), _addr(ql), _addr(cl),
                                            int(ql.size), int(n_q_heads), int(n_kv_heads), int(head_dim),
                                            float(scale), _ptr(out), 1 if out_is_fp32 else 0, _ptr(d_err_flag),
                                            _stream(stream)),
           "ppas_attention_step_noalloc")


def ppas_debug_wait_timeout(d_err_flag, limit_us: int, stream=None) -> None:
    _check(_lib.ppas_debug_wait_timeout(_ptr(d_err_flag), int(limit_us), _stream(stream)), "ppas_debug_wait_timeout")


# ---------------------------------------------------------------- planner object
class StepPlan:
    """Host copy of one ``ppas_step`` result (numpy arrays)."""

    def __init__(self, st: ppas_step, req_idx, q_len, ctx_len, table, slots):
        n = st.n_rows
        self.n_rows, self.n_decode, self.n_prefill = n, st.n_decode, st.n_prefill
        self.b_prefill, self.pressure, self.n_p, self.n_d = st.b_prefill, st.pressure, st.n_p, st.n_d
        self.prefill_tokens, self.total_tokens = st.prefill_tokens, st.total_tokens
        self.req_idx = req_idx[:n].copy()
        self.q_len = q_len[:n].copy()
        self.ctx_len = ctx_len[:n].copy()
        self.block_table = table[:n].copy()
        self.slot_mapping = slots[:st.total_tokens].copy()


class Scheduler:
    """Owns a ``ppas_sched`` handle, the request array and the plan buffers."""

    def __init__(self, num_blocks: int, free_order=None, cap_rows: int = 1024,
                 cap_blocks_per_seq: int = 4096, cap_tokens: int = 65536):
        self.handle = ppas_sched_create(num_blocks, free_order)
        self.reqs = (ppas_request * 0)()
        self.n_reqs = 0
        self._req_idx = np.zeros(cap_rows, np.int32)
        self._q_len = np.zeros(cap_rows, np.int32)
        self._ctx_len = np.zeros(cap_rows, np.int32)
        self._table = np.zeros((cap_rows, cap_blocks_per_seq), np.int32)
        self._slots = np.zeros(cap_tokens, np.int32)
        self._step = ppas_step(cap_rows=cap_rows, cap_blocks_per_seq=cap_blocks_per_seq, cap_tokens=cap_tokens,
                               req_idx=_p32(self._req_idx), q_len=_p32(self._q_len),
                               ctx_len=_p32(self._ctx_len), block_table=_p32(self._table),
                               slot_mapping=_p32(self._slots))

    def add_requests(self, specs) -> None:
        """Append requests given as (arrival_us, prompt_len, output_len) triples."""
        old = list(self.reqs[: self.n_reqs])
        specs = list(specs)
        arr = (ppas_request * (self.n_reqs + len(specs)))()
        for i, r in enumerate(old):
            arr[i] = r
        for k, (a, p, o) in enumerate(specs):
            arr[self.n_reqs + k] = ppas_request(int(a), int(p), int(o), 0, 0, PPAS_REQ_PENDING, 0)
        self.reqs, self.n_reqs = arr, self.n_reqs + len(specs)

    def plan(self, now_us: int, threshold: int = 2, mbt_hi: int = 16384, mbt_lo: int = 2048) -> StepPlan:
        _check(ppas_plan_step(self.handle, self.reqs, self.n_reqs, now_us, threshold, mbt_hi, mbt_lo, self._step),
               "ppas_plan_step")
        return StepPlan(self._step, self._req_idx, self._q_len, self._ctx_len, self._table, self._slots)

    def free_blocks(self) -> int:
        return ppas_sched_free_blocks(self.handle)

    def close(self) -> None:
        if self.handle:
            ppas_sched_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # pragma: no cover
            pass


# replay clock of the burst workload: base plus a per-prefill-token cost (us)
STEP_BASE_US = 15000
STEP_US_PER_PREFILL_TOKEN = 27


def replay(specs, num_blocks: int, free_order, threshold: int = 2, mbt_hi: int = 16384, mbt_lo: int = 2048,
           cap_blocks_per_seq: int = 4096, max_steps: int = 100000):
    """Drive ``ppas_plan_step`` over a request trace with the deterministic
    replay clock; returns ``[(now_us, StepPlan)]``."""
    sch = Scheduler(num_blocks, free_order, cap_blocks_per_seq=cap_blocks_per_seq)
    sch.add_requests(specs)
    now, out = 0, []
    try:
        for _ in range(max_steps):
            if all(sch.reqs[i].state == PPAS_REQ_FINISHED for i in range(sch.n_reqs)):
                return out
            st = sch.plan(now, threshold, mbt_hi, mbt_lo)
            if st.n_rows == 0:
                pending = [sch.reqs[i].arrival_us for i in range(sch.n_reqs)
                           if sch.reqs[i].state == PPAS_REQ_PENDING]
                if not pending:
                    raise RuntimeError("no runnable request and none pending")
                now = max(now, min(pending))
                continue
            out.append((now, st))
            now += STEP_BASE_US + STEP_US_PER_PREFILL_TOKEN * st.prefill_tokens
        raise RuntimeError("replay did not finish")
    finally:
        sch.close()
