"""Thin Python binding of libbsm (include/bsm.h).

Argument marshalling only: every step of the softmax and of the scheduling
runs inside libbsm.  Device buffers are passed as integers (device
addresses) or as torch tensors (their data_ptr()); host arrays as numpy
arrays.  Every call raises BsmError on a non-zero status.  If libbsm.so has
not been built, loading fails loudly: there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Sequence

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "_lib", "libbsm.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "bsm.h")

F32, BF16 = 0, 1
POLICY_WHOLE_GPU, POLICY_RR, POLICY_CBMF, POLICY_CBMF_LB, POLICY_DYNAMIC, POLICY_MINIMAX = range(6)
POLICIES = {"whole_gpu": POLICY_WHOLE_GPU, "rr": POLICY_RR, "cbmf": POLICY_CBMF,
            "cbmf_lb": POLICY_CBMF_LB, "dynamic": POLICY_DYNAMIC, "minimax": POLICY_MINIMAX}
POLICY_NAMES = {v: k for k, v in POLICIES.items()}
FLAG_CAUSAL = 1
OP_FORWARD, OP_BACKWARD = 0, 1
MAX_DIES = 4
MAX_SM = 256
DEV_BOUNDS, DEV_TIMEOUT, DEV_CHECK = 1, 2, 4

(OK, ERR_INVALID_ARG, ERR_MISALIGNED, ERR_UNSUPPORTED, ERR_CUDA, ERR_DEVICE_BOUNDS,
 ERR_TIMEOUT, ERR_NO_DEVICE, ERR_NOMEM, ERR_TOO_LARGE) = range(10)
NOALLOC_MAX_PATCHES = 65536
NOALLOC_MAX_ROW_BYTES = 115712      # 113 KiB: rows of bsm_softmax_noalloc fit one stage

c_i64p = ctypes.POINTER(ctypes.c_int64)
c_i32p = ctypes.POINTER(ctypes.c_int32)


class BsmError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = "%s: %s (status %d)" % (where, status_string(status), status)
        if status == ERR_CUDA:
            msg += " [%s]" % bsm_last_cuda_error()
        super().__init__(msg)


class PlanDesc(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("y", ctypes.c_void_p), ("num_slices", ctypes.c_int64),
                ("offsets", c_i64p), ("rows", c_i32p), ("cols", c_i32p),
                ("dtype", ctypes.c_int32), ("policy", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("rows_per_item", ctypes.c_int32), ("tie_seed", ctypes.c_uint64),
                ("lb_weighted", ctypes.c_int32), ("count_output_bytes", ctypes.c_int32),
                ("device", ctypes.c_int32), ("op", ctypes.c_int32), ("x2", ctypes.c_void_p)]


class Patch(ctypes.Structure):
    _fields_ = [("elem_offset", ctypes.c_int64), ("cols", ctypes.c_int32), ("nrows", ctypes.c_int32),
                ("row0", ctypes.c_int32), ("slice_rows", ctypes.c_int32), ("col0", ctypes.c_int32),
                ("part_count", ctypes.c_int32)]


class Layout(ctypes.Structure):
    _fields_ = [("stage_bytes", ctypes.c_int64), ("n_stages", ctypes.c_int32), ("group_k", ctypes.c_int32),
                ("n_patches", ctypes.c_int64), ("n_patches_phase1", ctypes.c_int64),
                ("long_rows", ctypes.c_int64)]


class PlanStats(ctypes.Structure):
    _fields_ = [("policy", ctypes.c_int32), ("n_die", ctypes.c_int32), ("n_items", ctypes.c_int64),
                ("N", ctypes.c_int64 * MAX_DIES), ("L", ctypes.c_int64 * MAX_DIES),
                ("overlap_items", ctypes.c_int64), ("tie_items", ctypes.c_int64),
                ("moved_items", ctypes.c_int64), ("queue_items", ctypes.c_int64 * MAX_DIES),
                ("queue_bytes", ctypes.c_int64 * MAX_DIES),
                ("est_finish_before", ctypes.c_double * MAX_DIES),
                ("est_finish_after", ctypes.c_double * MAX_DIES),
                ("stage_bytes", ctypes.c_int32), ("n_stages", ctypes.c_int32),
                ("grid", ctypes.c_int32), ("launches", ctypes.c_int32), ("steal", ctypes.c_int32),
                ("map_chunk_bytes", ctypes.c_int64), ("plan_ms", ctypes.c_double),
                ("long_items", ctypes.c_int64), ("group_rows", ctypes.c_int64),
                ("group_k", ctypes.c_int32), ("n_groups", ctypes.c_int32)]


class PlanSchedule(ctypes.Structure):
    _fields_ = [("n_queues", ctypes.c_int32), ("count_output_bytes", ctypes.c_int32),
                ("queue_begin", ctypes.c_int32 * MAX_DIES), ("queue_len", ctypes.c_int32 * MAX_DIES),
                ("units", ctypes.c_int32 * MAX_DIES), ("l_near", ctypes.c_int64),
                ("l_far", ctypes.c_int64), ("tie_seed", ctypes.c_uint64), ("n_items", ctypes.c_int64),
                ("map_chunk_bytes", ctypes.c_int64), ("n_map_chunks", ctypes.c_int64),
                ("n_moved", ctypes.c_int64), ("queue", c_i32p),
                ("x_map", ctypes.POINTER(ctypes.c_int8)), ("y_map", ctypes.POINTER(ctypes.c_int8)),
                ("moved", c_i32p)]


class Topology(ctypes.Structure):
    _fields_ = [("device", ctypes.c_int32), ("n_sm", ctypes.c_int32), ("n_die", ctypes.c_int32),
                ("separable", ctypes.c_int32), ("sm_die", ctypes.c_int8 * MAX_SM),
                ("sm_per_die", ctypes.c_int32 * MAX_DIES), ("l_near", ctypes.c_double),
                ("l_far", ctypes.c_double), ("separation", ctypes.c_double),
                ("granularity", ctypes.c_int64), ("probe_ms", ctypes.c_double)]


class ScheduleDesc(ctypes.Structure):
    _fields_ = [("n_banks", ctypes.c_int32), ("n_patches", ctypes.c_int64),
                ("patch_begin", c_i64p), ("patch_end", c_i64p), ("n_maps", ctypes.c_int32),
                ("chunk", ctypes.c_int64 * 2), ("n_chunks", ctypes.c_int64 * 2),
                ("bank_of_chunk", ctypes.POINTER(ctypes.c_int8) * 2),
                ("tie_seed", ctypes.c_uint64), ("balance", ctypes.c_int32), ("units", c_i32p),
                ("l_near", ctypes.c_int64), ("l_far", ctypes.c_int64), ("cost", c_i64p),
                ("method", ctypes.c_int32)]


class ScheduleOut(ctypes.Structure):
    _fields_ = [("bytes_on_bank", c_i64p), ("overlap", ctypes.POINTER(ctypes.c_uint8)),
                ("N", c_i64p), ("bank", c_i32p), ("L", c_i64p), ("queue_items", c_i32p),
                ("queue_len", c_i64p), ("moved", c_i32p), ("n_moved", ctypes.c_int64),
                ("work_before", c_i64p), ("work_after", c_i64p)]


_lib = None


def lib():
    """Load libbsm.so; raises if it was not built (run __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError("libbsm.so not found at %s: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`" % LIB_PATH)
    L = ctypes.CDLL(LIB_PATH)
    vp, i64, i32, u32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint32
    sig = {
        "bsm_softmax": ([vp, vp, i64, i64, i64, ctypes.c_int, ctypes.c_int, vp], ctypes.c_int),
        "bsm_softmax_ex": ([vp, vp, i64, i64, i64, ctypes.c_int, ctypes.c_int, u32, vp], ctypes.c_int),
        "bsm_softmax_ragged": ([vp, vp, i64, c_i64p, c_i32p, c_i32p, ctypes.c_int, ctypes.c_int, u32,
                                vp], ctypes.c_int),
        "bsm_softmax_noalloc": ([vp, vp, i64, i64, i64, ctypes.c_int, u32, vp], ctypes.c_int),
        "bsm_softmax_host": ([vp, vp, i64, i64, i64, ctypes.c_int, ctypes.c_int, u32, vp], ctypes.c_int),
        "bsm_bmm": ([vp, vp, vp, i64, i64, i64, i64, ctypes.c_int, ctypes.c_int, vp], ctypes.c_int),
        "bsm_bmm_ex": ([vp, vp, vp, i64, i64, i64, i64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                        ctypes.c_int, ctypes.c_int, vp], ctypes.c_int),
        "bsm_softmax_backward": ([vp, vp, vp, i64, i64, i64, ctypes.c_int, ctypes.c_int, vp], ctypes.c_int),
        "bsm_softmax_backward_ragged": ([vp, vp, vp, i64, c_i64p, c_i32p, c_i32p, ctypes.c_int,
                                         ctypes.c_int, vp], ctypes.c_int),
        "bsm_plan_desc_init": ([ctypes.POINTER(PlanDesc)], ctypes.c_int),
        "bsm_plan_create": ([ctypes.POINTER(vp), ctypes.POINTER(PlanDesc)], ctypes.c_int),
        "bsm_plan_execute": ([vp, vp], ctypes.c_int),
        "bsm_plan_get_stats": ([vp, ctypes.POINTER(PlanStats)], ctypes.c_int),
        "bsm_plan_destroy": ([vp], None),
        "bsm_plan_debug": ([vp, ctypes.c_int, i64], ctypes.c_int),
        "bsm_plan_get_schedule": ([vp, ctypes.POINTER(PlanSchedule)], ctypes.c_int),
        "bsm_plan_device_table": ([vp, ctypes.c_int, ctypes.POINTER(Patch), i64, ctypes.POINTER(i64)],
                                  ctypes.c_int),
        "bsm_die_check_read": ([ctypes.c_int, vp, i64, i64, ctypes.POINTER(ctypes.c_int8),
                                ctypes.POINTER(ctypes.c_int8), ctypes.c_int, ctypes.POINTER(u32),
                                ctypes.POINTER(ctypes.c_float)], ctypes.c_int),
        "bsm_addr_group_map": ([ctypes.c_int, vp, i64, i64, ctypes.POINTER(ctypes.c_int8),
                                ctypes.POINTER(ctypes.c_int8)], ctypes.c_int),
        "bsm_plan_layout_host": ([ctypes.POINTER(PlanDesc), i32, i64, ctypes.POINTER(Patch), i64,
                                  ctypes.POINTER(Patch), i64, ctypes.POINTER(Layout)], ctypes.c_int),
        "bsm_cache_clear": ([], None),
        "bsm_topology_probe": ([ctypes.c_int, ctypes.c_int, ctypes.POINTER(Topology)], ctypes.c_int),
        "bsm_addr_die_map": ([ctypes.c_int, vp, i64, i64, ctypes.POINTER(ctypes.c_int8)], ctypes.c_int),
        "bsm_probe_latency": ([ctypes.c_int, i32, c_i64p, i32, ctypes.POINTER(ctypes.c_float), c_i32p],
                              ctypes.c_int),
        "bsm_schedule_host": ([ctypes.POINTER(ScheduleDesc), ctypes.POINTER(ScheduleOut)], ctypes.c_int),
        "bsm_device_status": ([ctypes.c_int, ctypes.POINTER(u32)], ctypes.c_int),
        "bsm_device_status_clear": ([ctypes.c_int], ctypes.c_int),
        "bsm_max_row_bytes": ([ctypes.c_int], i64),
        "bsm_ragged_extent": ([i64, c_i64p, c_i32p, c_i32p], i64),
        "bsm_status_string": ([ctypes.c_int], ctypes.c_char_p),
        "bsm_version": ([], ctypes.c_int),
        "bsm_device_debug": ([ctypes.c_int, ctypes.POINTER(ctypes.c_uint32)], ctypes.c_int),
        "bsm_set_device_checks": ([ctypes.c_int], None),
        "bsm_last_cuda_error": ([], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _lib = L
    return L


def header_functions() -> list:
    """Names of the functions include/bsm.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(bsm_[a-z_0-9]+)\s*\(",
                                 text, flags=re.M)))


def status_string(status: int) -> str:
    return lib().bsm_status_string(status).decode()


def _check(rc: int, where: str):
    if rc != OK:
        raise BsmError(rc, where)


def _dptr(t, nbytes: Optional[int] = None, what: str = "buffer") -> Optional[int]:
    """Device address of a torch tensor, or an int passed through unchecked.
    A tensor must live on a CUDA device, be contiguous and (when nbytes is
    given) hold at least nbytes: the C ABI sees only the address, so these are
    checked here, before any launch."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not getattr(t, "is_cuda", True):
        raise ValueError("%s must be a CUDA tensor (got one on %s)" % (what, t.device))
    if hasattr(t, "is_contiguous") and not t.is_contiguous():
        raise ValueError("%s must be contiguous" % what)
    if nbytes is not None and hasattr(t, "numel") and t.numel() * t.element_size() < nbytes:
        raise ValueError("%s holds %d bytes, the call needs %d"
                         % (what, t.numel() * t.element_size(), nbytes))
    return int(t.data_ptr())


def _esize(dtype: int) -> int:
    return 4 if dtype == F32 else 2


def _bmm_bytes(B: int, M: int, N: int, K: int, out_dtype: int):
    """Bytes of a, bt and c for a batched product (bf16 operands)."""
    if min(B, M, N, K) <= 0:
        return 0, 0, 0
    return B * M * K * 2, B * N * K * 2, B * M * N * _esize(out_dtype)


def _extent(offsets, rows, cols) -> int:
    """Elements a ragged batch spans (the end of its furthest non-empty slice),
    computed by the library's host helper: microseconds even on tens of
    thousands of slices.  offsets/rows/cols: contiguous int64/int32/int32."""
    n = len(offsets)
    e = int(lib().bsm_ragged_extent(n, offsets.ctypes.data_as(c_i64p), rows.ctypes.data_as(c_i32p),
                                    cols.ctypes.data_as(c_i32p)))
    if e < 0:
        raise ValueError("ragged batch: negative offset or column count")
    return e


def _stream(s) -> Optional[int]:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


def _np(a, dt):
    return np.ascontiguousarray(np.asarray(a), dtype=dt)


def bsm_softmax(x, y, B: int, R: int, C: int, dtype: int, policy: int, stream=None):
    n = max(B * R * C, 0) * _esize(dtype)
    _check(lib().bsm_softmax(_dptr(x, n, "x"), _dptr(y, n, "y"), B, R, C, dtype, policy,
                             _stream(stream)), "bsm_softmax")


def bsm_softmax_ex(x, y, B: int, R: int, C: int, dtype: int, policy: int, flags: int = 0,
                   stream=None):
    n = max(B * R * C, 0) * _esize(dtype)
    _check(lib().bsm_softmax_ex(_dptr(x, n, "x"), _dptr(y, n, "y"), B, R, C, dtype, policy, flags,
                                _stream(stream)), "bsm_softmax_ex")


def bsm_softmax_host(x_host, y_host, B: int, R: int, C: int, dtype: int, policy: int,
                     flags: int = 0, stream=None):
    """Softmax of host buffers (pinned torch CPU tensors, numpy arrays or host
    addresses); copies in, computes and copies out in overlapping chunks."""
    def hptr(a):
        if isinstance(a, int):
            return a
        if isinstance(a, np.ndarray):
            return a.ctypes.data
        return int(a.data_ptr())
    _check(lib().bsm_softmax_host(hptr(x_host), hptr(y_host), B, R, C, dtype, policy, flags,
                                  _stream(stream)), "bsm_softmax_host")


def bsm_softmax_noalloc(x, y, B: int, R: int, C: int, dtype: int, flags: int = 0, stream=None):
    """The allocation-free entry point (fixed scratch inside the library)."""
    n = max(B * R * C, 0) * _esize(dtype)
    _check(lib().bsm_softmax_noalloc(_dptr(x, n, "x"), _dptr(y, n, "y"), B, R, C, dtype, flags,
                                     _stream(stream)), "bsm_softmax_noalloc")


def bsm_bmm(a, bt, c, B: int, M: int, N: int, K: int, out_dtype: int, policy: int, stream=None):
    """C_s = A_s Bt_s^T for every slice (bf16 inputs, fp32 or bf16 output)."""
    na, nb, nc = _bmm_bytes(B, M, N, K, out_dtype)
    _check(lib().bsm_bmm(_dptr(a, na, "a"), _dptr(bt, nb, "bt"), _dptr(c, nc, "c"), B, M, N, K,
                         out_dtype, policy, _stream(stream)), "bsm_bmm")


def bsm_bmm_ex(a, bt, c, B: int, M: int, N: int, K: int, out_dtype: int, policy: int,
               n_stages: int = 0, epi_bufs: int = 0, k_blocks_per_stage: int = 0, stream=None):
    """bsm_bmm with the shared-memory split (stages, store buffers, K blocks
    per stage) chosen."""
    na, nb, nc = _bmm_bytes(B, M, N, K, out_dtype)
    _check(lib().bsm_bmm_ex(_dptr(a, na, "a"), _dptr(bt, nb, "bt"), _dptr(c, nc, "c"), B, M, N, K,
                            out_dtype, policy, n_stages, epi_bufs, k_blocks_per_stage,
                            _stream(stream)), "bsm_bmm_ex")


def bsm_softmax_backward(y, dy, dx, B: int, R: int, C: int, dtype: int, policy: int, stream=None):
    n = max(B * R * C, 0) * _esize(dtype)
    _check(lib().bsm_softmax_backward(_dptr(y, n, "y"), _dptr(dy, n, "dy"), _dptr(dx, n, "dx"),
                                      B, R, C, dtype, policy, _stream(stream)),
           "bsm_softmax_backward")


def bsm_softmax_backward_ragged(y, dy, dx, offsets, rows, cols, dtype: int, policy: int,
                                stream=None):
    off = _np(offsets, np.int64)
    r = _np(rows, np.int32)
    c = _np(cols, np.int32)
    if not (len(off) == len(r) == len(c)):
        raise ValueError("offsets, rows and cols must have the same length")
    n = _extent(off, r, c) * _esize(dtype)
    _check(lib().bsm_softmax_backward_ragged(_dptr(y, n, "y"), _dptr(dy, n, "dy"), _dptr(dx, n, "dx"),
                                             len(off),
                                             off.ctypes.data_as(c_i64p), r.ctypes.data_as(c_i32p),
                                             c.ctypes.data_as(c_i32p), dtype, policy,
                                             _stream(stream)), "bsm_softmax_backward_ragged")


def bsm_softmax_ragged(x, y, offsets, rows, cols, dtype: int, policy: int, flags: int = 0,
                       stream=None):
    off = _np(offsets, np.int64)
    r = _np(rows, np.int32)
    c = _np(cols, np.int32)
    if not (len(off) == len(r) == len(c)):
        raise ValueError("offsets, rows and cols must have the same length")
    n = _extent(off, r, c) * _esize(dtype)
    _check(lib().bsm_softmax_ragged(_dptr(x, n, "x"), _dptr(y, n, "y"), len(off),
                                    off.ctypes.data_as(c_i64p), r.ctypes.data_as(c_i32p),
                                    c.ctypes.data_as(c_i32p), dtype, policy, flags,
                                    _stream(stream)), "bsm_softmax_ragged")


class Plan:
    """Owner of a bsm_plan; destroyed with the object."""

    def __init__(self, handle: int, keep):
        self.handle = handle
        self._keep = keep

    def execute(self, stream=None):
        bsm_plan_execute(self, stream)

    def stats(self) -> dict:
        return bsm_plan_get_stats(self)

    def close(self):
        if self.handle:
            lib().bsm_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def bsm_plan_create(x, y, rows, cols, dtype: int, policy: int, offsets=None, flags: int = 0,
                    rows_per_item: int = 0, tie_seed: Optional[int] = None,
                    lb_weighted: bool = True, count_output_bytes: bool = True,
                    device: int = -1, op: int = 0, x2=None) -> Plan:
    d = PlanDesc()
    _check(lib().bsm_plan_desc_init(ctypes.byref(d)), "bsm_plan_desc_init")
    r = _np(rows, np.int32)
    c = _np(cols, np.int32)
    off = None if offsets is None else _np(offsets, np.int64)
    if off is None:
        n = int(np.sum(r.astype(np.int64) * c.astype(np.int64))) * _esize(dtype)
    else:
        n = _extent(off, r, c) * _esize(dtype)
    d.x = _dptr(x, n, "x")
    d.y = _dptr(y, n, "y")
    d.num_slices = len(r)
    d.rows = r.ctypes.data_as(c_i32p)
    d.cols = c.ctypes.data_as(c_i32p)
    if off is not None:
        d.offsets = off.ctypes.data_as(c_i64p)
    d.dtype = dtype
    d.policy = policy
    d.flags = flags
    d.rows_per_item = rows_per_item
    if tie_seed is not None:
        d.tie_seed = tie_seed
    d.lb_weighted = 1 if lb_weighted else 0
    d.count_output_bytes = 1 if count_output_bytes else 0
    d.device = device
    d.op = op
    d.x2 = _dptr(x2, n, "x2")
    h = ctypes.c_void_p()
    _check(lib().bsm_plan_create(ctypes.byref(h), ctypes.byref(d)), "bsm_plan_create")
    return Plan(h.value, (x, y, x2))


def bsm_plan_execute(plan: Plan, stream=None):
    _check(lib().bsm_plan_execute(plan.handle, _stream(stream)), "bsm_plan_execute")


def bsm_plan_get_stats(plan: Plan) -> dict:
    s = PlanStats()
    _check(lib().bsm_plan_get_stats(plan.handle, ctypes.byref(s)), "bsm_plan_get_stats")
    out = {}
    for name, _ in PlanStats._fields_:
        v = getattr(s, name)
        out[name] = list(v) if not isinstance(v, (int, float)) else v
    return out


def _patch_array(buf, n):
    dt = np.dtype([(name, np.int64 if ct is ctypes.c_int64 else np.int32) for name, ct in Patch._fields_])
    return np.frombuffer(bytes(buf), dtype=dt, count=n) if n else np.zeros(0, dt)


def bsm_plan_get_schedule(plan: Plan) -> dict:
    """The schedule a plan was built with: queue slots (phase-0 patch index
    in slice order), the probed address -> die maps, moved patches and the
    planner's inputs (see include/bsm.h)."""
    sc = PlanSchedule()
    _check(lib().bsm_plan_get_schedule(plan.handle, ctypes.byref(sc)), "bsm_plan_get_schedule")
    q = np.zeros(max(sc.n_items, 1), np.int32)
    xm = np.zeros(max(sc.n_map_chunks, 1), np.int8)
    ym = np.full(max(sc.n_map_chunks, 1), -1, np.int8)
    mv = np.zeros(max(sc.n_moved, 1), np.int32)
    sc.queue = q.ctypes.data_as(c_i32p)
    sc.x_map = xm.ctypes.data_as(ctypes.POINTER(ctypes.c_int8))
    sc.y_map = ym.ctypes.data_as(ctypes.POINTER(ctypes.c_int8))
    sc.moved = mv.ctypes.data_as(c_i32p)
    _check(lib().bsm_plan_get_schedule(plan.handle, ctypes.byref(sc)), "bsm_plan_get_schedule")
    n, nm = sc.n_items, sc.n_map_chunks
    return {"n_queues": sc.n_queues, "count_output_bytes": sc.count_output_bytes,
            "queue_begin": list(sc.queue_begin), "queue_len": list(sc.queue_len),
            "units": list(sc.units), "l_near": sc.l_near, "l_far": sc.l_far,
            "tie_seed": sc.tie_seed, "n_items": n, "map_chunk_bytes": sc.map_chunk_bytes,
            "queue": q[:n] if sc.n_queues else None,
            "x_map": xm[:nm], "y_map": ym[:nm] if nm and ym[0] >= 0 else None,
            "moved": mv[:sc.n_moved]}


def bsm_plan_device_table(plan: Plan, phase: int = 0) -> np.ndarray:
    """The plan's device patch table as the kernel reads it (structured
    array with the fields of bsm_patch)."""
    n = ctypes.c_int64()
    _check(lib().bsm_plan_device_table(plan.handle, phase, None, 0, ctypes.byref(n)),
           "bsm_plan_device_table")
    buf = (Patch * max(n.value, 1))()
    _check(lib().bsm_plan_device_table(plan.handle, phase, buf, n.value, ctypes.byref(n)),
           "bsm_plan_device_table")
    return _patch_array(buf, n.value)


def bsm_die_check_read(ptr, nbytes: int, chunk: int, die_of_chunk, invert: bool = False,
                       sm_group=None, device: int = -1):
    """SMs of each die (or of each group of sm_group) read only the chunks the
    map places on their die (or, inverted, the others); returns (XOR of the
    words read, kernel ms)."""
    m = _np(die_of_chunk, np.int8)
    assert len(m) * chunk == nbytes
    g = None if sm_group is None else _np(sm_group, np.int8)
    assert g is None or len(g) == MAX_SM
    xo = ctypes.c_uint32()
    ms = ctypes.c_float()
    _check(lib().bsm_die_check_read(device, _dptr(ptr, nbytes, "buffer"), nbytes, chunk,
                                    m.ctypes.data_as(ctypes.POINTER(ctypes.c_int8)),
                                    None if g is None else g.ctypes.data_as(ctypes.POINTER(ctypes.c_int8)),
                                    1 if invert else 0, ctypes.byref(xo), ctypes.byref(ms)),
           "bsm_die_check_read")
    return xo.value, ms.value


def bsm_addr_group_map(ptr, nbytes: int, chunk: int, sm_group, device: int = -1) -> np.ndarray:
    """bsm_addr_die_map for a caller's grouping of the SMs (MAX_SM entries of
    0, 1 or -1)."""
    g = _np(sm_group, np.int8)
    assert len(g) == MAX_SM
    n = (nbytes + chunk - 1) // chunk
    out = np.zeros(n, np.int8)
    _check(lib().bsm_addr_group_map(device, _dptr(ptr), nbytes, chunk,
                                    g.ctypes.data_as(ctypes.POINTER(ctypes.c_int8)),
                                    out.ctypes.data_as(ctypes.POINTER(ctypes.c_int8))),
           "bsm_addr_group_map")
    return out


DEBUG_NONE, DEBUG_WITHHOLD_STAGE, DEBUG_CORRUPT_PATCH = 0, 1, 2


def bsm_plan_debug(plan, what: int, arg: int = 0):
    """Test-only fault injection (see include/bsm.h); plan None targets the
    launches of bsm_softmax_noalloc."""
    _check(lib().bsm_plan_debug(None if plan is None else plan.handle, what, arg),
           "bsm_plan_debug")


def bsm_plan_destroy(plan: Plan):
    plan.close()


def bsm_cache_clear():
    lib().bsm_cache_clear()


def bsm_topology_probe(device: int = -1, force: bool = False) -> dict:
    t = Topology()
    _check(lib().bsm_topology_probe(device, 1 if force else 0, ctypes.byref(t)),
           "bsm_topology_probe")
    return {"device": t.device, "n_sm": t.n_sm, "n_die": t.n_die, "separable": t.separable,
            "sm_die": list(t.sm_die), "sm_per_die": list(t.sm_per_die), "l_near": t.l_near,
            "l_far": t.l_far, "separation": t.separation, "granularity": t.granularity,
            "probe_ms": t.probe_ms}


def bsm_addr_die_map(ptr, nbytes: int, chunk: int, device: int = -1) -> np.ndarray:
    n = (nbytes + chunk - 1) // chunk
    out = np.zeros(n, np.int8)
    _check(lib().bsm_addr_die_map(device, _dptr(ptr), nbytes, chunk,
                                  out.ctypes.data_as(ctypes.POINTER(ctypes.c_int8))),
           "bsm_addr_die_map")
    return out


def bsm_probe_latency(line_off, reps: int = 8, device: int = -1):
    off = _np(line_off, np.int64)
    lat = np.zeros((MAX_SM, len(off)), np.float32)
    seen = np.zeros(MAX_SM, np.int32)
    _check(lib().bsm_probe_latency(device, len(off), off.ctypes.data_as(c_i64p), reps,
                                   lat.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                                   seen.ctypes.data_as(c_i32p)), "bsm_probe_latency")
    return lat, seen


def bsm_plan_layout_host(rows, cols, dtype: int, policy: int, n_sm: int, smem_optin: int,
                         offsets=None, rows_per_item: int = 0, op: int = 0, x: int = 1 << 40,
                         y: int = 1 << 41, x2: int = 1 << 42) -> dict:
    """The patch table bsm_plan_create would build on a device with n_sm SMs
    and smem_optin bytes of opt-in shared memory (host only).  x, y, x2 are
    addresses for the alignment and overlap checks, never dereferenced.
    Returns the stage figures and two structured arrays of patches (fields of
    bsm_patch): phase 0 in slice order, phase 1 in launch order."""
    d = PlanDesc()
    _check(lib().bsm_plan_desc_init(ctypes.byref(d)), "bsm_plan_desc_init")
    r = _np(rows, np.int32)
    c = _np(cols, np.int32)
    off = None if offsets is None else _np(offsets, np.int64)
    d.x, d.y, d.x2 = x, y, x2
    d.num_slices = len(r)
    d.rows = r.ctypes.data_as(c_i32p)
    d.cols = c.ctypes.data_as(c_i32p)
    if off is not None:
        d.offsets = off.ctypes.data_as(c_i64p)
    d.dtype, d.policy, d.rows_per_item, d.op = dtype, policy, rows_per_item, op
    out = Layout()
    _check(lib().bsm_plan_layout_host(ctypes.byref(d), n_sm, smem_optin, None, 0, None, 0,
                                      ctypes.byref(out)), "bsm_plan_layout_host")
    n0, n1 = out.n_patches, out.n_patches_phase1
    p0 = (Patch * max(n0, 1))()
    p1 = (Patch * max(n1, 1))()
    _check(lib().bsm_plan_layout_host(ctypes.byref(d), n_sm, smem_optin, p0, n0, p1, n1,
                                      ctypes.byref(out)), "bsm_plan_layout_host")
    dt = np.dtype([(name, np.int64 if ct is ctypes.c_int64 else np.int32) for name, ct in Patch._fields_])
    a0 = np.frombuffer(bytes(p0), dtype=dt, count=n0) if n0 else np.zeros(0, dt)
    a1 = np.frombuffer(bytes(p1), dtype=dt, count=n1) if n1 else np.zeros(0, dt)
    return {"stage_bytes": out.stage_bytes, "n_stages": out.n_stages, "long_rows": out.long_rows,
            "group_k": out.group_k, "phase0": a0, "phase1": a1}


def bsm_schedule_host(patches: Sequence, maps: Sequence, n_banks: int, tie_seed: int,
                      balance: bool = False, units=None, l_near: int = 1, l_far: int = 1,
                      cost=None, minimax: bool = False) -> dict:
    """patches: (begin, end) byte ranges; maps: (chunk, bank_of_chunk) pairs."""
    n = len(patches)
    pb = _np([p[0] for p in patches], np.int64)
    pe = _np([p[1] for p in patches], np.int64)
    d = ScheduleDesc()
    d.n_banks = n_banks
    d.n_patches = n
    d.patch_begin = pb.ctypes.data_as(c_i64p)
    d.patch_end = pe.ctypes.data_as(c_i64p)
    d.n_maps = len(maps)
    keep = []
    for k, (chunk, bank_of_chunk) in enumerate(maps):
        arr = _np(bank_of_chunk, np.int8)
        keep.append(arr)
        d.chunk[k] = chunk
        d.n_chunks[k] = len(arr)
        d.bank_of_chunk[k] = arr.ctypes.data_as(ctypes.POINTER(ctypes.c_int8))
    d.tie_seed = tie_seed
    d.balance = 1 if balance else 0
    u = _np(units if units is not None else [1] * n_banks, np.int32)
    d.units = u.ctypes.data_as(c_i32p)
    d.l_near = l_near
    d.l_far = l_far
    cst = _np(cost if cost is not None else [p[1] - p[0] for p in patches], np.int64)
    d.cost = cst.ctypes.data_as(c_i64p)
    d.method = 1 if minimax else 0
    bob = np.zeros((max(n, 1), n_banks), np.int64)
    ov = np.zeros(max(n, 1), np.uint8)
    N = np.zeros(n_banks, np.int64)
    bank = np.zeros(max(n, 1), np.int32)
    L = np.zeros(n_banks, np.int64)
    qi = np.zeros(max(n, 1), np.int32)
    ql = np.zeros(n_banks, np.int64)
    mv = np.zeros(max(n, 1), np.int32)
    wb = np.zeros(n_banks, np.int64)
    wa = np.zeros(n_banks, np.int64)
    o = ScheduleOut()
    o.bytes_on_bank = bob.ctypes.data_as(c_i64p)
    o.overlap = ov.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8))
    o.N = N.ctypes.data_as(c_i64p)
    o.bank = bank.ctypes.data_as(c_i32p)
    o.L = L.ctypes.data_as(c_i64p)
    o.queue_items = qi.ctypes.data_as(c_i32p)
    o.queue_len = ql.ctypes.data_as(c_i64p)
    o.moved = mv.ctypes.data_as(c_i32p)
    o.work_before = wb.ctypes.data_as(c_i64p)
    o.work_after = wa.ctypes.data_as(c_i64p)
    _check(lib().bsm_schedule_host(ctypes.byref(d), ctypes.byref(o)), "bsm_schedule_host")
    queues, pos = [], 0
    for b in range(n_banks):
        queues.append([int(v) for v in qi[pos:pos + ql[b]]])
        pos += int(ql[b])
    return {"bytes_on_bank": bob[:n].tolist(), "overlap": ov[:n].tolist(), "N": N.tolist(),
            "bank": bank[:n].tolist(), "L": L.tolist(), "queues": queues,
            "moved": mv[:o.n_moved].tolist(), "work_before": wb.tolist(),
            "work_after": wa.tolist()}


def bsm_device_status(device: int = -1) -> int:
    v = ctypes.c_uint32()
    _check(lib().bsm_device_status(device, ctypes.byref(v)), "bsm_device_status")
    return v.value


def bsm_device_status_clear(device: int = -1):
    _check(lib().bsm_device_status_clear(device), "bsm_device_status_clear")


def bsm_device_debug(device: int = -1) -> list:
    out = (ctypes.c_uint32 * 8)()
    _check(lib().bsm_device_debug(device, out), "bsm_device_debug")
    return list(out)


def bsm_set_device_checks(on: bool):
    lib().bsm_set_device_checks(1 if on else 0)


def bsm_last_cuda_error() -> str:
    return lib().bsm_last_cuda_error().decode()


def bsm_max_row_bytes(device: int = -1) -> int:
    return int(lib().bsm_max_row_bytes(device))


def bsm_version() -> int:
    return int(lib().bsm_version())
