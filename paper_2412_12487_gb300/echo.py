"""Python binding of the C ABI in ``include/echo.h`` (argument marshalling only).

Every step of the hot path runs in ``libecho.so``; this module only converts
numpy arrays / torch tensors to pointers and status codes to exceptions.  It has
no fallback: if the library is missing or fails to load, it raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, Optional, Tuple

import numpy as np

from . import build as _build

ECHO_OK = 0
STATUS_NAMES = {0: "ECHO_OK", 1: "ECHO_E_INVALID_ARG", 2: "ECHO_E_BAD_GRAPH", 3: "ECHO_E_CYCLE",
                4: "ECHO_E_STATE", 5: "ECHO_E_OOM", 6: "ECHO_E_CUDA", 7: "ECHO_E_TIMEOUT",
                8: "ECHO_E_OVERFLOW", 9: "ECHO_E_UNSUPPORTED", 10: "ECHO_E_BOUNDS"}

# every function the header declares (checked by the tests)
EXPORTS = ["echo_create", "echo_destroy", "echo_check_graph", "echo_check_replicas", "echo_overlap_candidates", "echo_load_graph", "echo_load_scenarios",
           "echo_estimate_collectives", "echo_compose", "echo_read_times", "echo_read_makespan",
           "echo_read_cc", "echo_read_overlap", "echo_cc_query", "echo_cc_query_noalloc",
           "echo_graph_info_get", "echo_set_cc_model",
           "echo_set_profiling", "echo_read_profile", "echo_measure_fp64", "echo_strerror", "echo_last_error"]


class EchoError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


CUDA_STREAM_LEGACY = 0x1  # cudaStreamLegacy
CC_MODEL_WHITEBOX, CC_MODEL_ALPHA_BETA = 0, 1
OVERLAP_WHOLE, OVERLAP_PROPORTIONAL = 0, 1
COMM_EXECUTION, COMM_LAUNCH = 0, 1
AR_PER_OP, AR_RING, AR_TREE, AR_AUTO = 0, 1, 2, 3


class GraphDesc(C.Structure):
    _fields_ = [("n_ops", C.c_int64), ("n_ranks", C.c_int32), ("n_streams", C.c_int32),
                ("gpus_per_node", C.c_int32), ("n_groups", C.c_int32),
                ("kind", C.c_void_p), ("kclass", C.c_void_p), ("group", C.c_void_p),
                ("cc_type", C.c_void_p), ("cc_algo", C.c_void_p), ("cc_bytes", C.c_void_p),
                ("pred_off", C.c_void_p), ("pred_idx", C.c_void_p), ("q_off", C.c_void_p),
                ("q_ops", C.c_void_p), ("grp_off", C.c_void_p), ("grp_rank", C.c_void_p),
                ("replica_of", C.c_void_p)]


class ScenDesc(C.Structure):
    _fields_ = [("n_scen", C.c_int32), ("n_kclass", C.c_int32), ("n_chunk", C.c_int32),
                ("dur", C.c_void_p), ("alpha_ns", C.c_void_p), ("bw_intra", C.c_void_p),
                ("lat_intra", C.c_void_p), ("bw_inter", C.c_void_p), ("lat_inter", C.c_void_p),
                ("delta", C.c_void_p), ("slowdown", C.c_void_p), ("chunk_max_bytes", C.c_void_p),
                ("chunk_bytes", C.c_void_p), ("dur_bits", C.c_int32)]


class ComposeOpts(C.Structure):
    _fields_ = [("refine_passes", C.c_int32), ("overlap_model", C.c_int32), ("comm_interval", C.c_int32),
                ("ar_algo_policy", C.c_int32), ("debug_bounds", C.c_int32)]


class CCQueryDesc(C.Structure):
    _fields_ = [("n", C.c_int64), ("cc_type", C.c_void_p), ("cc_algo", C.c_void_p),
                ("nbytes", C.c_void_p), ("n_ranks", C.c_void_p), ("n_nodes", C.c_void_p),
                ("alpha_ns", C.c_void_p), ("bw_intra", C.c_void_p), ("lat_intra", C.c_void_p),
                ("bw_inter", C.c_void_p), ("lat_inter", C.c_void_p), ("delta", C.c_void_p),
                ("n_chunk", C.c_int32), ("chunk_max_bytes", C.c_void_p), ("chunk_bytes", C.c_void_p)]


class GraphInfo(C.Structure):
    _fields_ = [("n_ops", C.c_int64), ("n_edges", C.c_int64), ("n_levels", C.c_int64),
                ("max_width", C.c_int64), ("n_queue_entries", C.c_int64), ("n_comm_ops", C.c_int64),
                ("n_signatures", C.c_int64), ("n_segments", C.c_int64), ("n_segment_levels", C.c_int64),
                ("n_overlap_candidates", C.c_int64), ("n_ops_composed", C.c_int64),
                ("n_ranks", C.c_int32), ("n_streams", C.c_int32), ("sigma", C.c_int32),
                ("replicas_folded", C.c_int32), ("n_validator_comm_entries", C.c_int64),
                ("n_kept_finishes", C.c_int64)]


class KernelStat(C.Structure):
    _fields_ = [("name", C.c_char * 48), ("launches", C.c_int64), ("total_ms", C.c_double)]


_lib = None


def library_path() -> str:
    return _build.LIB


def load_library(path: Optional[str] = None):
    """Load libecho.so (raises if it is not built)."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or _build.LIB
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is not built; run paper_2412_12487_gb300.build.build() "
                           "(there is no CPU fallback)")
    lib = C.CDLL(p)
    vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
    sig = {
        "echo_create": ([C.POINTER(vp), C.c_int, vp], C.c_int),
        "echo_destroy": ([vp], C.c_int),
        "echo_check_graph": ([C.POINTER(GraphDesc), C.POINTER(i64), C.POINTER(i64)], C.c_int),
        "echo_check_replicas": ([C.POINTER(GraphDesc), C.POINTER(i64)], C.c_int),
        "echo_overlap_candidates": ([C.POINTER(GraphDesc), vp, C.POINTER(i64)], C.c_int),
        "echo_load_graph": ([vp, C.POINTER(GraphDesc)], C.c_int),
        "echo_load_scenarios": ([vp, C.POINTER(ScenDesc)], C.c_int),
        "echo_estimate_collectives": ([vp], C.c_int),
        "echo_compose": ([vp, C.POINTER(ComposeOpts)], C.c_int),
        "echo_read_times": ([vp, i64, i64, i32, i32, vp, vp], C.c_int),
        "echo_read_makespan": ([vp, vp], C.c_int),
        "echo_read_cc": ([vp, i64, i64, vp], C.c_int),
        "echo_read_overlap": ([vp, i64, i64, vp], C.c_int),
        "echo_cc_query": ([vp, C.POINTER(CCQueryDesc), vp], C.c_int),
        "echo_cc_query_noalloc": ([C.POINTER(CCQueryDesc), vp, vp], C.c_int),
        "echo_graph_info_get": ([vp, C.POINTER(GraphInfo)], C.c_int),
        "echo_set_cc_model": ([vp, C.c_int], C.c_int),
        "echo_set_profiling": ([vp, C.c_int], C.c_int),
        "echo_read_profile": ([vp, C.POINTER(KernelStat), C.c_int, C.POINTER(C.c_int)], C.c_int),
        "echo_measure_fp64": ([C.c_int, vp], C.c_int),
        "echo_strerror": ([C.c_int], C.c_char_p),
        "echo_last_error": ([vp, C.c_char_p, C.c_size_t], C.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _ptr(x) -> Optional[int]:
    """Host pointer of a numpy array or a CPU torch tensor."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    raise TypeError(type(x))


def _graph_desc(g, keep: list) -> GraphDesc:
    def a(x, dt):
        y = _c(x, dt)
        keep.append(y)
        return y.ctypes.data

    return GraphDesc(int(g.kind.shape[0]), int(g.n_ranks), int(g.n_streams), int(g.gpus_per_node),
                     int(g.grp_off.shape[0] - 1),
                     a(g.kind, np.uint8), a(g.kclass, np.uint8), a(g.group, np.int32),
                     a(g.cc_type, np.uint8), a(g.cc_algo, np.uint8), a(g.cc_bytes, np.int64),
                     a(g.pred_off, np.int64), a(g.pred_idx, np.int32), a(g.q_off, np.int64),
                     a(g.q_ops, np.int32), a(g.grp_off, np.int64), a(g.grp_rank, np.int32),
                     a(g.replica_of, np.int32) if getattr(g, "replica_of", None) is not None else None)


def check_graph(g) -> Tuple[int, int]:
    """Host-only validation + levelling (no device needed): (n_levels, max_width)."""
    lib = load_library()
    keep: list = []
    d = _graph_desc(g, keep)
    L, W = C.c_int64(0), C.c_int64(0)
    rc = lib.echo_check_graph(C.byref(d), C.byref(L), C.byref(W))
    if rc:
        raise EchoError(rc, lib.echo_strerror(rc).decode())
    return int(L.value), int(W.value)


def check_replicas(g) -> int:
    """Host-only check of ``g.replica_of``: the number of ops the folded graph
    composes (``g.n_ops`` when nothing is folded)."""
    lib = load_library()
    keep: list = []
    d = _graph_desc(g, keep)
    n = C.c_int64(0)
    rc = lib.echo_check_replicas(C.byref(d), C.byref(n))
    if rc:
        raise EchoError(rc, lib.echo_strerror(rc).decode())
    return int(n.value)


def overlap_candidates(g) -> np.ndarray:
    """Host-only: uint8 [n_ops], 1 for the compute ops the validator tests (those
    that can overlap a comm op of their rank in some scenario)."""
    lib = load_library()
    keep: list = []
    d = _graph_desc(g, keep)
    out = np.zeros(int(g.kind.shape[0]), np.uint8)
    n = C.c_int64(0)
    rc = lib.echo_overlap_candidates(C.byref(d), _ptr(out) if out.size else None, C.byref(n))
    if rc:
        raise EchoError(rc, lib.echo_strerror(rc).decode())
    assert int(out.sum()) == int(n.value)
    return out


def measure_fp64(device: int = 0) -> Dict[str, float]:
    """fp64 add / multiply / divide rates of the device (operations per second)."""
    lib = load_library()
    r = np.zeros(3, np.float64)
    rc = lib.echo_measure_fp64(int(device), _ptr(r))
    if rc:
        raise EchoError(rc, lib.echo_strerror(rc).decode())
    return {"dadd": float(r[0]), "dmul": float(r[1]), "ddiv": float(r[2])}


class Echo:
    """One composer context on one device (see include/echo.h for the semantics)."""

    def __init__(self, device: int = 0, stream=None):
        self.lib = load_library()
        if stream is None:
            import torch
            stream = torch.cuda.current_stream(device)
        if hasattr(stream, "cuda_stream"):
            # torch's default stream has handle 0, the legacy default stream: pass it as
            # cudaStreamLegacy so the library's work stays in that stream's order
            handle = stream.cuda_stream or CUDA_STREAM_LEGACY
        else:
            handle = int(stream or 0)
        h = C.c_void_p()
        rc = self.lib.echo_create(C.byref(h), int(device), C.c_void_p(handle) if handle else None)
        if rc:
            raise EchoError(rc, "echo_create failed")
        self.h = h
        self.n_ops = 0
        self.n_scen = 0

    def _check(self, rc: int):
        if rc:
            buf = C.create_string_buffer(512)
            self.lib.echo_last_error(self.h, buf, 512)
            raise EchoError(rc, buf.value.decode(errors="replace"))

    def close(self):
        if getattr(self, "h", None):
            self.lib.echo_destroy(self.h)
            self.h = None

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- the calls of the C ABI -------------------------------------------------------
    def load_graph(self, g):
        keep: list = []
        d = _graph_desc(g, keep)
        self._check(self.lib.echo_load_graph(self.h, C.byref(d)))
        self.n_ops = int(g.kind.shape[0])

    def load_scenarios(self, sc, dur=None):
        """``dur`` overrides ``sc.dur`` (e.g. a pinned torch tensor of the same shape).
        int32 durations (numpy or torch) are uploaded as such, half the bytes of int64."""
        keep: list = []

        def a(x, dt):
            y = _c(x, dt)
            keep.append(y)
            return y.ctypes.data

        D = sc.dur if dur is None else dur
        bits = 32 if str(getattr(D, "dtype", "")) in ("int32", "torch.int32") else 64
        if isinstance(D, np.ndarray):
            D = _c(D, np.int32 if bits == 32 else np.int64)
            keep.append(D)
        S = int(sc.alpha_ns.shape[0])
        n_chunk = 0 if sc.chunk_max_bytes is None else len(sc.chunk_max_bytes)
        d = ScenDesc(S, int(sc.slowdown.shape[0]), n_chunk, _ptr(D),
                     a(sc.alpha_ns, np.float64), a(sc.bw_intra, np.float64), a(sc.lat_intra, np.float64),
                     a(sc.bw_inter, np.float64), a(sc.lat_inter, np.float64), a(sc.delta, np.float64),
                     a(sc.slowdown, np.float64),
                     a(sc.chunk_max_bytes, np.int64) if n_chunk else None,
                     a(sc.chunk_bytes, np.int64) if n_chunk else None, bits)
        self._check(self.lib.echo_load_scenarios(self.h, C.byref(d)))
        self.n_scen = S

    def estimate_collectives(self):
        self._check(self.lib.echo_estimate_collectives(self.h))

    def compose(self, refine_passes: int = 1, overlap_model: int = 0, comm_interval: int = 0,
                ar_algo_policy: int = 0, debug_bounds: bool = False):
        """overlap_model: OVERLAP_WHOLE (d * factor) or OVERLAP_PROPORTIONAL
        (d + (factor - 1) * overlapped length).  comm_interval: COMM_EXECUTION (a
        comm op's [start, finish)) or COMM_LAUNCH (from each member rank's launch).
        ar_algo_policy: AR_PER_OP (each all-reduce's own algorithm), AR_RING,
        AR_TREE or AR_AUTO for every all-reduce.  debug_bounds: device-side index
        checks (ECHO_E_BOUNDS from the next read when one fails)."""
        o = ComposeOpts(int(refine_passes), int(overlap_model), int(comm_interval), int(ar_algo_policy),
                        1 if debug_bounds else 0)
        self._check(self.lib.echo_compose(self.h, C.byref(o)))

    def read_times(self, op0: int = 0, op1: Optional[int] = None, start=True, finish=True,
                   s0: int = 0, s1: Optional[int] = None):
        """Start and finish of ops [op0, op1) in scenarios [s0, s1): int64 [op][s - s0]."""
        op1 = self.n_ops if op1 is None else op1
        s1 = self.n_scen if s1 is None else s1
        n, m = max(op1 - op0, 0), max(s1 - s0, 0)
        st = np.empty((n, m), np.int64) if start else None
        fn = np.empty((n, m), np.int64) if finish else None
        self._check(self.lib.echo_read_times(self.h, op0, op1, int(s0), int(s1), _ptr(st), _ptr(fn)))
        return st, fn

    def read_makespan(self, out=None):
        out = np.empty(self.n_scen, np.int64) if out is None else out
        self._check(self.lib.echo_read_makespan(self.h, _ptr(out)))
        return out

    def read_cc(self, op0: int = 0, op1: Optional[int] = None):
        op1 = self.n_ops if op1 is None else op1
        out = np.empty((max(op1 - op0, 0), self.n_scen), np.float64)
        self._check(self.lib.echo_read_cc(self.h, op0, op1, _ptr(out)))
        return out

    def read_overlap(self, op0: int = 0, op1: Optional[int] = None):
        op1 = self.n_ops if op1 is None else op1
        out = np.empty((max(op1 - op0, 0), self.n_scen), np.uint8)
        self._check(self.lib.echo_read_overlap(self.h, op0, op1, _ptr(out)))
        return out

    def cc_query(self, q) -> np.ndarray:
        keep: list = []

        def a(x, dt):
            y = _c(x, dt)
            keep.append(y)
            return y.ctypes.data

        n = int(q.cc_type.shape[0])
        d = CCQueryDesc(n, a(q.cc_type, np.uint8), a(q.cc_algo, np.uint8), a(q.nbytes, np.int64),
                        a(q.n_ranks, np.int32), a(q.n_nodes, np.int32), a(q.alpha_ns, np.float64),
                        a(q.bw_intra, np.float64), a(q.lat_intra, np.float64), a(q.bw_inter, np.float64),
                        a(q.lat_inter, np.float64), a(q.delta, np.float64), 0, None, None)
        out = np.empty(n, np.float64)
        self._check(self.lib.echo_cc_query(self.h, C.byref(d), _ptr(out)))
        return out

    def info(self) -> Dict[str, int]:
        gi = GraphInfo()
        self._check(self.lib.echo_graph_info_get(self.h, C.byref(gi)))
        return {k: int(getattr(gi, k)) for k, _ in GraphInfo._fields_}

    def set_cc_model(self, model: int):
        """CC_MODEL_WHITEBOX (Eqs. 2-5, default) or CC_MODEL_ALPHA_BETA for the next estimate."""
        self._check(self.lib.echo_set_cc_model(self.h, int(model)))

    def set_profiling(self, on: bool):
        self._check(self.lib.echo_set_profiling(self.h, 1 if on else 0))

    def read_profile(self) -> Dict[str, Tuple[int, float]]:
        buf = (KernelStat * 32)()
        n = C.c_int(0)
        self._check(self.lib.echo_read_profile(self.h, buf, 32, C.byref(n)))
        return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms)) for i in range(n.value)}
