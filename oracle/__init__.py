"""CPU oracle for the Echo timeline composer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may
import this package.  The product path never does: it runs on the CUDA library.

``compose`` runs the plain single-threaded C event-driven simulator of
``echo_oracle.c`` (Sec. 4.2, 5.2, 5.3 and the validator of Sec. 3/6); ``cc_ns``
evaluates one collective with Eqs. 2-5.  Scenario ranges may be composed from
several Python threads (ctypes releases the GIL), each range on one core.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "liboracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle with plain gcc (no FMA contraction, no fast-math)."""
    src = os.path.join(_HERE, "echo_oracle.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "echo_oracle.h"))):
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                               "-fPIC", "-shared", "-o", tmp, src, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class _Graph(C.Structure):
    _fields_ = [("n_ops", C.c_int64), ("n_ranks", C.c_int32), ("n_streams", C.c_int32),
                ("gpus_per_node", C.c_int32),
                ("n_groups", C.c_int32),
                ("kind", C.c_void_p), ("kclass", C.c_void_p), ("cc_type", C.c_void_p),
                ("cc_algo", C.c_void_p), ("group", C.c_void_p), ("cc_bytes", C.c_void_p),
                ("pred_off", C.c_void_p), ("pred_idx", C.c_void_p), ("q_off", C.c_void_p),
                ("q_ops", C.c_void_p), ("grp_off", C.c_void_p), ("grp_rank", C.c_void_p)]


class _Scen(C.Structure):
    _fields_ = [("n_scen", C.c_int32), ("n_kclass", C.c_int32), ("n_chunk", C.c_int32),
                ("dur", C.c_void_p), ("alpha_ns", C.c_void_p), ("bw_intra", C.c_void_p),
                ("lat_intra", C.c_void_p), ("bw_inter", C.c_void_p), ("lat_inter", C.c_void_p),
                ("delta", C.c_void_p), ("slowdown", C.c_void_p),
                ("chunk_max_bytes", C.c_void_p), ("chunk_bytes", C.c_void_p), ("cc_model", C.c_int32),
                ("overlap_model", C.c_int32), ("comm_interval", C.c_int32), ("ar_algo_policy", C.c_int32)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = C.CDLL(_SO)
            lib.oracle_chunk_bytes.restype = C.c_int64
            lib.oracle_chunk_bytes.argtypes = [C.c_int64, C.c_int, C.c_void_p, C.c_void_p]
            lib.oracle_cc_ns.restype = C.c_double
            lib.oracle_cc_ns.argtypes = [C.c_int, C.c_int, C.c_int64, C.c_int, C.c_int, C.c_int,
                                         C.c_double, C.c_void_p, C.c_int, C.c_void_p, C.c_void_p]
            lib.oracle_cc_ns_alpha_beta.restype = C.c_double
            lib.oracle_cc_ns_alpha_beta.argtypes = [C.c_int64, C.c_int, C.c_int, C.c_void_p]
            lib.oracle_compose.restype = C.c_int
            lib.oracle_compose.argtypes = [C.POINTER(_Graph), C.POINTER(_Scen), C.c_int32, C.c_int32,
                                           C.c_int32, C.c_uint64, C.c_void_p, C.c_void_p,
                                           C.c_void_p, C.c_void_p, C.c_void_p]
            _lib = lib
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def chunk_bytes(nbytes: int, table=None) -> int:
    lib = _load()
    if table is None:
        return int(lib.oracle_chunk_bytes(int(nbytes), 0, None, None))
    mx, cb = _c(table[0], np.int64), _c(table[1], np.int64)
    return int(lib.oracle_chunk_bytes(int(nbytes), len(mx), _p(mx), _p(cb)))


def cc_ns(cc_type: int, cc_algo: int, nbytes: int, N: int, M: int, K: int, lg: float,
          alpha: float, bw_intra: float, lat_intra: float, bw_inter: float, lat_inter: float,
          delta: float, table=None) -> float:
    lib = _load()
    prm = np.array([alpha, bw_intra, lat_intra, bw_inter, lat_inter, delta], np.float64)
    if table is None:
        return float(lib.oracle_cc_ns(cc_type, cc_algo, nbytes, N, M, K, lg, _p(prm), 0, None, None))
    mx, cb = _c(table[0], np.int64), _c(table[1], np.int64)
    return float(lib.oracle_cc_ns(cc_type, cc_algo, nbytes, N, M, K, lg, _p(prm), len(mx),
                                  _p(mx), _p(cb)))


def cc_ns_alpha_beta(nbytes: int, N: int, M: int, alpha: float, bw_intra: float, lat_intra: float,
                     bw_inter: float, lat_inter: float, delta: float) -> float:
    lib = _load()
    prm = np.array([alpha, bw_intra, lat_intra, bw_inter, lat_inter, delta], np.float64)
    return float(lib.oracle_cc_ns_alpha_beta(int(nbytes), int(N), int(M), _p(prm)))


class OracleResult:
    def __init__(self, start, finish, makespan, cc_ns, overlapped):
        self.start, self.finish, self.makespan = start, finish, makespan
        self.cc_ns, self.overlapped = cc_ns, overlapped


def compose(g, sc, refine_passes: int = 1, tie_seed: int = 0, threads: int = 1,
            want_cc: bool = True, want_overlap: bool = True, cc_model: int = 0,
            overlap_model: int = 0, comm_interval: int = 0, ar_algo_policy: int = 0,
            want_times: bool = True) -> OracleResult:
    """Compose every scenario of ``sc`` on graph ``g`` (workloads.Graph/Scenarios).
    cc_model 0 takes collective times from Eqs. 2-5, 1 from the alpha-beta model.
    overlap_model 0 slows an overlapped kernel to d * factor, 1 to
    d + (factor - 1) * (length of its overlap with the rank's communication).
    comm_interval 0 takes a comm op's execution interval [start, finish) on each
    member rank, 1 the interval from the rank's own launch of it to its finish.
    ar_algo_policy 0 keeps every all-reduce's own algorithm; 1 ring, 2 tree, 3 the
    faster of the two, for every all-reduce.  want_times False returns only the
    makespans (start and finish are None), for large batches."""
    lib = _load()
    V, S = g.n_ops, sc.n_scen
    keep = []

    def arr(a, dt):
        x = _c(a, dt)
        keep.append(x)
        return x.ctypes.data

    gs = _Graph(V, g.n_ranks, g.n_streams, g.gpus_per_node, g.n_groups,
                arr(g.kind, np.uint8), arr(g.kclass, np.uint8), arr(g.cc_type, np.uint8),
                arr(g.cc_algo, np.uint8), arr(g.group, np.int32), arr(g.cc_bytes, np.int64),
                arr(g.pred_off, np.int64), arr(g.pred_idx, np.int32), arr(g.q_off, np.int64),
                arr(g.q_ops, np.int32), arr(g.grp_off, np.int64), arr(g.grp_rank, np.int32))
    n_chunk = 0 if sc.chunk_max_bytes is None else len(sc.chunk_max_bytes)
    ss = _Scen(S, int(sc.slowdown.shape[0]), n_chunk, arr(sc.dur.reshape(-1) if V else np.zeros(1), np.int64),
               arr(sc.alpha_ns, np.float64), arr(sc.bw_intra, np.float64), arr(sc.lat_intra, np.float64),
               arr(sc.bw_inter, np.float64), arr(sc.lat_inter, np.float64), arr(sc.delta, np.float64),
               arr(sc.slowdown, np.float64),
               arr(sc.chunk_max_bytes, np.int64) if n_chunk else None,
               arr(sc.chunk_bytes, np.int64) if n_chunk else None, int(cc_model), int(overlap_model),
               int(comm_interval), int(ar_algo_policy))
    start = np.zeros((V, S), np.int64) if want_times else None
    finish = np.zeros((V, S), np.int64) if want_times else None
    mk = np.zeros(S, np.int64)
    ccn = np.full((V, S), np.nan) if want_cc else None
    ov = np.zeros((V, S), np.uint8) if want_overlap else None
    threads = max(1, min(int(threads), S)) if S else 1
    bounds = np.linspace(0, S, threads + 1).astype(int)
    rcs = [0] * threads

    def run(i):
        rcs[i] = lib.oracle_compose(C.byref(gs), C.byref(ss), int(bounds[i]), int(bounds[i + 1]),
                                    refine_passes, tie_seed, _p(start), _p(finish),
                                    mk.ctypes.data, _p(ccn), _p(ov))

    if threads == 1:
        run(0)
    else:
        ts = [threading.Thread(target=run, args=(i,)) for i in range(threads)]
        for t in ts:
            t.start()
        for t in ts:
            t.join()
    for rc in rcs:
        if rc == 2:
            raise RuntimeError("oracle: execution graph deadlocks (dependency cycle)")
        if rc:
            raise RuntimeError(f"oracle: error {rc}")
    return OracleResult(start, finish, mk, ccn, ov)
