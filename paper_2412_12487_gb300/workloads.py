"""Seeded synthetic inputs shaped like Megatron-LM 3D-parallel GPT training steps.

This module only *builds inputs*: multi-rank execution graphs (the per-rank graphs
of Echo's workload tracer, Sec. 4.1, with the 1F1B inter-stage matching rules of
Sec. 4.2 materialised as shared P2P nodes) and per-scenario parameters (kernel
durations, link parameters, slowdown factors).  It holds none of the composer's,
the CC estimator's or the validator's arithmetic; both the CUDA path and the CPU
oracle consume what it produces.

Graph format (the boundary's input format):

* ``kind[V]``      0 compute, 1 memcpy, 2 collective, 3 point-to-point
* ``kclass[V]``    kernel class of a compute op (index into the slowdown table)
* ``group[V]``     communicator group of a comm op (-1 otherwise)
* ``cc_type[V]``   0 all-reduce, 1 all-gather, 2 reduce-scatter, 3 send/recv
* ``cc_algo[V]``   0 ring, 1 tree, 2 auto (all-reduce only)
* ``cc_bytes[V]``  message size in bytes of a comm op
* ``pred_off/pred_idx``  CSR of *data* dependencies (cross-stream, cross-rank)
* ``q_off/q_ops``  program order: queue ``r*n_streams + k`` lists the ops that rank
  ``r`` issues on its stream ``k``, in issue order.  Stream 0 is the rank's compute
  timeline and holds every compute op of the rank and nothing else; streams 1.. are
  communication or memcpy timelines.  A comm op appears once in a stream of every
  member of its group.  The GPT workloads use one stream per communicator kind, as
  PyTorch's NCCL process groups do: 1 tensor-parallel, 2 pipeline, 3 data-parallel
  (and the global gradient-norm all-reduce), 4 memcpy.
* ``grp_off/grp_rank``  CSR of the member ranks of each group.

Durations (int64 ns) follow the recipe d(v, s) = rint(F_v / P_s * n_v): F_v is the
op's FLOP count (GEMM/bmm) or a FLOP-equivalent of its bytes for memory-bound
kernels, P_s the scenario's peak FLOP/ns and n_v ~ lognormal(0, 0.1) per op.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Tuple

import numpy as np

KIND_COMPUTE, KIND_MEMCPY, KIND_COLL, KIND_P2P = 0, 1, 2, 3
CC_ALLREDUCE, CC_ALLGATHER, CC_REDUCESCATTER, CC_SENDRECV = 0, 1, 2, 3
ALGO_RING, ALGO_TREE, ALGO_AUTO = 0, 1, 2
STREAM_COMPUTE, STREAM_TP, STREAM_PP, STREAM_DP, STREAM_MEMCPY = 0, 1, 2, 3, 4
# interleaved schedules: activation receives (STREAM_PP holds the sends), gradient
# sends and gradient receives on timelines of their own
STREAM_PP_RECV, STREAM_PP_GRAD, STREAM_PP_GRAD_RECV = 5, 6, 7
N_STREAMS = 5

# kernel classes (the kernel types the slowdown statistics of Sec. 2.3 distinguish)
KC_GEMM, KC_BMM, KC_SOFTMAX, KC_NORM, KC_ELEM, KC_OPT, KC_EMB, KC_LOSS = range(8)
N_KCLASS = 8

# FLOP-equivalent of one byte of a memory-bound kernel: 400 TFLOP/s / 2 TB/s
MEM_FLOP_PER_BYTE = 200.0
# FLOP-equivalent of one memcpy byte (about 50 GB/s at 400 TFLOP/s) and its fixed latency
COPY_FLOP_PER_BYTE = 8000.0
COPY_FIXED_FLOP = 4.0e5 * 2000.0          # 2 us at 400 TFLOP/s
DP_BUCKET_ELEMS = 40_000_000             # gradient bucket size (elements)
VOCAB = 51200

# H800-like two-tier defaults (Sec. 8.1 cluster description)
NVLINK_GBS, NVLINK_LAT_NS = 400.0, 2000.0
IB_GBS, IB_LAT_NS = 50.0, 5000.0
ALPHA_NS = 10_000.0
DELTA_NS_PER_B = 1657.72e3 / float(256 << 20)   # reduce time of a 256 MiB tensor (Table 6)


@dataclasses.dataclass
class Graph:
    n_ranks: int
    n_streams: int
    gpus_per_node: int
    kind: np.ndarray
    kclass: np.ndarray
    group: np.ndarray
    cc_type: np.ndarray
    cc_algo: np.ndarray
    cc_bytes: np.ndarray
    pred_off: np.ndarray
    pred_idx: np.ndarray
    q_off: np.ndarray
    q_ops: np.ndarray
    grp_off: np.ndarray
    grp_rank: np.ndarray
    work: np.ndarray      # FLOP(-equivalent) per op, input-recipe only
    noise: np.ndarray     # lognormal factor per op, input-recipe only
    name: str = ""
    replica_of: Optional[np.ndarray] = None  # int32 [n_ranks]: rank -> its representative

    @property
    def n_ops(self) -> int:
        return int(self.kind.shape[0])

    @property
    def n_edges(self) -> int:
        return int(self.pred_idx.shape[0])

    @property
    def n_groups(self) -> int:
        return int(self.grp_off.shape[0] - 1)

    def stats(self) -> Dict[str, int]:
        k = self.kind
        return {
            "V": self.n_ops, "E": self.n_edges, "ranks": self.n_ranks,
            "compute": int((k == KIND_COMPUTE).sum()), "memcpy": int((k == KIND_MEMCPY).sum()),
            "coll": int((k == KIND_COLL).sum()), "p2p": int((k == KIND_P2P).sum()),
            "queue_entries": int(self.q_ops.shape[0]), "groups": self.n_groups,
        }


@dataclasses.dataclass
class Scenarios:
    dur: np.ndarray           # int64 [V][S]; entries of comm ops are ignored (0)
    alpha_ns: np.ndarray      # float64 [S]
    bw_intra: np.ndarray      # bytes/ns (= GB/s)
    lat_intra: np.ndarray     # ns
    bw_inter: np.ndarray
    lat_inter: np.ndarray
    delta: np.ndarray         # ns per byte of reduction
    slowdown: np.ndarray      # float64 [C][S]
    peak_flop_per_ns: np.ndarray  # input-recipe only
    chunk_max_bytes: Optional[np.ndarray] = None
    chunk_bytes: Optional[np.ndarray] = None

    @property
    def n_scen(self) -> int:
        return int(self.alpha_ns.shape[0])


@dataclasses.dataclass
class GPTConfig:
    name: str
    layers: int
    hidden: int
    heads: int
    seq: int
    tp: int
    pp: int
    dp: int
    microbatches: int
    n_scen: int
    gpus_per_node: int = 8
    fixed_scenario: bool = False     # one fixed H800-like scenario instead of random draws
    graph_seed: int = 0
    scen_seed: int = 1000
    # DP replicas that run identical kernels (each replica op takes its replica-0
    # original's noise draw); the graph then carries replica_of for folding
    identical_replicas: bool = False
    # model chunks per rank: 1 = 1F1B, v > 1 = interleaved 1F1B over PP * v virtual stages
    virtual_stages: int = 1


# The five workloads (GPT shapes of Table 7; 3D-parallel layouts as in Sec. 8).
CONFIGS: Dict[str, GPTConfig] = {
    "tiny": GPTConfig("tiny-gpt-2L-h1024-tp2pp2dp2", 2, 1024, 16, 512, 2, 2, 2, 2, 1,
                      fixed_scenario=True, scen_seed=1001),
    "gpt1.3b": GPTConfig("gpt-1.3b-tp2pp4dp8-m8", 24, 2048, 16, 2048, 2, 4, 8, 8, 256,
                         scen_seed=1002),
    "gpt175b": GPTConfig("gpt-175b-tp8pp6dp2-m16", 96, 12288, 96, 2048, 8, 6, 2, 16, 1024,
                         scen_seed=1003),
    "gpt175b-1024": GPTConfig("gpt-175b-tp8pp16dp8-m64-v2", 96, 12288, 96, 2048, 8, 16, 8, 64, 64,
                              scen_seed=1004, virtual_stages=2),
    # a smaller case of the 1024-rank workload's structure (same ranks, schedule and
    # timelines; 32 layers, 16 micro-batches), for kernel profiles that must stay small
    "gpt175b-1024-small": GPTConfig("gpt-175b-tp8pp16dp8-m16-v2-32L", 32, 12288, 96, 2048, 8, 16, 8, 16, 64,
                                    scen_seed=1004, virtual_stages=2),
}


# ---------------------------------------------------------------------------------------
# per-stage program (template shared by every rank of a pipeline stage)
# ---------------------------------------------------------------------------------------
_E_COMP, _E_MEMCPY, _E_TP, _E_P2P, _E_DP, _E_WORLD, _E_P2P_RECV, _E_P2P_GRAD, _E_P2P_GRAD_RECV = range(9)
_E_P2P_ALL = (_E_P2P, _E_P2P_RECV, _E_P2P_GRAD, _E_P2P_GRAD_RECV)


class _StageProgram:
    def __init__(self) -> None:
        self.etype: List[int] = []
        self.kclass: List[int] = []
        self.work: List[float] = []
        self.nbytes: List[int] = []
        self.cctype: List[int] = []
        self.algo: List[int] = []
        self.key: List[object] = []
        self.src: List[int] = []
        self.dst: List[int] = []

    def _add(self, et, kc, work, nbytes, cct, algo, key, deps) -> int:
        i = len(self.etype)
        self.etype.append(et); self.kclass.append(kc); self.work.append(float(work))
        self.nbytes.append(int(nbytes)); self.cctype.append(cct); self.algo.append(algo)
        self.key.append(key)
        for d in deps:
            if d is not None:
                self.src.append(d); self.dst.append(i)
        return i

    def comp(self, kc, work, deps=()):
        return self._add(_E_COMP, kc, work, 0, 0, 0, None, deps)

    def memcpy(self, nbytes, deps=()):
        return self._add(_E_MEMCPY, KC_ELEM, COPY_FIXED_FLOP + COPY_FLOP_PER_BYTE * nbytes,
                         0, 0, 0, None, deps)

    def comm(self, et, nbytes, cct, algo, key, deps=()):
        return self._add(et, 0, 0.0, nbytes, cct, algo, key, deps)


def _fwd_kernels(c: GPTConfig):
    b, h, s, tp = c.seq, c.hidden, c.seq, c.tp
    a = c.heads
    M = MEM_FLOP_PER_BYTE
    att_elems = b * s * a / tp
    # (name, class, work); 'AR' marks a tensor-parallel all-reduce after the previous kernel
    return [
        ("ln1", KC_NORM, 4 * b * h * M),
        ("qkv", KC_GEMM, 2 * b * h * 3 * h / tp),
        ("qkv_bias", KC_ELEM, 4 * b * 3 * h / tp * M),
        ("rotary", KC_ELEM, 4 * b * 2 * h / tp * M),
        ("qk", KC_BMM, 2 * b * s * h / tp),
        ("softmax", KC_SOFTMAX, 4 * att_elems * M),
        ("attn_dropout", KC_ELEM, 4 * att_elems * M),
        ("av", KC_BMM, 2 * b * s * h / tp),
        ("transpose", KC_ELEM, 4 * b * h / tp * M),
        ("proj", KC_GEMM, 2 * b * h * h / tp),
        ("AR", None, None),
        ("bda1", KC_ELEM, 6 * b * h * M),
        ("ln2", KC_NORM, 4 * b * h * M),
        ("fc1", KC_GEMM, 2 * b * h * 4 * h / tp),
        ("bias_gelu", KC_ELEM, 4 * b * 4 * h / tp * M),
        ("fc2", KC_GEMM, 2 * b * 4 * h * h / tp),
        ("AR", None, None),
        ("bda2", KC_ELEM, 6 * b * h * M),
    ]


def _bwd_kernels(c: GPTConfig):
    b, h, s, tp = c.seq, c.hidden, c.seq, c.tp
    a = c.heads
    M = MEM_FLOP_PER_BYTE
    att_elems = b * s * a / tp
    p_qkv, p_proj, p_fc1, p_fc2 = 3 * h * h / tp, h * h / tp, 4 * h * h / tp, 4 * h * h / tp
    # (name, class, work, params whose gradient is complete after this kernel)
    return [
        ("bda2_bwd", KC_ELEM, 6 * b * h * M, 0),
        ("fc2_dgrad", KC_GEMM, 2 * b * 4 * h * h / tp, 0),
        ("fc2_wgrad", KC_GEMM, 2 * b * 4 * h * h / tp, 0),
        ("fc2_gacc", KC_ELEM, 8 * p_fc2 * M, p_fc2),
        ("gelu_bwd", KC_ELEM, 6 * b * 4 * h / tp * M, 0),
        ("fc1_dgrad", KC_GEMM, 2 * b * h * 4 * h / tp, 0),
        ("AR", None, None, 0),
        ("fc1_wgrad", KC_GEMM, 2 * b * h * 4 * h / tp, 0),
        ("fc1_gacc", KC_ELEM, 8 * p_fc1 * M, p_fc1),
        ("ln2_bwd", KC_NORM, 6 * b * h * M, 0),
        ("res2_add", KC_ELEM, 6 * b * h * M, 0),
        ("bda1_bwd", KC_ELEM, 6 * b * h * M, 0),
        ("proj_dgrad", KC_GEMM, 2 * b * h * h / tp, 0),
        ("proj_wgrad", KC_GEMM, 2 * b * h * h / tp, 0),
        ("proj_gacc", KC_ELEM, 8 * p_proj * M, p_proj),
        ("transpose_bwd", KC_ELEM, 4 * b * h / tp * M, 0),
        ("av_dv", KC_BMM, 2 * b * s * h / tp, 0),
        ("av_dp", KC_BMM, 2 * b * s * h / tp, 0),
        ("dropout_bwd", KC_ELEM, 4 * att_elems * M, 0),
        ("softmax_bwd", KC_SOFTMAX, 6 * att_elems * M, 0),
        ("qk_dq", KC_BMM, 2 * b * s * h / tp, 0),
        ("qk_dk", KC_BMM, 2 * b * s * h / tp, 0),
        ("rotary_bwd", KC_ELEM, 4 * b * 2 * h / tp * M, 0),
        ("qkv_bias_bwd", KC_ELEM, 4 * b * 3 * h / tp * M, 0),
        ("qkv_dgrad", KC_GEMM, 2 * b * h * 3 * h / tp, 0),
        ("AR", None, None, 0),
        ("qkv_wgrad", KC_GEMM, 2 * b * h * 3 * h / tp, 0),
        ("qkv_gacc", KC_ELEM, 8 * p_qkv * M, p_qkv),
        ("ln1_bwd", KC_NORM, 6 * b * h * M, 0),
        ("res1_add", KC_ELEM, 6 * b * h * M, 0),
    ]


def _stage_program(c: GPTConfig, p: int) -> _StageProgram:
    """Issue order of one rank of pipeline stage ``p`` under non-interleaved 1F1B.

    The inter-stage matching rule of Sec. 4.2 is made explicit: each batched
    send/recv call between stages b and b+1 becomes one 2-member P2P node keyed by
    ('fa', b, mb) for a lone activation transfer, ('pair', b, t) for the steady-state
    send-forward/recv-backward pair, and ('g', b, t) for a lone gradient transfer.
    """
    PP, m, tp, dp = c.pp, c.microbatches, c.tp, c.dp
    if c.layers % PP:
        raise ValueError("layers must divide evenly across pipeline stages")
    if m < PP:
        raise ValueError("1F1B generator needs microbatches >= pipeline stages")
    nl = c.layers // PP
    b, h = c.seq, c.hidden
    act_bytes = b * h * 2
    prog = _StageProgram()
    fwd = _fwd_kernels(c)
    bwd = _bwd_kernels(c)
    M = MEM_FLOP_PER_BYTE
    first, last = p == 0, p == PP - 1
    W = min(PP - p - 1, m)
    R = m - W
    act_in: Dict[int, int] = {}     # microbatch -> P2P entry that delivers its activation
    grad_in: Dict[int, int] = {}    # microbatch -> P2P entry that delivers its output gradient
    act_out: Dict[int, int] = {}
    grad_out: Dict[int, int] = {}
    dp_entries: List[int] = []
    bucket = [0.0]

    def tp_ar(dep):
        return prog.comm(_E_TP, act_bytes, CC_ALLREDUCE, ALGO_AUTO, None, deps=[dep])

    def flush_bucket(dep):
        if dp > 1 and bucket[0] > 0:
            e = prog.comm(_E_DP, int(bucket[0]) * 2, CC_ALLREDUCE, ALGO_AUTO, len(dp_entries),
                          deps=[dep])
            dp_entries.append(e)
        bucket[0] = 0.0

    def add_grad(params, dep, last_mb):
        if last_mb and dp > 1:
            bucket[0] += params
            if bucket[0] >= DP_BUCKET_ELEMS:
                flush_bucket(dep)

    def F(mb):
        dep = act_in.get(mb) if not first else None
        if first:
            mc = prog.memcpy(b * 8)
            dep = prog.comp(KC_EMB, 4 * b * h * M, deps=[mc])
        pend = [dep]
        for _ in range(nl):
            for name, kc, work in fwd:
                if name == "AR":
                    if tp > 1:
                        pend = [tp_ar(prev)]
                    continue
                prev = prog.comp(kc, work, deps=pend)
                pend = []
        if last:
            x = prog.comp(KC_NORM, 4 * b * h * M, deps=pend)
            x = prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            x = prog.comp(KC_LOSS, 4 * b * VOCAB / tp * M)
            prog.memcpy(4, deps=[x])
            prev = x
        act_out[mb] = prev

    def B(mb, last_mb):
        pend = [grad_in.get(mb)] if not last else []
        if last:
            prog.comp(KC_LOSS, 4 * b * VOCAB / tp * M, deps=pend)
            pend = []
            prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            g = prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            add_grad(h * VOCAB / tp, g, last_mb)
            prog.comp(KC_NORM, 6 * b * h * M)
        prev = None
        for _ in range(nl):
            for name, kc, work, params in bwd:
                if name == "AR":
                    if tp > 1:
                        pend = [tp_ar(prev)]
                    continue
                prev = prog.comp(kc, work, deps=pend)
                pend = []
                if params:
                    add_grad(params, prev, last_mb)
        if first:
            g = prog.comp(KC_EMB, 4 * b * h * M, deps=pend)
            add_grad(VOCAB * h / tp, g, last_mb)
            prev = g
        grad_out[mb] = prev
        if last_mb:
            flush_bucket(prev)

    def p2p(key, deps=()):
        return prog.comm(_E_P2P, act_bytes, CC_SENDRECV, ALGO_RING, key, deps=deps)

    # warm-up forwards
    for mb in range(W):
        if not first:
            act_in[mb] = p2p(("fa", p - 1, mb))
        F(mb)
        if not last:
            p2p(("fa", p, mb), deps=[act_out[mb]])
    if not first:
        act_in[W] = p2p(("fa", p - 1, W))
    # steady 1F1B
    for t in range(R):
        F(W + t)
        if not last:
            grad_in[t] = p2p(("pair", p, t), deps=[act_out[W + t]])
        B(t, t == m - 1)
        if not first:
            if t == R - 1:
                p2p(("g", p - 1, t), deps=[grad_out[t]])
            else:
                act_in[W + t + 1] = p2p(("pair", p - 1, t), deps=[grad_out[t]])
    # cool-down backwards
    for t in range(R, m):
        if not last:
            grad_in[t] = p2p(("g", p, t))
        B(t, t == m - 1)
        if not first:
            p2p(("g", p - 1, t), deps=[grad_out[t]])
    # gradient norm (waits for every gradient bucket), its all-reduce, optimizer
    gn = prog.comp(KC_ELEM, 4.0e5 * 20000.0, deps=dp_entries)
    n_params = nl * 12 * h * h / tp
    pend = [gn]
    if c.tp * c.pp * c.dp > 1:
        pend = [prog.comm(_E_WORLD, 4, CC_ALLREDUCE, ALGO_AUTO, None, deps=[gn])]
    for _ in range(3):
        prog.comp(KC_OPT, n_params * 16 / 3 * M, deps=pend)
        pend = []
    return prog


def _stage_program_interleaved(c: GPTConfig, p: int) -> _StageProgram:
    """Issue order of one rank of pipeline stage ``p`` under interleaved 1F1B: the
    rank holds v model chunks, chunk ch being virtual stage s = ch * PP + p of
    PP * v, each with layers / (PP * v) layers.  Virtual microbatch k runs
    microbatch (k // (PP * v)) * PP + k % PP on chunk (k // PP) % v (backwards
    take the chunks in reverse); a rank runs (PP - p - 1) * 2 + (v - 1) * PP
    forwards before its first backward (all of them when m == PP), then
    alternates.

    Every transfer between consecutive virtual stages is its own 2-member P2P
    node, keyed by ('fa' | 'g', lower physical stage, lower virtual stage,
    microbatch).  Sends and receives of activations and of gradients each take a
    timeline of their own (the schedule's batched asynchronous send/recv calls do
    not wait for one another), so every such timeline carries one link's transfers
    of one kind, which both ends issue in the same (forward or backward) order."""
    PP, m, tp, dp, v = c.pp, c.microbatches, c.tp, c.dp, c.virtual_stages
    if c.layers % (PP * v):
        raise ValueError("layers must divide evenly across the virtual pipeline stages")
    if m % PP:
        raise ValueError("interleaved 1F1B needs microbatches divisible by the pipeline stages")
    nl = c.layers // (PP * v)
    b, h = c.seq, c.hidden
    act_bytes = b * h * 2
    prog = _StageProgram()
    fwd = _fwd_kernels(c)
    bwd = _bwd_kernels(c)
    M = MEM_FLOP_PER_BYTE
    n_virtual = PP * v
    dp_entries: List[int] = []
    bucket = [0.0]
    act_out: Dict[Tuple[int, int], int] = {}

    def tp_ar(dep):
        return prog.comm(_E_TP, act_bytes, CC_ALLREDUCE, ALGO_AUTO, None, deps=[dep])

    def flush_bucket(dep):
        if dp > 1 and bucket[0] > 0:
            e = prog.comm(_E_DP, int(bucket[0]) * 2, CC_ALLREDUCE, ALGO_AUTO, len(dp_entries), deps=[dep])
            dp_entries.append(e)
        bucket[0] = 0.0

    def add_grad(params, dep, last_mb):
        if last_mb and dp > 1:
            bucket[0] += params
            if bucket[0] >= DP_BUCKET_ELEMS:
                flush_bucket(dep)

    def xfer(kind, s, mb, send, deps=()):
        et = {("fa", True): _E_P2P, ("fa", False): _E_P2P_RECV,
              ("g", True): _E_P2P_GRAD, ("g", False): _E_P2P_GRAD_RECV}[(kind, send)]
        return prog.comm(et, act_bytes, CC_SENDRECV, ALGO_RING, (kind, s % PP, s, mb), deps=deps)

    def F(mb, ch):
        s = ch * PP + p
        dep = xfer("fa", s - 1, mb, False) if s > 0 else None
        if s == 0:
            mc = prog.memcpy(b * 8)
            dep = prog.comp(KC_EMB, 4 * b * h * M, deps=[mc])
        pend = [dep]
        prev = dep
        for _ in range(nl):
            for name, kc, work in fwd:
                if name == "AR":
                    if tp > 1:
                        pend = [tp_ar(prev)]
                    continue
                prev = prog.comp(kc, work, deps=pend)
                pend = []
        if s == n_virtual - 1:
            x = prog.comp(KC_NORM, 4 * b * h * M, deps=pend)
            x = prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            x = prog.comp(KC_LOSS, 4 * b * VOCAB / tp * M)
            prog.memcpy(4, deps=[x])
            prev = x
        else:
            xfer("fa", s, mb, True, deps=[prev])
        act_out[(mb, ch)] = prev

    def B(mb, ch):
        s = ch * PP + p
        last_mb = mb == m - 1
        pend = [xfer("g", s, mb, False)] if s < n_virtual - 1 else []
        if s == n_virtual - 1:
            prog.comp(KC_LOSS, 4 * b * VOCAB / tp * M, deps=pend)
            pend = []
            prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            g = prog.comp(KC_GEMM, 2 * b * h * VOCAB / tp)
            add_grad(h * VOCAB / tp, g, last_mb)
            prog.comp(KC_NORM, 6 * b * h * M)
        prev = None
        for _ in range(nl):
            for name, kc, work, params in bwd:
                if name == "AR":
                    if tp > 1:
                        pend = [tp_ar(prev)]
                    continue
                prev = prog.comp(kc, work, deps=pend)
                pend = []
                if params:
                    add_grad(params, prev, last_mb)
        if s == 0:
            g = prog.comp(KC_EMB, 4 * b * h * M, deps=pend)
            add_grad(VOCAB * h / tp, g, last_mb)
            prev = g
        else:
            xfer("g", s - 1, mb, True, deps=[prev])
        if last_mb:
            flush_bucket(prev)

    total = m * v

    def mb_of(k):
        return (k // n_virtual) * PP + k % PP

    def chunk_of(k, forward):
        ch = (k % n_virtual) // PP
        return ch if forward else v - 1 - ch

    warm = total if m == PP else min((PP - p - 1) * 2 + (v - 1) * PP, total)
    kf = kb = 0
    for _ in range(warm):
        F(mb_of(kf), chunk_of(kf, True))
        kf += 1
    for _ in range(total - warm):
        F(mb_of(kf), chunk_of(kf, True))
        kf += 1
        B(mb_of(kb), chunk_of(kb, False))
        kb += 1
    while kb < total:
        B(mb_of(kb), chunk_of(kb, False))
        kb += 1
    gn = prog.comp(KC_ELEM, 4.0e5 * 20000.0, deps=dp_entries)
    n_params = nl * v * 12 * h * h / tp
    pend = [gn]
    if c.tp * c.pp * c.dp > 1:
        pend = [prog.comm(_E_WORLD, 4, CC_ALLREDUCE, ALGO_AUTO, None, deps=[gn])]
    for _ in range(3):
        prog.comp(KC_OPT, n_params * 16 / 3 * M, deps=pend)
        pend = []
    return prog


def _rank(c: GPTConfig, dp: int, p: int, t: int) -> int:
    return (dp * c.pp + p) * c.tp + t


def build_gpt_graph(c: GPTConfig) -> Graph:
    """Build the merged multi-rank execution graph of one training step."""
    TP, PP, DP = c.tp, c.pp, c.dp
    R = TP * PP * DP
    inter = c.virtual_stages > 1
    NS = N_STREAMS + 3 if inter else N_STREAMS
    progs = [(_stage_program_interleaved if inter else _stage_program)(c, p) for p in range(PP)]

    # P2P keys: every key must be issued by exactly the two adjacent stages
    p2p_keys: Dict[object, int] = {}
    p2p_seen: Dict[object, int] = {}
    for p, pr in enumerate(progs):
        for et, key in zip(pr.etype, pr.key):
            if et in _E_P2P_ALL:
                if key not in p2p_keys:
                    p2p_keys[key] = len(p2p_keys)
                p2p_seen[key] = p2p_seen.get(key, 0) + 1
    bad = [k for k, n in p2p_seen.items() if n != 2]
    if bad:
        raise RuntimeError(f"unmatched P2P calls: {bad[:4]}")

    # id blocks: per-rank local ops, TP all-reduces, P2P, DP all-reduces, world all-reduce
    next_id = 0
    loc_base, tp_base, dp_base = [], [], []
    for pr in progs:
        et = np.asarray(pr.etype)
        n_loc = int(((et == _E_COMP) | (et == _E_MEMCPY)).sum())
        loc_base.append((next_id, n_loc))
        next_id += n_loc * DP * TP
    for pr in progs:
        n_tp = int((np.asarray(pr.etype) == _E_TP).sum())
        tp_base.append(next_id)
        next_id += n_tp * DP
    p2p_base = next_id
    next_id += len(p2p_keys) * DP * TP
    for pr in progs:
        n_dp = int((np.asarray(pr.etype) == _E_DP).sum())
        dp_base.append(next_id)
        next_id += n_dp * TP
    world_id = -1
    if any(_E_WORLD in pr.etype for pr in progs):
        world_id = next_id
        next_id += 1
    V = next_id

    # groups
    g_tp = 0
    n_tpg = DP * PP if TP > 1 else 0
    g_p2p = g_tp + n_tpg
    n_links = PP if inter else PP - 1  # interleaved: also the last stage -> the first
    n_p2pg = n_links * DP * TP
    g_dp = g_p2p + n_p2pg
    n_dpg = PP * TP if DP > 1 else 0
    g_world = g_dp + n_dpg
    n_groups = g_world + (1 if world_id >= 0 else 0)
    members: List[np.ndarray] = []
    for d in range(DP):
        for p in range(PP):
            if TP > 1:
                members.append(np.array([_rank(c, d, p, t) for t in range(TP)], np.int32))
    for bb in range(n_links):
        for d in range(DP):
            for t in range(TP):
                members.append(np.array(sorted([_rank(c, d, bb, t), _rank(c, d, (bb + 1) % PP, t)]), np.int32))
    if DP > 1:
        for p in range(PP):
            for t in range(TP):
                members.append(np.array([_rank(c, d, p, t) for d in range(DP)], np.int32))
    if world_id >= 0:
        members.append(np.arange(R, dtype=np.int32))
    assert len(members) == n_groups
    grp_off = np.zeros(n_groups + 1, np.int64)
    grp_off[1:] = np.cumsum([len(x) for x in members])
    grp_rank = np.concatenate(members) if members else np.zeros(0, np.int32)

    kind = np.zeros(V, np.uint8)
    kclass = np.zeros(V, np.uint8)
    group = np.full(V, -1, np.int32)
    cc_type = np.zeros(V, np.uint8)
    cc_algo = np.zeros(V, np.uint8)
    cc_bytes = np.zeros(V, np.int64)
    work = np.zeros(V, np.float64)

    dpv = np.repeat(np.arange(DP), TP)          # rank-of-stage -> dp
    tpv = np.tile(np.arange(TP), DP)            # rank-of-stage -> tp
    srcs, dsts = [], []
    queues: Dict[int, np.ndarray] = {}
    for p, pr in enumerate(progs):
        et = np.asarray(pr.etype)
        n = len(et)
        base = np.zeros(n, np.int64)
        mdp = np.zeros(n, np.int64)
        mtp = np.zeros(n, np.int64)
        lb, n_loc = loc_base[p]
        loc = (et == _E_COMP) | (et == _E_MEMCPY)
        li = np.cumsum(loc) - 1
        base[loc] = lb + li[loc]
        mdp[loc] = TP * n_loc
        mtp[loc] = n_loc
        tpm = et == _E_TP
        ti = np.cumsum(tpm) - 1
        base[tpm] = tp_base[p] + ti[tpm] * DP
        mdp[tpm] = 1
        p2m = np.isin(et, _E_P2P_ALL)
        kidx = np.array([p2p_keys[k] if e in _E_P2P_ALL else 0 for e, k in zip(pr.etype, pr.key)], np.int64)
        base[p2m] = p2p_base + kidx[p2m] * DP * TP
        mdp[p2m] = TP
        mtp[p2m] = 1
        dpm = et == _E_DP
        di = np.cumsum(dpm) - 1
        base[dpm] = dp_base[p] + di[dpm] * TP
        mtp[dpm] = 1
        wm = et == _E_WORLD
        base[wm] = world_id
        ids = base[None, :] + dpv[:, None] * mdp[None, :] + tpv[:, None] * mtp[None, :]  # [DP*TP, n]

        # attributes (identical for every instance of an entry)
        kcl = np.asarray(pr.kclass, np.uint8)
        wk = np.asarray(pr.work, np.float64)
        nb = np.asarray(pr.nbytes, np.int64)
        cct = np.asarray(pr.cctype, np.uint8)
        alg = np.asarray(pr.algo, np.uint8)
        ekind = np.where(et == _E_COMP, KIND_COMPUTE,
                         np.where(et == _E_MEMCPY, KIND_MEMCPY,
                                  np.where(p2m, KIND_P2P, KIND_COLL))).astype(np.uint8)
        flat = ids.reshape(-1)
        kind[flat] = np.tile(ekind, DP * TP)
        kclass[flat] = np.tile(kcl, DP * TP)
        work[flat] = np.tile(wk, DP * TP)
        cc_bytes[flat] = np.tile(nb, DP * TP)
        cc_type[flat] = np.tile(cct, DP * TP)
        cc_algo[flat] = np.tile(alg, DP * TP)
        # groups of comm instances
        grp = np.full(ids.shape, -1, np.int64)
        grp[:, tpm] = g_tp + (dpv[:, None] * PP + p)
        grp[:, p2m] = g_p2p + ((np.array([pr.key[i][1] for i in np.nonzero(p2m)[0]], np.int64)[None, :]
                                * DP + dpv[:, None]) * TP + tpv[:, None]) if p2m.any() else 0
        grp[:, dpm] = g_dp + p * TP + tpv[:, None]
        grp[:, wm] = g_world
        comm_mask = tpm | p2m | dpm | wm
        group[ids[:, comm_mask].reshape(-1)] = grp[:, comm_mask].reshape(-1)

        # program order per stream
        lanes = ((STREAM_COMPUTE, et == _E_COMP), (STREAM_TP, tpm), (STREAM_PP, et == _E_P2P),
                 (STREAM_DP, dpm | wm), (STREAM_MEMCPY, et == _E_MEMCPY))
        if inter:
            lanes += ((STREAM_PP_RECV, et == _E_P2P_RECV), (STREAM_PP_GRAD, et == _E_P2P_GRAD),
                      (STREAM_PP_GRAD_RECV, et == _E_P2P_GRAD_RECV))
        for stream, mask in lanes:
            sel = ids[:, mask]
            for j in range(DP * TP):
                r = _rank(c, int(dpv[j]), p, int(tpv[j]))
                queues[r * NS + stream] = sel[j]
        # data edges
        if pr.src:
            s_e = np.asarray(pr.src, np.int64)
            d_e = np.asarray(pr.dst, np.int64)
            srcs.append(ids[:, s_e].reshape(-1))
            dsts.append(ids[:, d_e].reshape(-1))

    nq = R * NS
    q_lens = [len(queues.get(q, ())) for q in range(nq)]
    q_off = np.zeros(nq + 1, np.int64)
    q_off[1:] = np.cumsum(q_lens)
    q_ops = np.concatenate([queues.get(q, np.zeros(0, np.int64)) for q in range(nq)]).astype(np.int32)

    src = np.concatenate(srcs) if srcs else np.zeros(0, np.int64)
    dst = np.concatenate(dsts) if dsts else np.zeros(0, np.int64)
    key = np.unique(dst * V + src)
    dst, src = key // V, key % V
    pred_off = np.zeros(V + 1, np.int64)
    np.add.at(pred_off, dst + 1, 1)
    pred_off = np.cumsum(pred_off)
    pred_idx = src.astype(np.int32)

    rng = np.random.Generator(np.random.PCG64(c.graph_seed))
    noise = np.exp(rng.normal(0.0, 0.1, size=V))
    replica_of = None
    if c.identical_replicas and DP > 1:
        # rank (dp, p, t) mirrors rank (0, p, t): the op at each timeline position of a
        # replica takes the noise of the op at the same position of replica 0
        replica_of = (np.arange(R) % (PP * TP)).astype(np.int32)
        orig = np.arange(V)
        for q in range(nq):
            r, k = divmod(q, NS)
            qa = int(replica_of[r]) * NS + k
            if qa != q:
                orig[q_ops[q_off[q]:q_off[q + 1]]] = q_ops[q_off[qa]:q_off[qa + 1]]
        noise = noise[orig]
    g = Graph(R, NS, c.gpus_per_node, kind, kclass, group, cc_type, cc_algo, cc_bytes,
              pred_off, pred_idx, q_off, q_ops, grp_off, grp_rank.astype(np.int32), work, noise,
              name=c.name, replica_of=replica_of)
    return g


# ---------------------------------------------------------------------------------------
# scenarios
# ---------------------------------------------------------------------------------------
def scenario_params(c: GPTConfig, n_scen: Optional[int] = None) -> Scenarios:
    """Per-scenario parameters, without the duration matrix (``dur`` left empty)."""
    S = c.n_scen if n_scen is None else n_scen
    if c.fixed_scenario:
        peak = np.full(S, 4.0e5)
        bwa = np.full(S, NVLINK_GBS)
        bwe = np.full(S, IB_GBS)
        sf = np.full((N_KCLASS, S), 1.2)
    else:
        rng = np.random.Generator(np.random.PCG64(c.scen_seed))
        peak = rng.uniform(300.0, 1000.0, size=S) * 1.0e3     # TFLOP/s -> FLOP/ns
        bwa = rng.uniform(25.0, 900.0, size=S)
        bwe = bwa / 8.0
        sf = rng.uniform(1.0, 1.4, size=(N_KCLASS, S))
    return Scenarios(
        dur=np.zeros((0, S), np.int64),
        alpha_ns=np.full(S, ALPHA_NS), bw_intra=bwa, lat_intra=np.full(S, NVLINK_LAT_NS),
        bw_inter=bwe, lat_inter=np.full(S, IB_LAT_NS), delta=np.full(S, DELTA_NS_PER_B),
        slowdown=np.ascontiguousarray(sf), peak_flop_per_ns=peak)


def durations(g: Graph, peak_flop_per_ns: np.ndarray, out: Optional[np.ndarray] = None,
              chunk_rows: int = 1 << 16) -> np.ndarray:
    """d(v, s) = rint(work_v / P_s * n_v) for compute and memcpy ops, 0 for comm ops."""
    V, S = g.n_ops, int(peak_flop_per_ns.shape[0])
    if out is None:
        out = np.empty((V, S), np.int64)
    local = (g.kind == KIND_COMPUTE) | (g.kind == KIND_MEMCPY)
    P = np.asarray(peak_flop_per_ns, np.float64)[None, :]
    for r0 in range(0, V, chunk_rows):
        r1 = min(V, r0 + chunk_rows)
        x = (g.work[r0:r1, None] / P) * g.noise[r0:r1, None]
        np.rint(x, out=x)
        x[~local[r0:r1]] = 0.0
        out[r0:r1] = x.astype(np.int64)
    return out


def make_scenarios(g: Graph, c: GPTConfig, n_scen: Optional[int] = None,
                   dur_out: Optional[np.ndarray] = None) -> Scenarios:
    sc = scenario_params(c, n_scen)
    sc.dur = durations(g, sc.peak_flop_per_ns, out=dur_out)
    return sc


def select_scenarios(sc: Scenarios, g: Graph, cols) -> Scenarios:
    """The scenarios ``cols`` of ``sc`` (durations recomputed from the recipe)."""
    cols = np.asarray(cols, np.int64)
    out = Scenarios(dur=np.zeros((0, len(cols)), np.int64),
                    alpha_ns=sc.alpha_ns[cols].copy(), bw_intra=sc.bw_intra[cols].copy(),
                    lat_intra=sc.lat_intra[cols].copy(), bw_inter=sc.bw_inter[cols].copy(),
                    lat_inter=sc.lat_inter[cols].copy(), delta=sc.delta[cols].copy(),
                    slowdown=np.ascontiguousarray(sc.slowdown[:, cols]),
                    peak_flop_per_ns=sc.peak_flop_per_ns[cols].copy(),
                    chunk_max_bytes=sc.chunk_max_bytes, chunk_bytes=sc.chunk_bytes)
    out.dur = durations(g, out.peak_flop_per_ns)
    return out


# ---------------------------------------------------------------------------------------
# standalone CC-estimator queries
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass
class CCQueries:
    cc_type: np.ndarray     # uint8 [Q]
    cc_algo: np.ndarray     # uint8 [Q]
    nbytes: np.ndarray      # int64 [Q]
    n_ranks: np.ndarray     # int32 [Q]
    n_nodes: np.ndarray     # int32 [Q]
    alpha_ns: np.ndarray
    bw_intra: np.ndarray
    lat_intra: np.ndarray
    bw_inter: np.ndarray
    lat_inter: np.ndarray
    delta: np.ndarray

    @property
    def n(self) -> int:
        return int(self.cc_type.shape[0])


def make_cc_queries(n: int = 1_000_000, seed: int = 1005, gpus_per_node: int = 8) -> CCQueries:
    """Queries over {AR, AG, RS, send/recv} x log-uniform 1 KB..4 GB x group sizes
    {2^k, 3*2^k} in [2, 1024], spread over ceil(N/8) nodes; links drawn as for the
    GPT-1.3B batch.  Send/recv queries have N = 2 on one or two nodes."""
    rng = np.random.Generator(np.random.PCG64(seed))
    sizes = sorted({2 ** k for k in range(1, 11)} | {3 * 2 ** k for k in range(0, 9) if 3 * 2 ** k <= 1024})
    sizes = np.array(sizes, np.int32)
    t = rng.integers(0, 4, size=n).astype(np.uint8)
    algo = np.where(t == CC_ALLREDUCE, rng.integers(0, 3, size=n), ALGO_RING).astype(np.uint8)
    nbytes = np.rint(np.exp(rng.uniform(math.log(1024.0), math.log(4.0 * 2 ** 30), size=n))).astype(np.int64)
    N = sizes[rng.integers(0, len(sizes), size=n)]
    M = ((N + gpus_per_node - 1) // gpus_per_node).astype(np.int32)
    sr = t == CC_SENDRECV
    N = np.where(sr, 2, N).astype(np.int32)
    M = np.where(sr, rng.integers(1, 3, size=n), M).astype(np.int32)
    bwa = rng.uniform(25.0, 900.0, size=n)
    return CCQueries(t, algo, nbytes, N, M,
                     np.full(n, ALPHA_NS), bwa, np.full(n, NVLINK_LAT_NS), bwa / 8.0,
                     np.full(n, IB_LAT_NS), np.full(n, DELTA_NS_PER_B))


def config(name: str) -> GPTConfig:
    return CONFIGS[name]
