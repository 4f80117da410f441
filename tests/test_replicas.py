"""Replica folding on the host (no GPU): the premise, checked with the oracle, and
the checks of replica_of.

The premise of folding (the DDP single copy of Sec. 8.5, generalised): when the
replicas of a DP group run identical kernels, the full graph's composition gives
every replica op the times of its original, so composing the originals suffices.
The oracle composes the full graph; nothing here shares code with the library's
folding.
"""
import dataclasses

import numpy as np
import pytest

import oracle
from paper_2412_12487_gb300 import EchoError
from paper_2412_12487_gb300 import echo as E
from paper_2412_12487_gb300 import workloads as W
from tests import smallgraphs as SG


def _identical(name, **kw):
    c = dataclasses.replace(W.config(name), identical_replicas=True, **kw)
    return c, W.build_gpt_graph(c)


def originals(g):
    """op -> the op at the same timeline position of its rank's representative."""
    orig = np.arange(g.n_ops)
    for q in range(len(g.q_off) - 1):
        r, k = divmod(q, g.n_streams)
        qa = int(g.replica_of[r]) * g.n_streams + k
        if qa != q:
            orig[g.q_ops[g.q_off[q]:g.q_off[q + 1]]] = g.q_ops[g.q_off[qa]:g.q_off[qa + 1]]
    return orig


def test_identical_replicas_compose_symmetrically():
    c, g = _identical("tiny", fixed_scenario=False)
    sc = W.make_scenarios(g, c, n_scen=5)
    orig = originals(g)
    assert (orig != np.arange(g.n_ops)).sum() > g.n_ops // 3
    local = (g.kind == W.KIND_COMPUTE) | (g.kind == W.KIND_MEMCPY)
    assert np.array_equal(sc.dur[local], sc.dur[orig[local]])
    for civ in (0, 1):
        for model in (0, 1):
            r = oracle.compose(g, sc, refine_passes=2, overlap_model=model, comm_interval=civ)
            assert np.array_equal(r.finish, r.finish[orig])
            assert np.array_equal(r.start, r.start[orig])
            assert np.array_equal(r.overlapped, r.overlapped[orig])
            assert r.overlapped.any()


def test_folded_op_counts():
    _, g = _identical("tiny")
    assert E.check_replicas(g) == 439 and g.n_ops == 873
    _, g = _identical("gpt1.3b")
    # 8 identical replicas: each replica's own ops once, the DP and world all-reduces once
    orig = originals(g)
    assert E.check_replicas(g) == len(np.unique(orig)) == 17967
    g.replica_of = None
    assert E.check_replicas(g) == g.n_ops
    g.replica_of = np.arange(g.n_ranks, dtype=np.int32)
    assert E.check_replicas(g) == g.n_ops


def _rejected(g, code="ECHO_E_BAD_GRAPH"):
    with pytest.raises(EchoError) as ei:
        E.check_replicas(g)
    assert code in str(ei.value)


def test_replica_of_must_name_representatives():
    _, g = _identical("tiny")
    bad = g.replica_of.copy()
    bad[3] = g.n_ranks
    g2 = dataclasses.replace(g, replica_of=bad)
    _rejected(g2, "ECHO_E_INVALID_ARG")
    bad = g.replica_of.copy()
    r = int(np.nonzero(bad != np.arange(g.n_ranks))[0][0])  # a replica rank
    bad[0] = r                                             # mirrors a replica
    _rejected(dataclasses.replace(g, replica_of=bad))


def test_replica_that_differs_is_rejected():
    _, g = _identical("tiny")
    orig = originals(g)
    x = int(np.nonzero((orig != np.arange(g.n_ops)) & (g.kind == W.KIND_COMPUTE))[0][5])
    kc = g.kclass.copy()
    kc[x] = (kc[x] + 1) % W.N_KCLASS
    _rejected(dataclasses.replace(g, kclass=kc))
    # a replica op that loses one of its producers
    y = int(np.nonzero((orig != np.arange(g.n_ops)) & (np.diff(g.pred_off) > 0))[0][3])
    keep = np.ones(len(g.pred_idx), bool)
    keep[g.pred_off[y]] = False
    po = g.pred_off.copy()
    po[y + 1:] -= 1
    _rejected(dataclasses.replace(g, pred_off=po, pred_idx=g.pred_idx[keep]))


def _pair(mirror_launch=True, extra=False):
    """Ranks 0 and 1 (1 mirrors 0): kernels a0 / a1, then an all-reduce shared by
    both ranks; rank 0 launches it after a0, rank 1 after a1 unless mirror_launch is
    off.  extra adds a kernel to rank 1 only."""
    ops = [{"kind": W.KIND_COMPUTE, "kclass": 0}, {"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE, "cc_bytes": 1000,
            "preds": [0, 1] if mirror_launch else [0]}]
    queues = {(0, 0): [0], (1, 0): [1], (0, 1): [2], (1, 1): [2]}
    if extra:
        ops.append({"kind": W.KIND_COMPUTE, "kclass": 0})
        queues[(1, 0)] = [1, 3]
    g = SG.graph_from_lists(2, 2, ops, queues, [[0, 1]], gpus_per_node=2)
    g.replica_of = np.array([0, 0], np.int32)
    return g


def test_hand_built_pair():
    assert E.check_replicas(_pair()) == 2  # a0 and the all-reduce
    _rejected(_pair(mirror_launch=False))  # rank 1 would launch at 0, rank 0 after a0
    _rejected(_pair(extra=True))           # timelines of different lengths


def test_folding_interleaved_schedules():
    # 8 timelines per rank and lone transfers between virtual stages: replicas of a
    # DP group still mirror each other, and the oracle composes them symmetrically
    c = W.GPTConfig("i-L8-pp2-m2-v2-dp2", 8, 512, 8, 256, 2, 2, 2, 2, 3, virtual_stages=2,
                    identical_replicas=True)
    g = W.build_gpt_graph(c)
    assert g.n_streams == 8
    orig = originals(g)
    assert E.check_replicas(g) == len(np.unique(orig)) < g.n_ops
    sc = W.make_scenarios(g, c)
    r = oracle.compose(g, sc, refine_passes=1, comm_interval=1)
    assert np.array_equal(r.finish, r.finish[orig]) and np.array_equal(r.overlapped, r.overlapped[orig])
