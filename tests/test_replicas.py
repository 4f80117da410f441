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


def _replicate(rng, g0, sc0):
    """Two replicas of random graph g0 (ranks r and r + H, H = R0 rounded up to whole
    nodes, so that every copied group spans the same node layout).  Some collectives become
    one op shared by both replicas (members of both copies, producers of both), the
    rest are copied.  Returns the graph with replica_of, its scenarios, and for each
    op of g0 its (replica 0, replica 1) ids."""
    R0, NS, V0 = g0.n_ranks, g0.n_streams, g0.n_ops
    H = -(-R0 // g0.gpus_per_node) * g0.gpus_per_node
    comm = (g0.kind == W.KIND_COLL)
    shared = comm & (rng.random(V0) < 0.5)
    ids = np.zeros((V0, 2), np.int64)
    ops = []
    for v in range(V0):
        base = {"kind": int(g0.kind[v]), "kclass": int(g0.kclass[v]), "cc_type": int(g0.cc_type[v]),
                "cc_algo": int(g0.cc_algo[v]), "cc_bytes": int(g0.cc_bytes[v])}
        for rep in ((0,) if shared[v] else (0, 1)):
            ids[v, rep] = len(ops)
            ops.append(dict(base, rep=rep, orig=v))
        if shared[v]:
            ids[v, 1] = ids[v, 0]
    groups, gmap = [], {}
    for o in ops:
        v = o["orig"]
        if g0.kind[v] in (W.KIND_COLL, W.KIND_P2P):
            mem = g0.grp_rank[g0.grp_off[g0.group[v]]:g0.grp_off[g0.group[v] + 1]].tolist()
            m = sorted(mem + [x + H for x in mem]) if shared[v] else sorted(x + H * o["rep"] for x in mem)
            o["group"] = gmap.setdefault(tuple(m), len(groups))
            if o["group"] == len(groups):
                groups.append(m)
        preds = g0.pred_idx[g0.pred_off[v]:g0.pred_off[v + 1]].tolist()
        reps = (0, 1) if shared[v] else (o["rep"],)
        o["preds"] = sorted({int(ids[u, rp]) for u in preds for rp in reps})
    queues = {}
    for q in range(R0 * NS):
        r, k = divmod(q, NS)
        lst = g0.q_ops[g0.q_off[q]:g0.q_off[q + 1]].tolist()
        queues[(r, k)] = [int(ids[v, 0]) for v in lst]
        queues[(r + H, k)] = [int(ids[v, 1]) for v in lst]
    g = SG.graph_from_lists(2 * H, NS, ops, queues, groups, gpus_per_node=g0.gpus_per_node)
    g.replica_of = np.concatenate([np.arange(H), np.arange(R0), np.arange(R0, H)]).astype(np.int32)
    dur = np.zeros((len(ops), sc0.n_scen), np.int64)
    for v in range(V0):
        dur[ids[v, 0]] = sc0.dur[v]
        dur[ids[v, 1]] = sc0.dur[v]
    sc = W.Scenarios(dur=dur, alpha_ns=sc0.alpha_ns, bw_intra=sc0.bw_intra, lat_intra=sc0.lat_intra,
                     bw_inter=sc0.bw_inter, lat_inter=sc0.lat_inter, delta=sc0.delta,
                     slowdown=sc0.slowdown, peak_flop_per_ns=sc0.peak_flop_per_ns)
    return g, sc, ids


def test_folding_random_replicated_graphs():
    # random graphs in two replicas, some collectives shared by both: the host check
    # folds them back to the original op count, and the oracle's composition of the
    # full graph gives every copy its original's times
    rng = np.random.default_rng(808)
    folded = 0
    for case in range(60):
        g0 = SG.random_graph(rng, int(rng.integers(2, 40)), max_ranks=3, max_streams=4, p_edge=0.1)
        sc0 = SG.random_scenarios(rng, g0, 3, max_dur=40)
        g, sc, ids = _replicate(rng, g0, sc0)
        assert E.check_replicas(g) == g0.n_ops, case
        folded += g.n_ops > g0.n_ops
        for civ in (0, 1):
            r = oracle.compose(g, sc, refine_passes=2, comm_interval=civ)
            assert np.array_equal(r.finish[ids[:, 0]], r.finish[ids[:, 1]]), case
            assert np.array_equal(r.overlapped[ids[:, 0]], r.overlapped[ids[:, 1]]), case
    assert folded > 40
