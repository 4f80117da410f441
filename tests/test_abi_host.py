"""CPU tests of the C ABI library: it loads, exports every symbol the header
declares, and its host-side validation and levelling (echo_check_graph, which
needs no device) accept the generated workloads and reject malformed graphs with
the documented status codes."""
import copy
import os
import re

import numpy as np
import pytest

from paper_2412_12487_gb300 import EchoError, check_graph
from paper_2412_12487_gb300 import build as B
from paper_2412_12487_gb300 import echo as E
from paper_2412_12487_gb300 import workloads as W
from tests import smallgraphs as SG

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()
    E.load_library()


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "echo.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(echo_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_function():
    import ctypes
    lib = ctypes.CDLL(B.LIB)
    declared = _declared_functions()
    assert len(declared) >= 15
    for name in declared:
        assert hasattr(lib, name), name
    assert sorted(E.EXPORTS) == declared


def _levels_reference(g):
    preds = SG.merged_preds(g)
    depth = [0] * g.n_ops
    order = np.argsort(np.zeros(g.n_ops))  # placeholder, filled below
    # repeated relaxation in a topological order found by DFS
    seen, topo = [0] * g.n_ops, []

    def visit(v):
        stack = [(v, 0)]
        while stack:
            u, i = stack.pop()
            if i == 0:
                if seen[u]:
                    continue
                seen[u] = 1
            if i < len(preds[u]):
                stack.append((u, i + 1))
                if not seen[preds[u][i]]:
                    stack.append((preds[u][i], 0))
            else:
                topo.append(u)

    for v in range(g.n_ops):
        visit(v)
    for v in topo:
        depth[v] = max([depth[u] + 1 for u in preds[v]], default=0)
    del order
    if not g.n_ops:
        return 0, 0
    L = max(depth) + 1
    return L, int(np.bincount(depth).max())


@pytest.mark.parametrize("name", ["tiny", "gpt1.3b"])
def test_levelling_of_generated_workloads(name):
    g = W.build_gpt_graph(W.config(name))
    assert check_graph(g) == _levels_reference(g)


def test_levelling_of_random_graphs():
    rng = np.random.default_rng(5)
    for _ in range(300):
        g = SG.random_graph(rng, int(rng.integers(0, 40)), max_ranks=4, max_streams=4)
        assert check_graph(g) == _levels_reference(g)


def _tiny():
    return W.build_gpt_graph(W.config("tiny"))


def _expect(g, code):
    with pytest.raises(EchoError) as ei:
        check_graph(g)
    assert ei.value.code == code, str(ei.value)


def test_rejects_cycles():
    g = _tiny()
    # make the first op of rank 0's compute timeline wait for its last
    q = g.q_ops[g.q_off[0]:g.q_off[1]]
    first, last = int(q[0]), int(q[-1])
    g2 = copy.deepcopy(g)
    preds = [list(g.pred_idx[g.pred_off[v]:g.pred_off[v + 1]]) for v in range(g.n_ops)]
    preds[first].append(last)
    g2.pred_off = np.concatenate([[0], np.cumsum([len(p) for p in preds])]).astype(np.int64)
    g2.pred_idx = np.concatenate([np.array(p, np.int32) for p in preds]).astype(np.int32)
    _expect(g2, 3)
    g3 = copy.deepcopy(g)
    v = int(np.nonzero(np.diff(g.pred_off) > 0)[0][0])
    g3.pred_idx[g.pred_off[v]] = v  # self loop
    _expect(g3, 3)


def test_rejects_malformed_graphs():
    g = _tiny()
    bad = copy.deepcopy(g)
    bad.pred_idx[0] = g.n_ops  # predecessor out of range
    _expect(bad, 2)
    bad = copy.deepcopy(g)
    bad.kind[int(g.q_ops[g.q_off[0]])] = W.KIND_MEMCPY  # memcpy op on a compute timeline
    _expect(bad, 2)
    bad = copy.deepcopy(g)
    comm = int(np.nonzero(g.kind == W.KIND_COLL)[0][0])
    bad.group[comm] = g.n_groups  # group out of range
    _expect(bad, 2)
    bad = copy.deepcopy(g)
    bad.grp_rank[0] = g.n_ranks  # member rank out of range
    _expect(bad, 2)
    bad = copy.deepcopy(g)
    bad.cc_bytes[comm] = -1
    _expect(bad, 1)
    bad = copy.deepcopy(g)
    bad.kclass[int(np.nonzero(g.kind == W.KIND_COMPUTE)[0][0])] = 255
    _expect(bad, 2)
    bad = copy.deepcopy(g)
    bad.n_streams = 17
    _expect(bad, 9)
    bad = copy.deepcopy(g)
    p2p = int(np.nonzero(g.kind == W.KIND_P2P)[0][0])
    bad.cc_type[p2p] = W.CC_ALLREDUCE
    _expect(bad, 2)


def test_rejects_comm_op_missing_on_a_member():
    g = _tiny()
    comm = int(np.nonzero(g.kind == W.KIND_COLL)[0][0])
    keep = np.ones(g.q_ops.shape[0], bool)
    keep[int(np.nonzero(g.q_ops == comm)[0][0])] = False
    qid = np.repeat(np.arange(len(g.q_off) - 1), np.diff(g.q_off))
    bad = copy.deepcopy(g)
    bad.q_ops = g.q_ops[keep]
    bad.q_off = np.concatenate([[0], np.cumsum(np.bincount(qid[keep], minlength=len(g.q_off) - 1))]).astype(np.int64)
    _expect(bad, 2)


def test_rejects_comm_op_on_a_non_member():
    ops = [{"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE, "cc_bytes": 8}]
    g = SG.graph_from_lists(3, 2, ops, {(0, 1): [0], (2, 1): [0]}, [[0, 1]])
    _expect(g, 2)
    g = SG.graph_from_lists(3, 2, ops, {(0, 1): [0], (1, 1): [0]}, [[0, 1]])
    assert check_graph(g) == (1, 1)


def test_p2p_group_of_three_is_rejected():
    ops = [{"kind": W.KIND_P2P, "group": 0, "cc_type": W.CC_SENDRECV, "cc_bytes": 8}]
    g = SG.graph_from_lists(3, 2, ops, {(0, 1): [0], (1, 1): [0], (2, 1): [0]}, [[0, 1, 2]])
    _expect(g, 2)


def test_empty_graph_is_valid():
    g = SG.graph_from_lists(2, 3, [], {}, [])
    assert check_graph(g) == (0, 0)


def _interleaved(L=16, PP=4, m=4, v=2, tp=2, dp=2, hidden=512, seq=256):
    return W.GPTConfig(f"i-L{L}-pp{PP}-m{m}-v{v}", L, hidden, 8, seq, tp, PP, dp, m, 3, virtual_stages=v)


@pytest.mark.parametrize("shape", [(8, 2, 4, 2), (16, 4, 4, 2), (24, 4, 8, 3), (8, 2, 2, 2)])
def test_interleaved_schedule_graphs(shape):
    # interleaved 1F1B: a valid (acyclic) graph with the same compute work as 1F1B
    # and one activation and one gradient transfer per microbatch between
    # consecutive virtual stages
    L, PP, m, v = shape
    c = _interleaved(L, PP, m, v)
    g = W.build_gpt_graph(c)
    assert g.n_streams == 8
    assert check_graph(g) == _levels_reference(g)
    g1 = W.build_gpt_graph(W.GPTConfig(**{**c.__dict__, "virtual_stages": 1}))
    comp = g.kind == W.KIND_COMPUTE
    comp1 = g1.kind == W.KIND_COMPUTE
    assert comp.sum() == comp1.sum() and np.isclose(g.work[comp].sum(), g1.work[comp1].sum())
    # one activation and one gradient transfer per microbatch between consecutive virtual stages
    p2p = g.kind == W.KIND_P2P
    assert p2p.sum() == 2 * c.microbatches * (PP * v - 1) * c.dp * c.tp


def test_interleaving_shortens_a_compute_bound_pipeline():
    # with compute dominating (large hidden size), interleaving cuts the pipeline
    # bubble: the step is shorter than under 1F1B
    import oracle
    c = _interleaved(L=16, PP=4, m=4, v=2, tp=1, dp=1, hidden=8192, seq=2048)
    c = W.GPTConfig(**{**c.__dict__, "fixed_scenario": True, "n_scen": 1})
    c1 = W.GPTConfig(**{**c.__dict__, "virtual_stages": 1})
    mk = []
    for cc in (c, c1):
        g = W.build_gpt_graph(cc)
        mk.append(int(oracle.compose(g, W.make_scenarios(g, cc), refine_passes=0).makespan[0]))
    assert mk[0] < mk[1], mk
