"""GPU parity of replica folding: the library composes the folded graph and must
reproduce, bit for bit, the oracle's composition of the FULL graph, for every op
(a replica op reports its original's times).  A scenario batch whose replicas
differ runs the full graph, and the next identical batch folds again."""
import dataclasses
import os

import numpy as np
import pytest

import oracle
from paper_2412_12487_gb300 import Echo
from paper_2412_12487_gb300.echo import check_replicas
from paper_2412_12487_gb300 import workloads as W
from tests.test_gpu_parity import assert_same
from tests.test_replicas import originals

pytestmark = pytest.mark.gpu
THREADS = max(1, min(16, os.cpu_count() or 1))


def _compose(e, g, sc, refine=1, overlap_model=0, comm_interval=0, dur=None):
    e.load_scenarios(sc, dur=dur)
    e.estimate_collectives()
    e.compose(refine_passes=refine, overlap_model=overlap_model, comm_interval=comm_interval)
    st, fn = e.read_times()
    return dict(start=st, finish=fn, makespan=e.read_makespan(), cc=e.read_cc(), ov=e.read_overlap(),
                info=e.info())


@pytest.mark.parametrize("name,n_scen", [("tiny", 7), ("gpt1.3b", 24)])
def test_folded_replicas_match_the_full_graph(name, n_scen):
    c = dataclasses.replace(W.config(name), identical_replicas=True, fixed_scenario=False)
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=n_scen)
    with Echo(0) as e:
        e.load_graph(g)
        for refine, model, civ in ((1, 0, 0), (2, 1, 1), (1, 0, 1)):
            got = _compose(e, g, sc, refine, model, civ)
            assert got["info"]["replicas_folded"] == 1
            assert got["info"]["n_ops_composed"] == check_replicas(g) < g.n_ops
            want = oracle.compose(g, sc, refine_passes=refine, overlap_model=model, comm_interval=civ,
                                  threads=THREADS)
            assert_same(got, want, g, refine)
        # int32 durations take the same path
        got = _compose(e, g, sc, dur=sc.dur.astype(np.int32))
        assert got["info"]["replicas_folded"] == 1
        assert_same(got, oracle.compose(g, sc, threads=THREADS), g, 1)


def test_differing_replicas_run_the_full_graph():
    c = dataclasses.replace(W.config("gpt1.3b"), identical_replicas=True, fixed_scenario=False)
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=9)
    orig = originals(g)
    x = int(np.nonzero((orig != np.arange(g.n_ops)) & (g.kind == W.KIND_COMPUTE))[0][-100])
    bumped = dataclasses.replace(sc, dur=sc.dur.copy())
    bumped.dur[x, 4] += 1  # one replica kernel, one scenario
    with Echo(0) as e:
        e.load_graph(g)
        for s, folded in ((sc, 1), (bumped, 0), (sc, 1), (bumped, 0)):
            got = _compose(e, g, s)
            assert got["info"]["replicas_folded"] == folded
            assert_same(got, oracle.compose(g, s, threads=THREADS), g, 1)
