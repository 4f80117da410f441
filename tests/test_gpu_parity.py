"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Timelines are int64 ns and must match bit for bit; CC estimates are fp64 and must
agree within 1e-9 relative (the build evaluates the same closed forms with
explicit round-to-nearest operations, so in practice they are identical).
"""
import os

import numpy as np
import pytest

import oracle
from paper_2412_12487_gb300 import Echo, EchoError
from paper_2412_12487_gb300 import workloads as W
from tests import smallgraphs as SG

pytestmark = pytest.mark.gpu
CC_RTOL = 1e-9
THREADS = max(1, min(16, os.cpu_count() or 1))


def run_gpu(g, sc, refine=1, ctx=None, overlap_model=0, comm_interval=0, ar_algo_policy=0):
    e = ctx or Echo(0)
    try:
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=refine, overlap_model=overlap_model, comm_interval=comm_interval,
                  ar_algo_policy=ar_algo_policy)
        st, fn = e.read_times()
        return dict(start=st, finish=fn, makespan=e.read_makespan(), cc=e.read_cc(),
                    ov=e.read_overlap(), info=e.info())
    finally:
        if ctx is None:
            e.close()


def assert_same(got, want, g, refine=1):
    assert np.array_equal(got["finish"], want.finish)
    assert np.array_equal(got["start"], want.start)
    assert np.array_equal(got["makespan"], want.makespan)
    comm = (g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P)
    assert np.isnan(got["cc"][~comm]).all()
    np.testing.assert_allclose(got["cc"][comm], want.cc_ns[comm], rtol=CC_RTOL, atol=0)
    if refine > 0:
        assert np.array_equal(got["ov"], want.overlapped)


def test_tiny_gpt_bit_exact():
    c = W.config("tiny")
    g = W.build_gpt_graph(c)
    for S, refine in [(1, 1), (4, 0), (4, 1), (5, 2)]:
        sc = W.make_scenarios(g, c, n_scen=S) if S == 1 else W.make_scenarios(
            g, W.GPTConfig(**{**c.__dict__, "fixed_scenario": False}), n_scen=S)
        assert_same(run_gpu(g, sc, refine), oracle.compose(g, sc, refine_passes=refine), g, refine)


@pytest.mark.parametrize("S", [1, 3, 33, 130])
def test_random_graphs_bit_exact(S):
    rng = np.random.default_rng(77 + S)
    e = Echo(0)
    try:
        for case in range(60):
            g = SG.random_graph(rng, int(rng.integers(1, 60)), max_ranks=5, max_streams=5, p_edge=0.08)
            sc = SG.random_scenarios(rng, g, S, max_dur=50)
            for refine in (0, 1, 3):
                got = run_gpu(g, sc, refine, ctx=e)
                assert_same(got, oracle.compose(g, sc, refine_passes=refine), g, refine)
    finally:
        e.close()


@pytest.mark.parametrize("S", [33, 130])
def test_validator_many_comm_timelines_long_compute_timelines(S):
    """Ranks with up to 15 comm timelines and several hundred compute ops each:
    the overlap test's cursors cross chunk and warp-shuffle boundaries, and every
    register-cursor width (1..15 comm timelines) is exercised."""
    rng = np.random.default_rng(900 + S)
    e = Echo(0)
    try:
        for case in range(16):
            g = SG.random_graph(rng, int(rng.integers(300, 900)), max_ranks=3, max_streams=16,
                                min_streams=6 if case % 2 else 2, p_edge=0.004)
            sc = SG.random_scenarios(rng, g, S, max_dur=50)
            for refine in (1, 2):
                got = run_gpu(g, sc, refine, ctx=e)
                assert_same(got, oracle.compose(g, sc, refine_passes=refine), g, refine)
    finally:
        e.close()


def test_slowdown_rounding_is_exact():
    """The validator's rint(d * factor): every scenario slows one kernel that overlaps
    a collective from time 0, with edge-case durations (around 2^31, 2^52, 2^53,
    large) and factors (exact ties, 1 + 2^-52, 1/3, tiny, subnormal), and the slowed
    duration must equal numpy's fp64 product rounded to nearest even."""
    ops = [{"kind": W.KIND_COMPUTE, "kclass": 0}, {"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE, "cc_bytes": 1 << 20}]
    g = SG.graph_from_lists(2, 2, ops, {(0, 0): [0], (1, 0): [1], (0, 1): [2], (1, 1): [2]}, [[0, 1]])
    edge_d = [0, 1, 2, 3, 5, 7, 2**31 - 1, 2**31, 2**32 + 1, 2**52 - 1, 2**52, 2**52 + 1, 2**53 - 1, 2**53,
              2**53 + 1, 2**53 + 3, 2**54 + 2, 2**55 + 7, 2**56 + 12345, 2**57 - 1]
    edge_f = [1.0, 1.5, 2.5, 0.5, 0.25, 1.0000000000000002, 1.4, 1.2, 1 / 3, 0.9999999999999999, 3.0,
              1e-300, 5e-324, 2.2250738585072014e-308, 1.1, 1.3999999999999999, 1.25, 0.1]
    rng = np.random.default_rng(2024)
    pairs = [(d, f) for d in edge_d for f in edge_f]
    for _ in range(3000):
        d = int(rng.integers(0, 1 << int(rng.choice([3, 10, 20, 31, 40, 50, 53, 54, 56]))))
        f = float(rng.choice([rng.uniform(1.0, 1.4), rng.uniform(0.0, 3.0), rng.integers(1, 48) / 16]))
        pairs.append((d, f))
    S = len(pairs)
    d = np.array([p[0] for p in pairs], np.int64)
    f = np.array([p[1] for p in pairs], np.float64)
    sc = W.Scenarios(dur=np.stack([d, d, np.zeros(S, np.int64)]), alpha_ns=np.full(S, 100.0),
                     bw_intra=np.full(S, 50.0), lat_intra=np.full(S, 10.0), bw_inter=np.full(S, 5.0),
                     lat_inter=np.full(S, 20.0), delta=np.zeros(S), slowdown=f[None, :].copy(),
                     peak_flop_per_ns=np.ones(S))
    got = run_gpu(g, sc, 1)
    want = np.rint(d.astype(np.float64) * f).astype(np.int64)
    want[d == 0] = 0
    for v in (0, 1):
        assert np.array_equal(got["finish"][v] - got["start"][v], want)
    assert_same(got, oracle.compose(g, sc, refine_passes=1), g, 1)


def test_alpha_beta_cost_model_bit_exact():
    """The alpha-beta comparison model (size / bandwidth + latency) through
    echo_set_cc_model, against the oracle's; then back to Eqs. 2-5."""
    from paper_2412_12487_gb300.echo import CC_MODEL_ALPHA_BETA, CC_MODEL_WHITEBOX
    c = W.config("tiny")
    c = W.GPTConfig(**{**c.__dict__, "fixed_scenario": False})
    rng = np.random.default_rng(4242)
    cases = [(W.build_gpt_graph(c), None)]
    for _ in range(12):
        cases.append((SG.random_graph(rng, int(rng.integers(5, 60)), max_ranks=5, max_streams=4, p_edge=0.08),
                      None))
    e = Echo(0)
    try:
        for k, (g, _) in enumerate(cases):
            sc = W.make_scenarios(g, c, n_scen=6) if k == 0 else SG.random_scenarios(rng, g, 37, max_dur=50)
            e.set_cc_model(CC_MODEL_ALPHA_BETA)
            got = run_gpu(g, sc, 1, ctx=e)
            assert_same(got, oracle.compose(g, sc, refine_passes=1, cc_model=1), g, 1)
            e.set_cc_model(CC_MODEL_WHITEBOX)
            got = run_gpu(g, sc, 1, ctx=e)
            assert_same(got, oracle.compose(g, sc, refine_passes=1, cc_model=0), g, 1)
        with pytest.raises(EchoError):
            e.set_cc_model(7)
    finally:
        e.close()


@pytest.mark.parametrize("kernel", ["auto", "dataflow"])
def test_allreduce_policy_bit_exact(kernel, monkeypatch):
    """ring / tree / faster-of-the-two for every all-reduce (echo_compose_opts
    ar_algo_policy), against the oracle's policy: GPT-1.3B (per-op AUTO all-reduces)
    and random graphs mixing the per-op algorithms; switching the policy between
    compositions of one context re-estimates the collectives."""
    import dataclasses
    if kernel == "dataflow":
        monkeypatch.setenv("ECHO_COMPOSE_KERNEL", "dataflow")
    c = W.config("gpt1.3b")
    rng = np.random.default_rng(9900)
    cases = [(W.build_gpt_graph(c), None)]
    for _ in range(6):
        g = SG.random_graph(rng, int(rng.integers(10, 80)), max_ranks=5, max_streams=4, p_edge=0.06)
        cases.append((dataclasses.replace(g, cc_bytes=np.where(g.cc_bytes > 0, g.cc_bytes * 4096, 0)), None))
    e = Echo(0)
    try:
        for k, (g, _) in enumerate(cases):
            sc = W.make_scenarios(g, c, n_scen=40) if k == 0 else SG.random_scenarios(rng, g, 37, max_dur=2000)
            e.load_graph(g)
            e.load_scenarios(sc)
            e.estimate_collectives()
            for policy in (1, 2, 3, 0, 2):
                e.compose(refine_passes=1, ar_algo_policy=policy)
                st, fn = e.read_times()
                got = dict(start=st, finish=fn, makespan=e.read_makespan(), cc=e.read_cc(),
                           ov=e.read_overlap())
                want = oracle.compose(g, sc, refine_passes=1, ar_algo_policy=policy,
                                      threads=THREADS if k == 0 else 1)
                assert_same(got, want, g, 1)
        with pytest.raises(EchoError):
            e.compose(refine_passes=1, ar_algo_policy=4)
    finally:
        e.close()


@pytest.mark.parametrize("kernel", ["direct", "staged", "pipelined", "dataflow"])
def test_debug_bounds_checks_pass_and_change_nothing(kernel, monkeypatch):
    """debug_bounds: every composer and the validator check each index they gather
    through; on well-formed inputs no check fails and the timelines are the
    oracle's, for GPT-1.3B and random graphs with all validator variants."""
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", kernel)
    if kernel != "dataflow":
        monkeypatch.setenv("ECHO_SIGMA", "1" if kernel == "staged" else "4")
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    rng = np.random.default_rng(3300)
    e = Echo(0)
    try:
        sc = W.make_scenarios(g, c, n_scen=33)
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=2, debug_bounds=True)
        st, fn = e.read_times()
        got = dict(start=st, finish=fn, makespan=e.read_makespan(), cc=e.read_cc(), ov=e.read_overlap())
        assert_same(got, oracle.compose(g, sc, refine_passes=2, threads=THREADS), g, 2)
        for case in range(8):
            g = SG.random_graph(rng, int(rng.integers(20, 300)), max_ranks=5, max_streams=8, p_edge=0.03)
            sc = SG.random_scenarios(rng, g, 35, max_dur=60)
            model, civ = case % 2, (case // 2) % 2
            e.load_graph(g)
            e.load_scenarios(sc)
            e.estimate_collectives()
            e.compose(refine_passes=1 + case % 3, overlap_model=model, comm_interval=civ, debug_bounds=True)
            st, fn = e.read_times()
            got = dict(start=st, finish=fn, makespan=e.read_makespan(), cc=e.read_cc(), ov=e.read_overlap())
            want = oracle.compose(g, sc, refine_passes=1 + case % 3, overlap_model=model, comm_interval=civ)
            assert_same(got, want, g, 1 + case % 3)
    finally:
        e.close()


def test_read_times_scenario_range():
    """echo_read_times over a scenario range [s0, s1): the matching columns of the
    full readback, into host and device buffers; bad ranges are rejected."""
    import torch
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=70)
    with Echo(0) as e:
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=1)
        st, fn = e.read_times()
        for op0, op1, s0, s1 in ((0, g.n_ops, 0, 70), (17, 4000, 3, 41), (g.n_ops - 5, g.n_ops, 69, 70),
                                 (100, 100, 5, 9), (0, 1000, 64, 70)):
            a, b = e.read_times(op0, op1, s0=s0, s1=s1)
            assert np.array_equal(a, st[op0:op1, s0:s1]) and np.array_equal(b, fn[op0:op1, s0:s1])
        # device output buffers
        dst = torch.empty((300, 11), dtype=torch.int64, device="cuda")
        rc = e.lib.echo_read_times(e.h, 50, 350, 20, 31, None, dst.data_ptr())
        assert rc == 0
        assert np.array_equal(dst.cpu().numpy(), fn[50:350, 20:31])
        for bad in ((0, 10, -1, 5), (0, 10, 5, 71), (0, 10, 6, 5), (0, 10, 5, 5)):
            with pytest.raises(EchoError):
                e.read_times(bad[0], bad[1], s0=bad[2], s1=bad[3])


def test_int32_durations_give_the_same_timelines():
    """Durations passed as int32 (half the upload) compose exactly like int64 ones."""
    import dataclasses
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=40)
    assert sc.dur.max() < 2**31
    sc32 = dataclasses.replace(sc, dur=sc.dur.astype(np.int32))
    e = Echo(0)
    try:
        a = run_gpu(g, sc, 2, ctx=e)
        b = run_gpu(g, sc32, 2, ctx=e)
        for k in ("start", "finish", "makespan", "ov"):
            assert np.array_equal(a[k], b[k]), k
        np.testing.assert_array_equal(a["cc"], b["cc"])
        bad = sc32.dur.copy()
        bad[int(np.nonzero(g.kind == W.KIND_COMPUTE)[0][7]), 3] = -1
        with pytest.raises(EchoError) as ei:
            e.load_scenarios(dataclasses.replace(sc32, dur=bad))
        assert ei.value.code == 1
    finally:
        e.close()


def test_proportional_overlap_model_bit_exact():
    """Overlapped kernels lengthened by (factor - 1) x the covered length of their
    interval (union over the rank's comm intervals), against the oracle."""
    rng = np.random.default_rng(5150)
    e = Echo(0)
    try:
        for case in range(14):
            g = SG.random_graph(rng, int(rng.integers(20, 400)), max_ranks=4, max_streams=16,
                                min_streams=2 if case % 2 else 5, p_edge=0.01)
            sc = SG.random_scenarios(rng, g, 45, max_dur=60)
            for refine in (1, 2):
                got = run_gpu(g, sc, refine, ctx=e, overlap_model=1)
                assert_same(got, oracle.compose(g, sc, refine_passes=refine, overlap_model=1), g, refine)
        c = W.config("gpt1.3b")
        g = W.build_gpt_graph(c)
        sc = W.make_scenarios(g, c, n_scen=24)
        got = run_gpu(g, sc, 1, ctx=e, overlap_model=1)
        assert_same(got, oracle.compose(g, sc, refine_passes=1, overlap_model=1, threads=THREADS), g, 1)
        with pytest.raises(EchoError):
            e.compose(refine_passes=1, overlap_model=5)
    finally:
        e.close()


def test_launch_interval_bit_exact():
    """Comm intervals counted from each member rank's launch, with either overlap
    model, against the oracle: random multi-rank graphs (up to 16 timelines), the
    hand-built case, and GPT-1.3B."""
    from tests.test_oracle_pins import _launch_case
    rng = np.random.default_rng(6160)
    e = Echo(0)
    try:
        for d_b in (100, 300):
            g, sc = _launch_case(d_b)
            for model in (0, 1):
                got = run_gpu(g, sc, 1, ctx=e, overlap_model=model, comm_interval=1)
                assert_same(got, oracle.compose(g, sc, overlap_model=model, comm_interval=1), g, 1)
        for case in range(16):
            g = SG.random_graph(rng, int(rng.integers(20, 400)), max_ranks=4, max_streams=16,
                                min_streams=2 if case % 2 else 5, p_edge=0.01 if case % 4 < 2 else 0.05)
            sc = SG.random_scenarios(rng, g, 37, max_dur=60)
            for refine, model in ((1, 0), (2, 1), (2, 0)):
                got = run_gpu(g, sc, refine, ctx=e, overlap_model=model, comm_interval=1)
                want = oracle.compose(g, sc, refine_passes=refine, overlap_model=model, comm_interval=1)
                assert_same(got, want, g, refine)
        c = W.config("gpt1.3b")
        g = W.build_gpt_graph(c)
        sc = W.make_scenarios(g, c, n_scen=24)
        for model in (0, 1):
            got = run_gpu(g, sc, 1, ctx=e, overlap_model=model, comm_interval=1)
            want = oracle.compose(g, sc, refine_passes=1, overlap_model=model, comm_interval=1, threads=THREADS)
            assert_same(got, want, g, 1)
        base = oracle.compose(g, sc, refine_passes=1, threads=THREADS)
        assert (want.overlapped >= base.overlapped).all() and (want.overlapped > base.overlapped).any()
        with pytest.raises(EchoError):
            e.compose(refine_passes=1, comm_interval=2)
    finally:
        e.close()


def test_gpt13b_all_ops_all_scenarios_bit_exact():
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c)
    assert sc.n_scen == 256
    got = run_gpu(g, sc)
    want = oracle.compose(g, sc, threads=THREADS)
    assert_same(got, want, g)
    assert got["ov"].any() and (got["makespan"] > 0).all()


def test_degenerate_inputs():
    # empty graph
    g = SG.graph_from_lists(2, 3, [], {}, [])
    sc = W.Scenarios(dur=np.zeros((0, 3), np.int64), alpha_ns=np.zeros(3), bw_intra=np.ones(3),
                     lat_intra=np.zeros(3), bw_inter=np.ones(3), lat_inter=np.zeros(3),
                     delta=np.zeros(3), slowdown=np.ones((1, 3)), peak_flop_per_ns=np.ones(3))
    got = run_gpu(g, sc)
    assert (got["makespan"] == 0).all() and got["finish"].shape == (0, 3)
    # one op, zero duration; a chain of zero durations; compute-only single stream
    ops = [{"kind": W.KIND_COMPUTE} for _ in range(5)]
    g = SG.graph_from_lists(1, 1, ops, {(0, 0): list(range(5))}, [])
    sc = W.Scenarios(dur=np.zeros((5, 2), np.int64), alpha_ns=np.zeros(2), bw_intra=np.ones(2),
                     lat_intra=np.zeros(2), bw_inter=np.ones(2), lat_inter=np.zeros(2),
                     delta=np.zeros(2), slowdown=np.ones((1, 2)), peak_flop_per_ns=np.ones(2))
    got = run_gpu(g, sc)
    assert (got["finish"] == 0).all() and (got["makespan"] == 0).all()
    sc.dur[:, 1] = [3, 0, 5, 0, 7]
    got = run_gpu(g, sc)
    assert got["finish"][:, 1].tolist() == [3, 3, 8, 8, 15]


def test_high_fan_in_collective_and_global_frontier():
    # 1024 ranks join one all-reduce: 1024 timeline reads and 1024 data preds for
    # one node; 4096 ranks x 16 streams puts the frontier in global memory.
    for R, NS in [(1024, 2), (4096, 16)]:
        ops, queues = [], {}
        for r in range(R):
            ops.append({"kind": W.KIND_COMPUTE, "kclass": r % 3})
            queues[(r, 0)] = [r]
        ops.append({"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE,
                    "cc_algo": W.ALGO_AUTO, "cc_bytes": 1 << 26, "preds": list(range(R))})
        for r in range(R):
            queues[(r, 1 + r % (NS - 1))] = [R]
            ops.append({"kind": W.KIND_COMPUTE, "kclass": 0, "preds": [R]})
            queues[(r, 0)].append(R + 1 + r)
        g = SG.graph_from_lists(R, NS, ops, queues, [list(range(R))], gpus_per_node=8)
        rng = np.random.default_rng(R)
        sc = SG.random_scenarios(rng, g, 17, max_dur=10_000)
        sc.bw_intra[:] = 300.0
        sc.bw_inter[:] = 40.0
        got = run_gpu(g, sc)
        assert_same(got, oracle.compose(g, sc), g)


@pytest.mark.parametrize("kernel", ["pipelined", "auto"])
def test_many_scenarios_several_waves(kernel, monkeypatch):
    # 3001 scenarios: the levelled composer at its widest blocks (sigma 16, 188
    # blocks: more than one wave), and whichever composer the cost model picks
    if kernel != "auto":
        monkeypatch.setenv("ECHO_COMPOSE_KERNEL", kernel)
    c = W.config("tiny")
    g = W.build_gpt_graph(c)
    cr = W.GPTConfig(**{**c.__dict__, "fixed_scenario": False})
    sc = W.make_scenarios(g, cr, n_scen=3001)
    got = run_gpu(g, sc)
    want = oracle.compose(g, sc, threads=THREADS)
    assert_same(got, want, g)
    if kernel != "auto":
        assert got["info"]["sigma"] == 16


def test_cc_queries_match_oracle():
    q = W.make_cc_queries(1_000_000)
    with Echo(0) as e:
        got = e.cc_query(q)
    lib = oracle._load()
    import ctypes as C
    prm = np.stack([q.alpha_ns, q.bw_intra, q.lat_intra, q.bw_inter, q.lat_inter, q.delta], 1)
    prm = np.ascontiguousarray(prm)
    want = np.empty(q.n)
    K = -(-q.n_ranks // q.n_nodes)
    lg = np.log2(q.n_nodes.astype(np.float64))
    base = prm.ctypes.data
    for i in range(q.n):
        want[i] = lib.oracle_cc_ns(int(q.cc_type[i]), int(q.cc_algo[i]), int(q.nbytes[i]),
                                   int(q.n_ranks[i]), int(q.n_nodes[i]), int(K[i]), float(lg[i]),
                                   C.c_void_p(base + 48 * i), 0, None, None)
    np.testing.assert_allclose(got, want, rtol=CC_RTOL, atol=0)
    assert (got > 0).all()


def test_call_order_and_input_errors():
    c = W.config("tiny")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c)
    with Echo(0) as e:
        with pytest.raises(EchoError) as ei:
            e.estimate_collectives()
        assert ei.value.code == 4
        e.load_graph(g)
        with pytest.raises(EchoError) as ei:
            e.compose()
        assert ei.value.code == 4
        bad = W.Scenarios(**{**sc.__dict__, "dur": sc.dur.copy()})
        bad.dur[int(np.nonzero(g.kind == W.KIND_COMPUTE)[0][3]), 0] = -5
        with pytest.raises(EchoError) as ei:
            e.load_scenarios(bad)
        assert ei.value.code == 1
        bad = W.Scenarios(**{**sc.__dict__, "bw_inter": np.zeros(1)})
        with pytest.raises(EchoError) as ei:
            e.load_scenarios(bad)
        assert ei.value.code == 1
        huge = W.Scenarios(**{**sc.__dict__, "dur": sc.dur * 0 + (1 << 55)})
        e.load_scenarios(huge)
        with pytest.raises(EchoError) as ei:
            e.estimate_collectives()
        assert ei.value.code == 8
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose()
        with pytest.raises(EchoError) as ei:
            e.read_times(0, g.n_ops + 1)
        assert ei.value.code == 1
        a = e.read_makespan().copy()
        e.compose()
        assert np.array_equal(a, e.read_makespan())


def _full_batch_parity(name, time_cols, refine=1):
    """The whole batch of a full-size workload: every scenario's makespan against
    the oracle's (run threaded over the host cores), and every op's start and
    finish in the scenarios `time_cols`, read back one scenario column at a time
    through echo_read_times' scenario range."""
    c = W.config(name)
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c)
    with Echo(0) as e:
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=refine)
        mk = e.read_makespan()
        info = e.info()
        fin = np.empty((g.n_ops, len(time_cols)), np.int64)
        st = np.empty((g.n_ops, len(time_cols)), np.int64)
        for k, s in enumerate(time_cols):
            a, b = e.read_times(s0=s, s1=s + 1)
            st[:, k], fin[:, k] = a[:, 0], b[:, 0]
        assert (st >= 0).all() and (fin >= st).all()
        assert np.array_equal(mk[time_cols], fin.max(0))
    want_mk = oracle.compose(g, sc, refine_passes=refine, threads=THREADS, want_cc=False, want_overlap=False,
                             want_times=False).makespan
    assert np.array_equal(mk, want_mk), np.nonzero(mk != want_mk)[0][:10]
    del sc
    sub = W.select_scenarios(W.scenario_params(c), g, list(time_cols))
    want = oracle.compose(g, sub, refine_passes=refine, threads=THREADS, want_cc=False, want_overlap=False)
    assert np.array_equal(fin, want.finish)
    assert np.array_equal(st, want.start)
    return info


@pytest.mark.slow
def test_gpt175b_full_batch_bit_exact():
    # all 1024 makespans; every op in 128 scenarios, one in each scenario block of
    # the levelled composer (sigma 8) and every scenario position of a block
    # sixteen times over
    info = _full_batch_parity("gpt175b", [8 * b + b % 8 for b in range(128)])
    assert info["sigma"] == 8


@pytest.mark.slow
def test_gpt175b_1024_ranks_full_batch_bit_exact():
    # all 64 makespans (both groups of 32 scenarios of the dataflow composer); every
    # op in the first and last scenario of each group
    info = _full_batch_parity("gpt175b-1024", [0, 31, 32, 63])
    assert info["sigma"] == 32


@pytest.mark.parametrize("sigma", ["1", "2", "4", "8", "16"])
@pytest.mark.parametrize("kernel", ["direct", "staged", "pipelined"])
def test_every_compose_variant_bit_exact(sigma, kernel, monkeypatch):
    # the three compose kernels (global-memory, cp.async-staged, bulk-copy pipelined;
    # the pipelined one needs an even block width) at every scenario-block width,
    # with full and partial scenario blocks
    monkeypatch.setenv("ECHO_SIGMA", sigma)
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", kernel)
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    for S in (32, 37):
        sc = W.make_scenarios(g, c, n_scen=S)
        for refine in (0, 1, 2):
            got = run_gpu(g, sc, refine)
            assert_same(got, oracle.compose(g, sc, refine_passes=refine, threads=THREADS), g, refine)
    rng = np.random.default_rng(int(sigma) * 7 + len(kernel))
    e = Echo(0)
    try:
        for _ in range(15):
            g = SG.random_graph(rng, int(rng.integers(1, 80)), max_ranks=6, max_streams=4, p_edge=0.05)
            sc = SG.random_scenarios(rng, g, int(rng.choice([16, 32, 48, 64, 37])), max_dur=30)
            got = run_gpu(g, sc, 1, ctx=e)
            assert_same(got, oracle.compose(g, sc, refine_passes=1), g, 1)
    finally:
        e.close()


def test_dataflow_compose_bit_exact(monkeypatch):
    # the dataflow composer (a warp per rank and 32 scenarios, flag-synchronized
    # joins): GPT-1.3B with full and partial scenario groups and every validator
    # variant, and random graphs with data edges across ranks (export flags) and
    # groups of more than 8 members (two-hop joins)
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", "dataflow")
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    e = Echo(0)
    try:
        for S, refine, model, civ in ((32, 0, 0, 0), (37, 1, 0, 0), (64, 2, 1, 1), (5, 1, 0, 1)):
            sc = W.make_scenarios(g, c, n_scen=S)
            got = run_gpu(g, sc, refine, ctx=e, overlap_model=model, comm_interval=civ)
            assert got["info"]["sigma"] == 32
            want = oracle.compose(g, sc, refine_passes=refine, overlap_model=model, comm_interval=civ,
                                  threads=THREADS)
            assert_same(got, want, g, refine)
        rng = np.random.default_rng(404)
        for case in range(24):
            g = SG.random_graph(rng, int(rng.integers(1, 150)), max_ranks=14 if case % 2 else 5,
                                max_streams=5, p_edge=0.04)
            sc = SG.random_scenarios(rng, g, int(rng.choice([1, 31, 32, 33, 70])), max_dur=30)
            got = run_gpu(g, sc, 2, ctx=e)
            assert_same(got, oracle.compose(g, sc, refine_passes=2), g, 2)
    finally:
        e.close()


@pytest.mark.parametrize("streams", [(2, 4), (5, 7), (8, 16)])
def test_dataflow_validator_variants_bit_exact(streams, monkeypatch):
    """The dataflow composer with the validator between its compositions (cursor
    sets 3-, 4-, 6-, 8- and 16-wide): random multi-rank graphs with 1 to 15 comm
    timelines per rank and long compute timelines, both overlap models, both comm
    intervals and 1 to 3 validator passes, against the oracle."""
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", "dataflow")
    lo, hi = streams
    rng = np.random.default_rng(7100 + hi)
    e = Echo(0)
    try:
        for case in range(10):
            g = SG.random_graph(rng, int(rng.integers(100, 700)), max_ranks=4, max_streams=hi,
                                min_streams=lo, p_edge=0.004 if case % 2 else 0.02)
            sc = SG.random_scenarios(rng, g, int(rng.choice([7, 32, 45, 64])), max_dur=60)
            refine, model, civ = [(1, 0, 0), (2, 1, 0), (3, 0, 1), (1, 1, 1), (2, 0, 0)][case % 5]
            got = run_gpu(g, sc, refine, ctx=e, overlap_model=model, comm_interval=civ)
            assert got["info"]["sigma"] == 32
            want = oracle.compose(g, sc, refine_passes=refine, overlap_model=model, comm_interval=civ)
            assert_same(got, want, g, refine)
    finally:
        e.close()


def test_dataflow_bounded_wait_reports_timeout(monkeypatch):
    # failure detection without a GPU fault: one member never publishes its partial
    # launch time of a collective, the other members' bounded waits give up after
    # 20 ms, every warp leaves, and the host reports the timeout
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=64)
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", "dataflow")
    monkeypatch.setenv("ECHO_TEST_SKIP_LEVEL", "5")
    monkeypatch.setenv("ECHO_TEST_WAIT_LIMIT_MS", "20")
    with Echo(0) as e:
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=0)
        with pytest.raises(EchoError) as ei:
            e.read_makespan()
        assert ei.value.code == 7  # ECHO_E_TIMEOUT
    monkeypatch.delenv("ECHO_TEST_SKIP_LEVEL")
    monkeypatch.delenv("ECHO_TEST_WAIT_LIMIT_MS")
    got = run_gpu(g, sc, 1)
    assert_same(got, oracle.compose(g, sc, refine_passes=1, threads=THREADS), g, 1)


def test_bounded_wait_reports_timeout(monkeypatch):
    # failure detection without a GPU fault: the producer of the pipelined kernel
    # never fills one segment level, every consumer's bounded wait gives up after
    # 20 ms, the block records the timeout and exits, and the host reports it
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=64)
    monkeypatch.setenv("ECHO_SIGMA", "2")
    monkeypatch.setenv("ECHO_COMPOSE_KERNEL", "pipelined")
    monkeypatch.setenv("ECHO_TEST_SKIP_LEVEL", "5")
    monkeypatch.setenv("ECHO_TEST_WAIT_LIMIT_MS", "20")
    with Echo(0) as e:
        e.load_graph(g)
        e.load_scenarios(sc)
        e.estimate_collectives()
        e.compose(refine_passes=0)
        with pytest.raises(EchoError) as ei:
            e.read_makespan()
        assert ei.value.code == 7  # ECHO_E_TIMEOUT
    # the device is still usable: a context without the injected fault is exact
    monkeypatch.delenv("ECHO_TEST_SKIP_LEVEL")
    monkeypatch.delenv("ECHO_TEST_WAIT_LIMIT_MS")
    got = run_gpu(g, sc, 1)
    assert_same(got, oracle.compose(g, sc, refine_passes=1, threads=THREADS), g, 1)
