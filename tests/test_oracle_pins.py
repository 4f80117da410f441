"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each pin is chosen so that a plausible slip in the oracle (a dropped term, a wrong
index or sign, a swapped link, an off-by-one in the chunk count, a wrong tie-break,
a wrong overlap rule) fails at least one of them:

* Table 6 chunk sizes (golden fixture) and its reduce-time row.
* Textbook ring collective costs (Thakur/Rabenseifner/Gropp 2005; Patarasuk/Yuan
  2009) at one chunk; the bandwidth term's independence of the chunk count; the
  number of rounds eta = ceil(S / (N*C)) read off the latency term; the binary tree
  and the intra-node chain of Eq. 5; a single transfer for send/recv.
* Brute-force longest paths on every small random DAG, with the validator's overlap
  checked pair by pair; invariants (tie-break order, monotonicity, shift,
  scenario permutation); hand-built join and overlap examples with known answers.
"""
import math
import os

import numpy as np
import pytest

import oracle
from paper_2412_12487_gb300 import workloads as W
from tests import smallgraphs as SG

HERE = os.path.dirname(os.path.abspath(__file__))
MiB = 1 << 20


def _table6():
    rows = []
    with open(os.path.join(HERE, "golden", "table6_chunk_sizes.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                mb, kb, us = line.split()
                rows.append((int(mb), int(kb), float(us)))
    return rows


# ------------------------------------------------------------------------------------
# CC estimator (Sec. 5.3, Eqs. 2-5; Table 6)
# ------------------------------------------------------------------------------------
def test_chunk_size_matches_table6():
    for mb, kb, _ in _table6():
        assert oracle.chunk_bytes(mb * MiB) == kb * 1000, mb


def test_chunk_size_between_and_beyond_table():
    assert oracle.chunk_bytes(1) == 18000
    assert oracle.chunk_bytes(4 * MiB + 1) == 36000
    assert oracle.chunk_bytes(8 * MiB + 1) == 72000
    assert oracle.chunk_bytes(64 * MiB + 1) == 144000
    assert oracle.chunk_bytes(128 * MiB + 1) == 288000
    assert oracle.chunk_bytes(8 << 30) == 288000
    tbl = (np.array([100, 1000]), np.array([7, 11]))
    assert oracle.chunk_bytes(50, tbl) == 7 and oracle.chunk_bytes(101, tbl) == 11
    assert oracle.chunk_bytes(5000, tbl) == 11


def test_reduce_row_of_table6_matches_default_delta():
    # the default reduce throughput is taken from the 256 MB column of Table 6
    for mb, _, us in _table6():
        if mb == 256:
            assert W.DELTA_NS_PER_B * (mb * MiB) == pytest.approx(us * 1e3, rel=1e-12)


def _prm(rng):
    return dict(alpha=float(rng.uniform(0, 5e4)), bw_intra=float(rng.uniform(25, 900)),
                lat_intra=float(rng.uniform(0, 5e3)), bw_inter=float(rng.uniform(3, 120)),
                lat_inter=float(rng.uniform(0, 1e4)), delta=float(rng.uniform(0, 1e-2)))


def _cc(t, a, S, N, M, K, p):
    return oracle.cc_ns(t, a, S, N, M, K, math.log2(M), p["alpha"], p["bw_intra"], p["lat_intra"],
                        p["bw_inter"], p["lat_inter"], p["delta"])


@pytest.mark.parametrize("N", [2, 3, 4, 8, 16, 96])
def test_ring_allreduce_one_chunk_is_textbook(N):
    # Ring all-reduce = reduce-scatter + all-gather, 2(N-1) steps of S/N bytes:
    # alpha + 2(N-1) L + 2 (N-1)/N * S/B (+ the reduction), one node.
    rng = np.random.default_rng(N)
    for _ in range(50):
        p = _prm(rng)
        S = int(rng.integers(1, N * 18000 + 1))  # at most one chunk per rank
        want = p["alpha"] + 2 * (N - 1) * p["lat_intra"] + 2 * (N - 1) / N * S / p["bw_intra"] \
            + p["delta"] * S
        got = _cc(W.CC_ALLREDUCE, W.ALGO_RING, S, N, 1, N, p)
        assert got == pytest.approx(want, rel=1e-12)


@pytest.mark.parametrize("N", [2, 5, 8])
def test_ring_reducescatter_and_allgather_one_chunk_are_textbook(N):
    rng = np.random.default_rng(100 + N)
    for _ in range(50):
        p = _prm(rng)
        S = int(rng.integers(1, N * 18000 + 1))
        rs = p["alpha"] + (N - 1) * (p["lat_intra"] + S / N / p["bw_intra"]) + p["delta"] * S
        ag = p["alpha"] + (N - 1) * (p["lat_intra"] + S / N / p["bw_intra"])
        assert _cc(W.CC_REDUCESCATTER, 0, S, N, 1, N, p) == pytest.approx(rs, rel=1e-12)
        assert _cc(W.CC_ALLGATHER, 0, S, N, 1, N, p) == pytest.approx(ag, rel=1e-12)


def test_allgather_of_two_ranks_is_one_half_transfer():
    rng = np.random.default_rng(7)
    for _ in range(50):
        p = _prm(rng)
        S = int(rng.integers(1, 2 * 18000 + 1))
        one = p["alpha"] + p["lat_intra"] + (S / 2) / p["bw_intra"]
        assert _cc(W.CC_ALLGATHER, 0, S, 2, 1, 2, p) == pytest.approx(one, rel=1e-12)
        # across two nodes the step uses the inter-node link
        two = p["alpha"] + p["lat_inter"] + (S / 2) / p["bw_inter"]
        assert _cc(W.CC_ALLGATHER, 0, S, 2, 2, 1, p) == pytest.approx(two, rel=1e-12)


def test_ring_bandwidth_term_is_independent_of_chunking():
    # with zero latency, chunking into eta rounds moves the same bytes per link:
    # 2 (N-1)/N * S/B, the bandwidth-optimal all-reduce bound
    rng = np.random.default_rng(11)
    for _ in range(200):
        p = _prm(rng)
        p["lat_intra"] = p["lat_inter"] = 0.0
        N = int(rng.choice([2, 4, 8, 12]))
        S = int(rng.integers(1, 3 << 30))
        want = p["alpha"] + 2 * (N - 1) / N * S / p["bw_intra"] + p["delta"] * S
        assert _cc(W.CC_ALLREDUCE, W.ALGO_RING, S, N, 1, N, p) == pytest.approx(want, rel=1e-11)


def test_ring_rounds_from_latency_term():
    # with infinite bandwidth only the 2*eta*(N-1) step latencies remain, and eta is
    # the number of chunk rounds NCCL needs: ceil(S / (N * chunk)) with Table 6's chunk
    p = dict(alpha=0.0, bw_intra=1e300, lat_intra=1.0, bw_inter=1e300, lat_inter=1.0, delta=0.0)
    for S, N, eta in [(256 * MiB, 8, 117), (4 * MiB, 8, 30), (4 * MiB, 256, 1),
                      (128 * MiB, 32, 30), (64 * MiB, 2, 467), (1, 4, 1)]:
        assert _cc(W.CC_ALLREDUCE, W.ALGO_RING, S, N, 1, N, p) == 2 * eta * (N - 1)
        assert _cc(W.CC_ALLGATHER, 0, S, N, 1, N, p) == eta * (N - 1)


def test_tree_allreduce_special_cases():
    rng = np.random.default_rng(3)
    for _ in range(100):
        p = _prm(rng)
        S = int(rng.integers(1, 18000 + 1))   # one chunk
        # one node: a chain of K ranks, reduce up and broadcast down, 2(K-1) hops
        K = int(rng.integers(2, 9))
        chain = p["alpha"] + 2 * (K - 1) * (p["lat_intra"] + S / p["bw_intra"]) + p["delta"] * S
        assert _cc(W.CC_ALLREDUCE, W.ALGO_TREE, S, K, 1, K, p) == pytest.approx(chain, rel=1e-12)
        # one GPU per node: a binary tree over M nodes, 2 log2(M) inter-node hops
        M = int(rng.choice([2, 4, 8, 16, 32]))
        bt = p["alpha"] + 2 * math.log2(M) * (p["lat_inter"] + S / p["bw_inter"]) + p["delta"] * S
        assert _cc(W.CC_ALLREDUCE, W.ALGO_TREE, S, M, M, 1, p) == pytest.approx(bt, rel=1e-12)


def test_tree_pipelining_adds_one_inter_hop_per_extra_chunk():
    # eta chunks pipelined through the tree: each chunk after the first adds gamma
    p = dict(alpha=0.0, bw_intra=1e300, lat_intra=0.0, bw_inter=1e300, lat_inter=3.0, delta=0.0)
    for S in [18000, 18001, 5 * MiB, 100 * MiB, 300 * MiB]:
        eta = -(-S // oracle.chunk_bytes(S))
        got = _cc(W.CC_ALLREDUCE, W.ALGO_TREE, S, 16, 2, 8, p)
        assert got == pytest.approx(3.0 * (eta - 1) + 2 * 3.0 * 1.0, rel=1e-12)


def test_sendrecv_is_one_transfer():
    rng = np.random.default_rng(5)
    for _ in range(100):
        p = _prm(rng)
        S = int(rng.integers(1, 1 << 31))
        p0 = dict(p, lat_intra=0.0, lat_inter=0.0)
        assert _cc(W.CC_SENDRECV, 0, S, 2, 1, 2, p0) == pytest.approx(
            p["alpha"] + S / p["bw_intra"], rel=1e-12)
        assert _cc(W.CC_SENDRECV, 0, S, 2, 2, 1, p0) == pytest.approx(
            p["alpha"] + S / p["bw_inter"], rel=1e-12)
        # each chunk pays the link latency once
        eta = -(-S // oracle.chunk_bytes(S))
        assert _cc(W.CC_SENDRECV, 0, S, 2, 1, 2, p) == pytest.approx(
            p["alpha"] + eta * p["lat_intra"] + S / p["bw_intra"], rel=1e-12)


def test_reduction_term_and_degenerate_cases():
    rng = np.random.default_rng(9)
    for _ in range(100):
        p = _prm(rng)
        S = int(rng.integers(1, 1 << 30))
        N = int(rng.choice([2, 8, 24]))
        M = max(1, N // 8)
        K = N // M
        p0 = dict(p, delta=0.0)
        for t, a in [(W.CC_ALLREDUCE, W.ALGO_RING), (W.CC_ALLREDUCE, W.ALGO_TREE),
                     (W.CC_REDUCESCATTER, 0)]:
            assert _cc(t, a, S, N, M, K, p) - _cc(t, a, S, N, M, K, p0) == pytest.approx(
                p["delta"] * S, rel=1e-9, abs=1e-6)
        # all-gather and send/recv reduce nothing
        assert _cc(W.CC_ALLGATHER, 0, S, N, M, K, p) == _cc(W.CC_ALLGATHER, 0, S, N, M, K, p0)
        for t in range(4):
            assert _cc(t, 2, 0, N, M, K, p) == 0.0
            assert _cc(t, 2, S, 1, 1, 1, p) == 0.0


def test_alpha_beta_model_is_size_over_bandwidth_plus_latency():
    """The comparison model of Sec. 2.3: message size / bandwidth + latency, on the
    intra-node link inside a node and the inter-node one across nodes; setup
    (alpha) and reduction (delta) costs play no part, nor does the chunk table."""
    # 1 MiB at 50 B/ns with a 5 us latency: 5000 + 20971.52 ns
    assert oracle.cc_ns_alpha_beta(1 << 20, 8, 1, 10000.0, 50.0, 5000.0, 6.25, 9000.0, 1e-3) == 25971.52
    # across nodes: 1 MiB at 6.25 B/ns with 9 us: 9000 + 167772.16 ns
    assert oracle.cc_ns_alpha_beta(1 << 20, 16, 2, 10000.0, 50.0, 5000.0, 6.25, 9000.0, 1e-3) == 176772.16
    assert oracle.cc_ns_alpha_beta(1 << 20, 1, 1, 10000.0, 50.0, 5000.0, 6.25, 9000.0, 1e-3) == 0.0
    assert oracle.cc_ns_alpha_beta(0, 8, 2, 10000.0, 50.0, 5000.0, 6.25, 9000.0, 1e-3) == 0.0


def test_alpha_beta_composition_times_every_collective_by_the_model():
    g = W.build_gpt_graph(W.config("tiny"))
    sc = W.make_scenarios(g, W.config("tiny"), n_scen=1)
    r = oracle.compose(g, sc, refine_passes=0, cc_model=1)
    comm = np.nonzero((g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P))[0]
    assert len(comm) > 10
    for v in comm:
        members = g.grp_rank[g.grp_off[g.group[v]]:g.grp_off[g.group[v] + 1]]
        nodes = len(set(int(m) // g.gpus_per_node for m in members))
        B, L = (sc.bw_inter[0], sc.lat_inter[0]) if nodes > 1 else (sc.bw_intra[0], sc.lat_intra[0])
        want = 0 if len(members) <= 1 or g.cc_bytes[v] == 0 else int(np.rint(L + g.cc_bytes[v] / B))
        assert r.finish[v, 0] - r.start[v, 0] == want
    # the white-box times differ from these
    w = oracle.compose(g, sc, refine_passes=0, cc_model=0)
    assert not np.array_equal(w.finish[comm] - w.start[comm], r.finish[comm] - r.start[comm])


def _overlap_case(two_streams):
    """Rank 0 runs kernel c (100 ns) from 0; on its comm timeline(s) a memcpy (50 or
    70 ns) precedes a send/recv with rank 1 of 1000 B at 10 B/ns (100 ns, no setup
    or latency), so the send/recv runs [50, 150) (and the second one [70, 170))."""
    ops = [{"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_MEMCPY},
           {"kind": W.KIND_P2P, "group": 0, "cc_type": W.CC_SENDRECV, "cc_bytes": 1000}]
    queues = {(0, 0): [0], (0, 1): [1, 2], (1, 1): [2]}
    groups = [[0, 1]]
    if two_streams:
        ops += [{"kind": W.KIND_MEMCPY},
                {"kind": W.KIND_P2P, "group": 1, "cc_type": W.CC_SENDRECV, "cc_bytes": 1000}]
        queues.update({(0, 2): [3, 4], (1, 2): [4]})
        groups.append([0, 1])
    g = SG.graph_from_lists(2, 3 if two_streams else 2, ops, queues, groups, gpus_per_node=2)
    dur = np.zeros((len(ops), 1), np.int64)
    dur[0, 0], dur[1, 0] = 100, 50
    if two_streams:
        dur[3, 0] = 70
    sc = W.Scenarios(dur=dur, alpha_ns=np.zeros(1), bw_intra=np.full(1, 10.0), lat_intra=np.zeros(1),
                     bw_inter=np.full(1, 10.0), lat_inter=np.zeros(1), delta=np.zeros(1),
                     slowdown=np.full((1, 1), 1.5), peak_flop_per_ns=np.ones(1))
    return g, sc


def test_whole_kernel_and_proportional_slowdown_by_hand():
    g, sc = _overlap_case(False)
    r = oracle.compose(g, sc, refine_passes=1, overlap_model=0)
    assert (r.start[2, 0], r.finish[2, 0]) == (50, 150)
    assert r.overlapped[0, 0] == 1 and r.finish[0, 0] - r.start[0, 0] == 150  # 100 * 1.5
    r = oracle.compose(g, sc, refine_passes=1, overlap_model=1)
    assert r.finish[0, 0] - r.start[0, 0] == 125  # 100 + 0.5 * 50 (overlap [50, 100))


def test_proportional_slowdown_counts_overlapping_comm_once():
    g, sc = _overlap_case(True)
    r = oracle.compose(g, sc, refine_passes=1, overlap_model=1)
    assert (r.start[4, 0], r.finish[4, 0]) == (70, 170)
    # [50, 100) and [70, 100) cover [50, 100): 50 ns, not 80
    assert r.finish[0, 0] - r.start[0, 0] == 125
    r = oracle.compose(g, sc, refine_passes=1, overlap_model=0)
    assert r.finish[0, 0] - r.start[0, 0] == 150


def test_proportional_model_never_exceeds_whole_kernel_model():
    rng = np.random.default_rng(31)
    for _ in range(200):
        g = SG.random_graph(rng, int(rng.integers(2, 30)), max_ranks=3, max_streams=4, p_edge=0.1)
        sc = SG.random_scenarios(rng, g, 3, max_dur=40)
        a = oracle.compose(g, sc, refine_passes=1, overlap_model=0)
        b = oracle.compose(g, sc, refine_passes=1, overlap_model=1)
        assert np.array_equal(a.overlapped, b.overlapped)  # same decisions from the same first pass
        comp = g.kind == W.KIND_COMPUTE
        # slowdown factors are >= 1: the overlapped part is at most the whole kernel
        assert ((b.finish - b.start)[comp] <= (a.finish - a.start)[comp]).all()


def _launch_case(d_b):
    """Rank 0 runs kernels a (10 ns) then b; rank 1 runs kernel c (200 ns).  An
    all-reduce of ranks 0 and 1 needs a's and c's outputs: 500 B at 10 B/ns, no
    setup, latency or reduction cost, so it runs [200, 250).  Rank 0 has launched
    it at 10, rank 1 at 200."""
    ops = [{"kind": W.KIND_COMPUTE, "kclass": 0}, {"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE, "cc_algo": W.ALGO_RING,
            "cc_bytes": 500, "preds": [0, 2]}]
    queues = {(0, 0): [0, 1], (1, 0): [2], (0, 1): [3], (1, 1): [3]}
    g = SG.graph_from_lists(2, 2, ops, queues, [[0, 1]], gpus_per_node=2)
    dur = np.array([[10], [d_b], [200], [0]], np.int64)
    sc = W.Scenarios(dur=dur, alpha_ns=np.zeros(1), bw_intra=np.full(1, 10.0), lat_intra=np.zeros(1),
                     bw_inter=np.full(1, 10.0), lat_inter=np.zeros(1), delta=np.zeros(1),
                     slowdown=np.full((1, 1), 1.5), peak_flop_per_ns=np.ones(1))
    return g, sc


def test_launch_interval_by_hand():
    g, sc = _launch_case(100)
    r = oracle.compose(g, sc, refine_passes=1, comm_interval=0)
    assert (r.start[3, 0], r.finish[3, 0]) == (200, 250)
    assert r.overlapped[:, 0].tolist() == [0, 0, 0, 0]  # b runs [10, 110)
    for model in (0, 1):
        r = oracle.compose(g, sc, refine_passes=1, overlap_model=model, comm_interval=1)
        # on rank 0 the all-reduce holds [10, 250): b overlaps it over its whole length;
        # on rank 1 it holds [200, 250), which only touches c
        assert r.overlapped[:, 0].tolist() == [0, 1, 0, 0]
        assert r.finish[1, 0] - r.start[1, 0] == 150  # 100 * 1.5 = 100 + 0.5 * 100
    g, sc = _launch_case(300)  # b runs [10, 310)
    assert oracle.compose(g, sc, overlap_model=1, comm_interval=0).finish[1, 0] == 10 + 325  # 300 + 0.5 * 50
    assert oracle.compose(g, sc, overlap_model=1, comm_interval=1).finish[1, 0] == 10 + 420  # 300 + 0.5 * 240
    assert oracle.compose(g, sc, overlap_model=0, comm_interval=1).finish[1, 0] == 10 + 450


def test_launch_interval_on_one_rank_is_the_execution_interval():
    # with one rank every launch condition of a comm op is that rank's, so it
    # launches exactly when it starts
    rng = np.random.default_rng(37)
    for _ in range(200):
        g = SG.random_graph(rng, int(rng.integers(2, 30)), max_ranks=1, max_streams=4, p_edge=0.1)
        sc = SG.random_scenarios(rng, g, 3, max_dur=40)
        for model in (0, 1):
            a = oracle.compose(g, sc, refine_passes=2, overlap_model=model, comm_interval=0)
            b = oracle.compose(g, sc, refine_passes=2, overlap_model=model, comm_interval=1)
            assert np.array_equal(a.finish, b.finish) and np.array_equal(a.overlapped, b.overlapped)


def test_launch_interval_only_adds_overlaps():
    # the same first composition, and every launch interval holds the execution one
    rng = np.random.default_rng(41)
    grew = 0
    for _ in range(300):
        g = SG.random_graph(rng, int(rng.integers(2, 30)), max_ranks=3, max_streams=4, p_edge=0.1)
        sc = SG.random_scenarios(rng, g, 3, max_dur=40)
        a = oracle.compose(g, sc, refine_passes=1, comm_interval=0)
        b = oracle.compose(g, sc, refine_passes=1, comm_interval=1)
        assert (b.overlapped >= a.overlapped).all()
        grew += int((b.overlapped > a.overlapped).any())
    assert grew > 10  # the variant does change decisions on multi-rank graphs


@pytest.mark.parametrize("seed", range(4))
def test_brute_force_launch_intervals(seed):
    rng = np.random.default_rng(2000 + seed)
    for case in range(400):
        g = SG.random_graph(rng, int(rng.integers(1, 11)))
        sc = SG.random_scenarios(rng, g, 2)
        for passes in (1, 2):
            r = oracle.compose(g, sc, refine_passes=passes, comm_interval=1)
            for s in range(sc.n_scen):
                st, fn, ov = SG.brute_compose(g, sc, s, passes, oracle.cc_ns, comm_interval=1)
                assert (r.finish[:, s] == fn).all(), (seed, case, passes)
                assert (r.overlapped[:, s] == ov).all(), (seed, case, passes)


@pytest.mark.parametrize("seed", range(3))
def test_brute_force_proportional_slowdown(seed):
    # the proportional model against a pair-by-pair brute force whose covered
    # length comes from coordinate compression, with either comm interval
    # sparse graphs with several comm timelines, so that kernels often run under
    # two concurrent comm ops (where the union differs from the sum)
    rng = np.random.default_rng(3000 + seed)
    for case in range(150):
        g = SG.random_graph(rng, int(rng.integers(4, 26)), max_ranks=2, max_streams=5, p_edge=0.04,
                            min_streams=3)
        sc = SG.random_scenarios(rng, g, 2)
        for passes, civ in ((1, 0), (2, 1), (1, 1)):
            r = oracle.compose(g, sc, refine_passes=passes, overlap_model=1, comm_interval=civ)
            for s in range(sc.n_scen):
                st, fn, ov = SG.brute_compose(g, sc, s, passes, oracle.cc_ns, comm_interval=civ, overlap_model=1)
                assert (r.finish[:, s] == fn).all(), (seed, case, passes, civ)
                assert (r.overlapped[:, s] == ov).all(), (seed, case, passes, civ)


def test_covered_length_helper():
    # the brute force's own union length, by hand
    assert SG.covered_length([]) == 0
    assert SG.covered_length([(0, 10), (5, 15)]) == 15
    assert SG.covered_length([(0, 2), (4, 6), (1, 5)]) == 6
    assert SG.covered_length([(3, 4), (3, 4)]) == 1


def test_auto_takes_the_faster_algorithm():
    rng = np.random.default_rng(13)
    for _ in range(300):
        p = _prm(rng)
        S = int(rng.integers(1, 1 << 31))
        N = int(rng.choice([2, 8, 16, 64, 96, 1024]))
        M = max(1, -(-N // 8))
        K = -(-N // M)
        r = _cc(W.CC_ALLREDUCE, W.ALGO_RING, S, N, M, K, p)
        t = _cc(W.CC_ALLREDUCE, W.ALGO_TREE, S, N, M, K, p)
        assert _cc(W.CC_ALLREDUCE, W.ALGO_AUTO, S, N, M, K, p) == min(r, t)


@pytest.mark.parametrize("seed", range(4))
def test_allreduce_policy_equals_rewriting_every_allreduce(seed):
    """Sec. 5.1: NCCL runs an all-reduce as a ring or a tree.  A policy that forces
    ring, tree or the faster of the two must give exactly the composition of the
    same graph with every all-reduce's own algorithm rewritten to it, must leave
    every other collective's estimate alone, and AUTO must be the per-op minimum
    of the forced ring and tree estimates.  The graphs mix the three per-op
    algorithms, and the large messages make ring and tree differ."""
    import dataclasses
    rng = np.random.default_rng(8800 + seed)
    differs = False
    for _ in range(12):
        g = SG.random_graph(rng, int(rng.integers(10, 60)), max_ranks=5, max_streams=4, p_edge=0.08)
        g = dataclasses.replace(g, cc_bytes=np.where(g.cc_bytes > 0, g.cc_bytes * 4096, 0))
        sc = SG.random_scenarios(rng, g, 5, max_dur=2000)
        ar = (g.cc_type == W.CC_ALLREDUCE) & ((g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P))
        comm = (g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P)
        base = oracle.compose(g, sc, refine_passes=1)
        got = {}
        for policy, algo in ((1, W.ALGO_RING), (2, W.ALGO_TREE), (3, W.ALGO_AUTO)):
            forced = oracle.compose(g, sc, refine_passes=1, ar_algo_policy=policy)
            g2 = dataclasses.replace(g, cc_algo=np.where(ar, algo, g.cc_algo).astype(np.uint8))
            rewritten = oracle.compose(g2, sc, refine_passes=1)
            assert np.array_equal(forced.finish, rewritten.finish)
            assert np.array_equal(forced.start, rewritten.start)
            np.testing.assert_array_equal(forced.cc_ns[comm], rewritten.cc_ns[comm])
            np.testing.assert_array_equal(forced.cc_ns[comm & ~ar], base.cc_ns[comm & ~ar])
            got[policy] = forced
        np.testing.assert_array_equal(got[3].cc_ns[ar], np.minimum(got[1].cc_ns[ar], got[2].cc_ns[ar]))
        differs |= bool((got[1].cc_ns[ar] != got[2].cc_ns[ar]).any())
    assert differs
    with pytest.raises(RuntimeError):
        oracle.compose(g, sc, ar_algo_policy=4)


def test_monotone_in_size_and_inverse_bandwidth():
    rng = np.random.default_rng(17)
    for _ in range(300):
        p = _prm(rng)
        t = int(rng.integers(0, 4))
        a = int(rng.integers(0, 3))
        N = 2 if t == W.CC_SENDRECV else int(rng.choice([2, 8, 16, 48]))
        M = max(1, -(-N // 8))
        K = -(-N // M)
        S = int(rng.integers(1, 1 << 30))
        base = _cc(t, a, S, N, M, K, p)
        assert _cc(t, a, 2 * S, N, M, K, p) >= base
        slow = dict(p, bw_intra=p["bw_intra"] / 2, bw_inter=p["bw_inter"] / 2)
        assert _cc(t, a, S, N, M, K, slow) >= base


# ------------------------------------------------------------------------------------
# composer (Sec. 4.2, 5.2) and validator (Sec. 2.3 / 3)
# ------------------------------------------------------------------------------------
def _scen_fixed(S=1, n_kclass=1, sf=1.0, dur=None, alpha=0.0):
    return W.Scenarios(
        dur=dur if dur is not None else np.zeros((0, S), np.int64),
        alpha_ns=np.full(S, alpha), bw_intra=np.full(S, 1e300), lat_intra=np.zeros(S),
        bw_inter=np.full(S, 1e300), lat_inter=np.zeros(S), delta=np.zeros(S),
        slowdown=np.full((n_kclass, S), sf), peak_flop_per_ns=np.ones(S))


def test_pure_chain_is_sum_of_durations():
    rng = np.random.default_rng(0)
    for n in [1, 2, 7, 50]:
        ops = [{"kind": W.KIND_COMPUTE} for _ in range(n)]
        g = SG.graph_from_lists(1, 2, ops, {(0, 0): list(range(n))}, [])
        d = rng.integers(0, 1000, size=(n, 3)).astype(np.int64)
        r = oracle.compose(g, _scen_fixed(3, dur=d))
        assert (r.makespan == d.sum(0)).all()
        assert (r.start == np.cumsum(d, 0) - d).all()


def test_without_comm_each_rank_is_its_own_critical_path():
    rng = np.random.default_rng(1)
    for _ in range(20):
        R = int(rng.integers(1, 5))
        ops, queues = [], {}
        for r in range(R):
            for k in range(int(rng.integers(1, 12))):
                v = len(ops)
                ops.append({"kind": W.KIND_COMPUTE})
                queues.setdefault((r, 0), []).append(v)
            for k in range(int(rng.integers(0, 4))):
                v = len(ops)
                ops.append({"kind": W.KIND_MEMCPY})
                queues.setdefault((r, 1), []).append(v)
        g = SG.graph_from_lists(R, 2, ops, queues, [])
        d = rng.integers(0, 500, size=(len(ops), 2)).astype(np.int64)
        r = oracle.compose(g, _scen_fixed(2, dur=d))
        want = np.zeros(2, np.int64)
        for q in queues.values():
            want = np.maximum(want, d[q].sum(0))  # independent streams: per-stream sums
        assert (r.makespan == want).all()


@pytest.mark.parametrize("seed", range(10))
def test_brute_force_small_dags(seed):
    # every small DAG: finish = longest path sum; with the validator, the overlap
    # bits and the second composition also match a pair-by-pair brute force
    rng = np.random.default_rng(1000 + seed)
    for case in range(1000):
        n = int(rng.integers(1, 11))
        g = SG.random_graph(rng, n)
        sc = SG.random_scenarios(rng, g, 2)
        for passes in (0, 1, 2):
            r = oracle.compose(g, sc, refine_passes=passes)
            for s in range(sc.n_scen):
                st, fn, ov = SG.brute_compose(g, sc, s, passes, oracle.cc_ns)
                assert (r.finish[:, s] == fn).all(), (seed, case, passes)
                assert (r.start[:, s] == st).all(), (seed, case, passes)
                assert (r.overlapped[:, s] == ov).all(), (seed, case, passes)
                assert r.makespan[s] == (fn.max() if n else 0)


def test_start_is_latest_predecessor_finish():
    rng = np.random.default_rng(21)
    for _ in range(300):
        g = SG.random_graph(rng, int(rng.integers(2, 30)), max_ranks=4, max_streams=4)
        sc = SG.random_scenarios(rng, g, 3)
        r = oracle.compose(g, sc, refine_passes=1)
        preds = SG.merged_preds(g)
        for v in range(g.n_ops):
            want = np.zeros(3, np.int64)
            for u in preds[v]:
                want = np.maximum(want, r.finish[u])
            assert (r.start[v] == want).all()


def test_tie_break_order_does_not_change_times():
    rng = np.random.default_rng(22)
    for _ in range(200):
        g = SG.random_graph(rng, int(rng.integers(2, 40)), max_ranks=4, max_streams=4)
        sc = SG.random_scenarios(rng, g, 2, max_dur=3)   # many equal times
        a = oracle.compose(g, sc, refine_passes=1)
        for seed in (1, 2, 3):
            b = oracle.compose(g, sc, refine_passes=1, tie_seed=seed)
            assert (a.start == b.start).all() and (a.finish == b.finish).all()
    c = W.config("tiny")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c)
    a = oracle.compose(g, sc)
    b = oracle.compose(g, sc, tie_seed=12345)
    assert (a.finish == b.finish).all()


def test_monotone_in_durations_without_validator():
    rng = np.random.default_rng(23)
    for _ in range(200):
        g = SG.random_graph(rng, int(rng.integers(2, 30)), max_ranks=3)
        sc = SG.random_scenarios(rng, g, 1)
        a = oracle.compose(g, sc, refine_passes=0)
        v = int(rng.integers(0, g.n_ops))
        sc.dur[v, 0] += int(rng.integers(1, 100))
        b = oracle.compose(g, sc, refine_passes=0)
        assert (b.finish >= a.finish).all()


def test_adding_to_every_source_shifts_every_finish():
    rng = np.random.default_rng(24)
    for _ in range(200):
        g = SG.random_graph(rng, int(rng.integers(1, 30)), max_ranks=3)
        g.kind[(g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P)] = W.KIND_MEMCPY
        # the comm ops, now memcpy, sit in several timelines; keep only the first
        keep = np.zeros(g.q_ops.shape[0], bool)
        seen = set()
        for i, v in enumerate(g.q_ops.tolist()):
            if v not in seen:
                keep[i] = True
                seen.add(v)
        qid = np.repeat(np.arange(len(g.q_off) - 1), np.diff(g.q_off))
        g.q_ops = g.q_ops[keep]
        g.q_off = np.concatenate([[0], np.cumsum(np.bincount(qid[keep], minlength=len(g.q_off) - 1))])
        sc = SG.random_scenarios(rng, g, 1)
        sc.dur[:, 0] = rng.integers(0, 50, size=g.n_ops)
        a = oracle.compose(g, sc, refine_passes=0)
        preds = SG.merged_preds(g)
        c = int(rng.integers(1, 1000))
        for v in range(g.n_ops):
            if not preds[v]:
                sc.dur[v, 0] += c
        b = oracle.compose(g, sc, refine_passes=0)
        assert (b.finish == a.finish + c).all()


def test_scenario_permutation_and_duplication():
    c = W.config("gpt1.3b")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c, n_scen=4)
    a = oracle.compose(g, sc)
    cols = [2, 0, 3, 3, 1]
    b = oracle.compose(g, W.select_scenarios(sc, g, cols))
    assert (b.finish == a.finish[:, cols]).all()
    assert (b.start == a.start[:, cols]).all()
    assert (b.makespan == a.makespan[cols]).all()


def test_collective_starts_when_last_member_launches():
    # Sec. 5.2: three ranks compute 10, 20 and 30 ns, then join one all-reduce of
    # fixed cost 100 ns; every member sees it start at 30 and finish at 130, and
    # each rank's next kernel (which consumes the result) starts at 130.
    ops = [{"kind": W.KIND_COMPUTE} for _ in range(3)]
    ops.append({"kind": W.KIND_COLL, "group": 0, "cc_type": W.CC_ALLREDUCE,
                "cc_algo": W.ALGO_RING, "cc_bytes": 1, "preds": [0, 1, 2]})
    ops += [{"kind": W.KIND_COMPUTE, "preds": [3]} for _ in range(3)]
    queues = {(0, 0): [0, 4], (1, 0): [1, 5], (2, 0): [2, 6], (0, 1): [3], (1, 1): [3], (2, 1): [3]}
    g = SG.graph_from_lists(3, 2, ops, queues, [[0, 1, 2]])
    dur = np.array([[10], [20], [30], [0], [5], [5], [5]], np.int64)
    r = oracle.compose(g, _scen_fixed(1, dur=dur, alpha=100.0), refine_passes=0)
    assert r.start[3, 0] == 30 and r.finish[3, 0] == 130
    assert (r.start[4:, 0] == 130).all() and r.makespan[0] == 135


def test_overlap_slows_the_whole_kernel():
    # one rank: kernel A [0,50), kernel B [50,150) and a send/recv of fixed cost 100
    # that waits for A, so it runs [50,150) beside B.  With factor 1.5 the validator
    # stretches B to 150 ns: B [50,200), makespan 200.  A only touches the comm
    # interval, so it is not slowed.
    ops = [{"kind": W.KIND_COMPUTE, "kclass": 0}, {"kind": W.KIND_COMPUTE, "kclass": 0},
           {"kind": W.KIND_P2P, "group": 0, "cc_type": W.CC_SENDRECV, "cc_bytes": 1, "preds": [0]}]
    queues = {(0, 0): [0, 1], (0, 1): [2], (1, 1): [2]}
    g = SG.graph_from_lists(2, 2, ops, queues, [[0, 1]])
    dur = np.array([[50], [100], [0]], np.int64)
    r0 = oracle.compose(g, _scen_fixed(1, sf=1.5, dur=dur, alpha=100.0), refine_passes=0)
    assert list(r0.start[:, 0]) == [0, 50, 50] and list(r0.finish[:, 0]) == [50, 150, 150]
    r = oracle.compose(g, _scen_fixed(1, sf=1.5, dur=dur, alpha=100.0), refine_passes=1)
    assert list(r.overlapped[:, 0]) == [0, 1, 0]
    assert list(r.start[:, 0]) == [0, 50, 50] and list(r.finish[:, 0]) == [50, 200, 150]
    assert r.makespan[0] == 200


def test_unit_slowdown_or_no_comm_leaves_times_unchanged():
    c = W.config("tiny")
    g = W.build_gpt_graph(c)
    sc = W.make_scenarios(g, c)
    sc.slowdown[:] = 1.0
    a = oracle.compose(g, sc, refine_passes=0)
    b = oracle.compose(g, sc, refine_passes=1)
    assert (a.finish == b.finish).all() and b.overlapped.any()
    rng = np.random.default_rng(25)
    for _ in range(100):
        gg = SG.random_graph(rng, int(rng.integers(1, 20)))
        gg.kind[(gg.kind == W.KIND_COLL) | (gg.kind == W.KIND_P2P)] = W.KIND_MEMCPY
        s2 = SG.random_scenarios(rng, gg, 2)
        x = oracle.compose(gg, s2, refine_passes=0)
        y = oracle.compose(gg, s2, refine_passes=2)
        assert (x.finish == y.finish).all() and not y.overlapped.any()


def test_cycle_is_reported():
    ops = [{"kind": W.KIND_COMPUTE, "preds": [1]}, {"kind": W.KIND_COMPUTE}]
    g = SG.graph_from_lists(1, 2, ops, {(0, 0): [0, 1]}, [])
    with pytest.raises(RuntimeError, match="cycle"):
        oracle.compose(g, _scen_fixed(1, dur=np.ones((2, 1), np.int64)))


def test_empty_graph_and_no_scenarios():
    g = SG.graph_from_lists(1, 2, [], {}, [])
    r = oracle.compose(g, _scen_fixed(3, dur=np.zeros((0, 3), np.int64)))
    assert (r.makespan == 0).all()


def test_overlap_candidates_cover_every_overlap():
    # the library's static candidate set (host analysis) must contain every kernel
    # that the oracle's validator ever slows, in any scenario and variant; and it is
    # a real filter on the GPT workloads
    from paper_2412_12487_gb300.echo import overlap_candidates
    rng = np.random.default_rng(4040)
    for case in range(120):
        g = SG.random_graph(rng, int(rng.integers(2, 40)), max_ranks=4, max_streams=5,
                            p_edge=float(rng.choice([0.03, 0.1, 0.25])))
        cand = overlap_candidates(g).astype(bool)
        assert not cand[g.kind != W.KIND_COMPUTE].any()
        sc = SG.random_scenarios(rng, g, 6, max_dur=int(rng.choice([5, 40, 400])))
        for civ in (0, 1):
            for model in (0, 1):
                r = oracle.compose(g, sc, refine_passes=2, overlap_model=model, comm_interval=civ)
                slowed = r.overlapped.any(axis=1).astype(bool)
                assert not (slowed & ~cand).any(), (case, civ, model, np.nonzero(slowed & ~cand)[0])
    for name, lo, hi in (("tiny", 0.05, 0.6), ("gpt1.3b", 0.05, 0.3)):
        c = W.config(name)
        g = W.build_gpt_graph(c)
        cand = overlap_candidates(g).astype(bool)
        comp = g.kind == W.KIND_COMPUTE
        assert lo < cand.sum() / comp.sum() < hi, (name, cand.sum() / comp.sum())
        r = oracle.compose(g, W.make_scenarios(g, c, n_scen=4), refine_passes=1, comm_interval=1)
        assert not (r.overlapped.any(axis=1).astype(bool) & ~cand).any()
