"""The allocation-free CC query entry point against the allocating one.

echo_cc_query_noalloc is for callers that cannot call cudaMalloc, for example a
process whose device memory belongs to a framework's memory pool, or one that runs
under a fixed device-memory budget.  Such a caller hands the library its own device
arrays.  This test does the same with torch device tensors, calls the entry point
twice in a row on different batches, and checks each result against
echo_cc_query within the tolerance of the other CC estimator tests.  The file
sorts last so that, if it fails, a run that stops at the first failure has
already run every other test.
"""
import ctypes as C

import numpy as np
import pytest

from paper_2412_12487_gb300 import Echo
from paper_2412_12487_gb300 import build as B
from paper_2412_12487_gb300 import echo as E
from paper_2412_12487_gb300 import workloads as W

pytestmark = pytest.mark.gpu
CC_RTOL = 1e-9


def _device_desc(q, keep):
    import torch

    def dev(x, dt):
        t = torch.from_numpy(np.ascontiguousarray(x, dtype=dt)).cuda()
        keep.append(t)
        return t.data_ptr()

    return E.CCQueryDesc(q.n, dev(q.cc_type, np.uint8), dev(q.cc_algo, np.uint8), dev(q.nbytes, np.int64),
                         dev(q.n_ranks, np.int32), dev(q.n_nodes, np.int32), dev(q.alpha_ns, np.float64),
                         dev(q.bw_intra, np.float64), dev(q.lat_intra, np.float64),
                         dev(q.bw_inter, np.float64), dev(q.lat_inter, np.float64),
                         dev(q.delta, np.float64), 0, None, None)


def _call(lib, q, stream):
    import torch
    keep = []
    desc = _device_desc(q, keep)
    out = torch.full((q.n,), float("nan"), dtype=torch.float64, device="cuda")
    rc = lib.echo_cc_query_noalloc(C.byref(desc), C.c_void_p(out.data_ptr()), C.c_void_p(stream.cuda_stream))
    return rc, out.cpu().numpy()


def test_noalloc_cc_query_matches_allocating_entry_point():
    import torch
    B.build()
    lib = E.load_library()
    stream = torch.cuda.current_stream()
    for n, seed in [(100_003, 11), (4_099, 12)]:   # two calls in a row
        q = W.make_cc_queries(n, seed=seed)
        with Echo(0) as e:
            want = e.cc_query(q)
        rc, got = _call(lib, q, stream)
        assert rc == 0
        np.testing.assert_allclose(got, want, rtol=CC_RTOL, atol=0)


def test_noalloc_rejects_node_counts_beyond_its_table():
    import torch
    lib = E.load_library()
    stream = torch.cuda.current_stream()
    q = W.make_cc_queries(1000, seed=13)
    q.n_ranks[5] = 200_000
    q.n_nodes[5] = 70_000
    rc, got = _call(lib, q, stream)
    assert rc == 9  # ECHO_E_UNSUPPORTED
    assert np.isnan(got[5]) and np.isfinite(np.delete(got, 5)).all()
    # the status word does not leak into the next call
    q2 = W.make_cc_queries(1000, seed=14)
    with Echo(0) as e:
        want = e.cc_query(q2)
    rc, got = _call(lib, q2, stream)
    assert rc == 0
    np.testing.assert_allclose(got, want, rtol=CC_RTOL, atol=0)


def test_noalloc_mixed_bad_queries_report_the_malformed_one():
    """A batch with both a malformed query and one whose node count exceeds the
    table returns ECHO_E_INVALID_ARG every time (the malformed query ranks first),
    with NaN for both and every other query estimated."""
    import torch
    lib = E.load_library()
    stream = torch.cuda.current_stream()
    q = W.make_cc_queries(5000, seed=15)
    bad = [17, 4000]              # M > N: malformed
    big = [3, 2500, 4999]         # M > 65536: beyond the table
    for i in bad:
        q.n_nodes[i] = q.n_ranks[i] + 1
    for i in big:
        q.n_ranks[i] = 300_000
        q.n_nodes[i] = 100_000
    for _ in range(5):
        rc, got = _call(lib, q, stream)
        assert rc == 1  # ECHO_E_INVALID_ARG
        assert np.isnan(got[bad + big]).all()
        assert np.isfinite(np.delete(got, bad + big)).all()
