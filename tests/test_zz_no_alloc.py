"""The allocation-free search entry point, nest_knn_search_static.

Callers that must not allocate device memory during a step (an application
whose own allocator owns the GPU's memory, or a serving loop that may never
run a device-synchronizing cudaMalloc/cudaFree) use nest_knn_search_static,
which keeps the search's candidate lists in a fixed array compiled into the
library instead of handle-owned scratch.  This file checks, through the C
ABI:

* its results against nest_knn_search on the same inputs, for two calls in
  a row (the shared array keeps the first call's contents), on the narrow
  scan, the ragged scan, the large-batch path and its CTA-pair kernels, each
  right after a call of another shape;
* one case against the fp64 oracle directly;
* that a call on a fresh handle takes no device memory (the free memory the
  driver reports does not change), while nest_knn_search on another fresh
  handle does;
* that a search too large for the array is refused before anything runs.

The file name makes pytest collect it last.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from parity import check_search, dist_rel_tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _inputs(seed, N=50003, d=1024, centres=16):
    g = torch.Generator().manual_seed(seed)
    c = torch.randn(centres, d, generator=g)
    K = c[torch.randint(0, centres, (N,), generator=g)] + 0.3 * torch.randn(N, d, generator=g)
    V = torch.randint(0, 1000, (N,), generator=g, dtype=torch.int32)
    return K.to(torch.bfloat16).cuda(), V.cuda()


def _queries(seed, K, B):
    g = torch.Generator().manual_seed(seed)
    pick = torch.randint(0, K.shape[0], (B,), generator=g)
    q = K[pick.cuda()].float() + 0.05 * torch.randn(B, K.shape[1], generator=g).cuda()
    return q.to(torch.bfloat16).contiguous()


def _call(lib, fn, ds, q, r, seg_off=None):
    B = q.shape[0]
    s = torch.empty(B, r, dtype=torch.float32, device="cuda")
    idx = torch.empty(B, r, dtype=torch.int64, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    rc = getattr(lib, fn)(ds.handle, q.data_ptr(), B, r,
                          seg_off.data_ptr() if seg_off is not None else None,
                          s.data_ptr(), idx.data_ptr(), stream)
    return rc, s, idx


def _same_search(s_a, i_a, s_b, i_b):
    """Equal neighbour sets per row; distances equal within the bf16 tolerance."""
    s_a, s_b = s_a.cpu().double().numpy(), s_b.cpu().double().numpy()
    i_a, i_b = i_a.cpu().numpy(), i_b.cpu().numpy()
    rel = dist_rel_tol("bf16")
    for b in range(s_a.shape[0]):
        assert set(i_a[b].tolist()) == set(i_b[b].tolist()), f"row {b}: neighbour sets differ"
        real = i_a[b] >= 0
        db = dict(zip(i_b[b].tolist(), (-s_b[b]).tolist()))
        Da = -s_a[b][real]
        Db = np.array([db[int(k)] for k in i_a[b][real]])
        assert np.all(np.abs(Da - Db) <= rel * np.abs(Db)), f"row {b}: distances differ"


def _static_then_reference(nest, lib, ds, q, r, seg_off=None):
    rc, s_st, i_st = _call(lib, "nest_knn_search_static", ds, q, r, seg_off)
    assert rc == 0, f"static search: status {rc}"
    rc, s_ref, i_ref = _call(lib, "nest_knn_search", ds, q, r, seg_off)
    assert rc == 0
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    _same_search(s_st, i_st, s_ref, i_ref)
    return s_st, i_st


def test_static_search_matches_search_on_two_calls_in_a_row(nest):
    lib = nest.load_library()
    K, V = _inputs(1)
    ds = nest.Datastore(K, V, 1000)
    assert ds.search_path(4, 256) == "tc_scan_kernel"
    for seed in (10, 11):
        _static_then_reference(nest, lib, ds, _queries(seed, K, 4), 256)
    ds.close()


def test_static_search_ragged_matches_search(nest):
    lib = nest.load_library()
    K, V = _inputs(2, N=20000, d=512)
    ds = nest.Datastore(K, V, 1000)
    off = torch.tensor([0, 3000, 3000, 9000, 9005, 20000], dtype=torch.int64, device="cuda")
    # a full scan of another shape first: the array holds its words
    _static_then_reference(nest, lib, ds, _queries(19, K, 3), 100)
    for seed in (20, 21):
        _static_then_reference(nest, lib, ds, _queries(seed, K, 5), 64, seg_off=off)
    ds.close()


def test_static_search_large_batch_path_after_another_shape(nest):
    """The large-batch path (its counters in the shared array start from a
    memset on every call), right after a narrow search left other words at
    those offsets, then again with another batch."""
    lib = nest.load_library()
    K, V = _inputs(4, N=20000, d=128, centres=12)
    ds = nest.Datastore(K, V, 1000)
    assert ds.search_path(32, 16) == "tc_wide_kernel"
    _static_then_reference(nest, lib, ds, _queries(40, K, 3), 500)
    for seed in (41, 42):
        _static_then_reference(nest, lib, ds, _queries(seed, K, 32), 16)
    ds.close()


def test_static_search_on_cta_pairs(nest):
    """Batches of 129 to 512 queries run on CTA pairs (clusters of two CTAs)
    by default; through the static entry point too, as one group of 256
    (B = 200) and as one group of 512 (B = 300), each twice in a row after a
    narrow search of another shape."""
    lib = nest.load_library()
    for B, N in ((200, 4000), (300, 2500)):
        K, V = _inputs(7 + B, N=N, d=128, centres=10)
        ds = nest.Datastore(K, V, 1000)
        assert ds.search_path(B, 16) == "tc_wide_pair_kernel"
        _static_then_reference(nest, lib, ds, _queries(70 + B, K, 2), 300)
        for seed in (71 + B, 72 + B):
            _static_then_reference(nest, lib, ds, _queries(seed, K, B), 16)
        ds.close()


def test_static_search_matches_the_oracle(nest):
    lib = nest.load_library()
    K, V = _inputs(5, N=30011, d=256)
    ds = nest.Datastore(K, V, 1000)
    q = _queries(50, K, 6)
    r = 200
    for _ in range(2):
        rc, s, idx = _call(lib, "nest_knn_search_static", ds, q, r)
        assert rc == 0
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        K_np, q_np = synth.to_numpy_raw(K), synth.to_numpy_raw(q)
        s_or, i_or = oracle.knn_search(K_np, q_np, r)
        check_search(s.cpu().numpy(), idx.cpu().numpy(), s_or, i_or, K_np, q_np, "bf16",
                     np.full(q.shape[0], K.shape[0]))
    ds.close()


def test_static_search_takes_no_device_memory(nest):
    """On a fresh handle (whose own scratch is still unallocated), a static
    search leaves the device's free memory unchanged; nest_knn_search on
    another fresh handle allocates its scratch, which the same measurement
    sees.  An earlier call loads every kernel, so module loading is not
    counted."""
    lib = nest.load_library()
    K, V = _inputs(6, N=200000, d=1024)
    q = _queries(60, K, 4)
    warm = nest.Datastore(K, V, 1000)
    assert _call(lib, "nest_knn_search_static", warm, q, 1024)[0] == 0
    assert _call(lib, "nest_knn_search", warm, q, 1024)[0] == 0
    torch.cuda.synchronize()
    warm.close()

    outs = [torch.empty(4, 1024, dtype=torch.float32, device="cuda"),
            torch.empty(4, 1024, dtype=torch.int64, device="cuda")]
    stream = torch.cuda.current_stream().cuda_stream

    def free_after(fn, ds):
        torch.cuda.synchronize()
        before = torch.cuda.mem_get_info()[0]
        rc = getattr(lib, fn)(ds.handle, q.data_ptr(), 4, 1024, None, outs[0].data_ptr(),
                              outs[1].data_ptr(), stream)
        torch.cuda.synchronize()
        assert rc == 0
        return before - torch.cuda.mem_get_info()[0]

    ds = nest.Datastore(K, V, 1000)
    assert free_after("nest_knn_search_static", ds) == 0
    assert free_after("nest_knn_search_static", ds) == 0
    ds.close()
    ds = nest.Datastore(K, V, 1000)
    assert free_after("nest_knn_search", ds) > 0
    ds.close()


def test_static_search_refuses_searches_beyond_the_array(nest):
    lib = nest.load_library()
    K, V = _inputs(3, N=300000, d=64)
    ds = nest.Datastore(K, V, 1000)
    q = _queries(30, K, 512)
    rc, _, _ = _call(lib, "nest_knn_search_static", ds, q, 4096)
    assert rc == nest.nest.STATUS_CODE["NEST_ERR_OVERFLOW"]
    ds.close()
