"""The allocation-free search entry point, nest_knn_search_static.

Callers that must not allocate device memory during a step (an application
whose own allocator owns the GPU's memory, or a serving loop that may never
run a device-synchronizing cudaMalloc/cudaFree) use nest_knn_search_static,
which keeps the search's candidate lists in a fixed array compiled into the
library instead of handle-owned scratch.  This file checks it through the
C ABI against nest_knn_search on the same inputs, for two calls in a row
(the shared array keeps the first call's contents), and that a search too
large for the array is refused before anything runs.

The file name makes pytest collect it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from parity import FLOOR, dist_rel_tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _inputs(seed, N=50003, d=1024, B=4, centres=16):
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


def _same_search(s_a, i_a, s_b, i_b, K, q):
    """Equal neighbour sets per row; distances within the parity tolerance."""
    s_a, s_b = s_a.cpu().double().numpy(), s_b.cpu().double().numpy()
    i_a, i_b = i_a.cpu().numpy(), i_b.cpu().numpy()
    qn = q.float().pow(2).sum(1).cpu().double().numpy()
    kn_all = K.float().pow(2).sum(1).cpu().double().numpy()
    rel = dist_rel_tol("bf16")
    for b in range(s_a.shape[0]):
        assert set(i_a[b].tolist()) == set(i_b[b].tolist()), f"row {b}: neighbour sets differ"
        real = i_a[b] >= 0
        ka = i_a[b][real]
        db = dict(zip(i_b[b].tolist(), (-s_b[b]).tolist()))
        Da = -s_a[b][real]
        Db = np.array([db[int(k)] for k in ka])
        bound = rel * np.abs(Db) + FLOOR * (qn[b] + kn_all[ka])
        assert np.all(np.abs(Da - Db) <= bound), f"row {b}: distances differ"


def test_static_search_matches_search_on_two_calls_in_a_row(nest):
    lib = nest.load_library()
    K, V = _inputs(1)
    ds = nest.Datastore(K, V, 1000)
    r = 256
    for call, seed in enumerate((10, 11)):
        q = _queries(seed, K, 4)
        rc, s_st, i_st = _call(lib, "nest_knn_search_static", ds, q, r)
        assert rc == 0, f"call {call}: status {rc}"
        rc, s_ref, i_ref = _call(lib, "nest_knn_search", ds, q, r)
        assert rc == 0
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        _same_search(s_st, i_st, s_ref, i_ref, K, q)
    ds.close()


def test_static_search_ragged_matches_search(nest):
    lib = nest.load_library()
    K, V = _inputs(2, N=20000, d=512)
    ds = nest.Datastore(K, V, 1000)
    off = torch.tensor([0, 3000, 3000, 9000, 9005, 20000], dtype=torch.int64, device="cuda")
    for seed in (20, 21):
        q = _queries(seed, K, 5)
        rc, s_st, i_st = _call(lib, "nest_knn_search_static", ds, q, 64, seg_off=off)
        assert rc == 0
        rc, s_ref, i_ref = _call(lib, "nest_knn_search", ds, q, 64, seg_off=off)
        assert rc == 0
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        _same_search(s_st, i_st, s_ref, i_ref, K, q)
    ds.close()


def test_static_search_refuses_searches_beyond_the_array(nest):
    lib = nest.load_library()
    K, V = _inputs(3, N=300000, d=64)
    ds = nest.Datastore(K, V, 1000)
    q = _queries(30, K, 512)
    rc, _, _ = _call(lib, "nest_knn_search_static", ds, q, 4096)
    assert rc == nest.nest.STATUS_CODE["NEST_ERR_OVERFLOW"]
    ds.close()
