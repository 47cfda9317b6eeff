"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Seeded synthetic inputs shaped like the paper's workloads (tiny fp32 case,
decode-batch full scan, ragged second-stage search) plus edge cases: ragged
tails, d not a multiple of 64, B not a multiple of the query group, r > N,
r = N, r = 1, empty and short segments, exact ties on integer lattices, a key
equal to the query, the largest row and the largest r.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from parity import check_mix, check_mix_end_to_end, check_search

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _np(t):
    return synth.to_numpy_raw(t)


def _cand_counts(B, N, seg_off):
    if seg_off is None:
        return np.full(B, N)
    so = seg_off.cpu().numpy()
    return so[1:] - so[:-1]


def run_and_check(nest, K, V, q, p_lm, r, mu, lam, vocab, dtype, seg_off=None, exact=False,
                  oracle_threads=None, check_rows=None, pairs=None, label=None):
    """GPU step through the C ABI, then the oracle on the same bytes.

    ``check_rows`` restricts the oracle (and the comparison) to those query
    rows of a full-scan batch; the GPU always runs the whole batch.
    ``pairs`` chooses CTA pairs or single CTAs for groups of 256 queries.
    """
    dev = torch.device("cuda")
    K, V, q, p_lm = K.to(dev), V.to(dev), q.to(dev), p_lm.to(dev)
    so = seg_off.to(dev) if seg_off is not None else None
    ds = nest.Datastore(K, V, vocab)
    if pairs is not None:
        ds.use_cta_pairs(pairs)
    out = ds.step(q, r, p_lm, mu, lam, seg_off=so, want_p_knn=True)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    rows_sel = slice(None) if check_rows is None else list(check_rows)
    s_g = out["s"].cpu().numpy()[rows_sel]
    i_g = out["idx"].cpu().numpy()[rows_sel]
    K_np, V_np = _np(K), V.cpu().numpy()
    q_np = _np(q)[rows_sel]
    p_lm_np = p_lm.cpu().numpy()[rows_sel]
    so_np = seg_off.cpu().numpy() if seg_off is not None else None
    ref = oracle.knn_step(K_np, V_np, q_np, r, p_lm_np, mu, lam, vocab, seg_off=so_np,
                          nthreads=oracle_threads)
    rows = check_search(s_g, i_g, ref["s"], ref["idx"], K_np, q_np, dtype,
                        _cand_counts(q_np.shape[0], K.shape[0], seg_off), exact=exact,
                        label=label)
    p_m = out["p_m"].cpu().numpy()[rows_sel]
    check_mix(p_m, s_g, i_g, V_np, p_lm_np, mu, lam, vocab,
              p_knn_gpu=out["p_knn"].cpu().numpy()[rows_sel])
    check_mix_end_to_end(p_m, ref["p_m"], rows)
    ds.close()
    return out, ref, rows


# ---------------------------------------------------------------- the paper-shaped workloads

def test_tiny_workload(nest):
    w = synth.WORKLOADS["tiny"]
    x = synth.make_inputs(w)
    _, _, rows = run_and_check(nest, x.K, x.V, x.q, x.p_lm, w.r, w.mu, w.lam, w.vocab, w.dtype,
                               label="config 1: tiny fp32 d=64")
    assert len(rows) == w.B


def test_decode_workload_full_size(nest):
    """bf16 d=4096, N=1,048,576 clustered keys, B=4, r=1024: the benchmarked launch."""
    w = synth.WORKLOADS["decode"]
    x = synth.make_inputs(w, device="cuda")
    run_and_check(nest, x.K, x.V, x.q, x.p_lm, w.r, w.mu, w.lam, w.vocab, w.dtype,
                  label="config 2: decode, 1M keys, d=4096, r=1024")


def test_ragged_workload_full_size(nest):
    """32 queries x 40 passages x 256 keys, segment offsets, r=64."""
    w = synth.WORKLOADS["ragged"]
    x = synth.make_inputs(w, device="cuda")
    _, _, rows = run_and_check(nest, x.K, x.V, x.q, x.p_lm, w.r, w.mu, w.lam, w.vocab, w.dtype,
                               seg_off=x.seg_off, label="config 3: ragged, 32 x 10,240 keys")
    assert len(rows) >= w.B // 2


# ---------------------------------------------------------------- shapes and edges

def _random_case(N, d, B, vocab, dtype, seed, centres=8):
    g = torch.Generator().manual_seed(seed)
    c = torch.randn(centres, d, generator=g)
    K = (c[torch.randint(0, centres, (N,), generator=g)] + 0.3 * torch.randn(N, d, generator=g))
    q = (c[torch.randint(0, centres, (B,), generator=g)] + 0.3 * torch.randn(B, d, generator=g))
    dt = synth.torch_dtype(dtype)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g) * 2, dim=1)
    return K.to(dt), V, q.to(dt), p_lm


@pytest.mark.parametrize("N,d,B,r,dtype", [
    (20003, 72, 5, 33, "bf16"),      # ragged tail, d % 64 != 0, B % 4 != 0
    (4099, 8, 3, 7, "bf16"),         # smallest bf16 row (16 bytes)
    (3001, 4096, 2, 100, "f32"),     # fp32 4096: four chunks per thread, two queries
    (2500, 8192, 1, 64, "bf16"),     # largest row (16 KiB), one query
    (5000, 256, 9, 1, "f32"),        # r = 1
    (9000, 128, 4, 2048, "bf16"),    # r > 1024: fewer queries per CTA
    (1500, 64, 1, 4096, "f32"),      # r = NEST_MAX_R > N: padded rows
    (600, 16, 6, 600, "f32"),        # r = N
    (12, 32, 4, 16, "f32"),          # r > N, N below one stage per CTA
])
def test_shapes(nest, N, d, B, r, dtype):
    K, V, q, p_lm = _random_case(N, d, B, 500, dtype, seed=N + d)
    run_and_check(nest, K, V, q, p_lm, r, 1 / np.sqrt(d), 0.7, 500, dtype)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_integer_lattice_is_bit_exact_with_ties(nest, dtype):
    """Small-integer keys: distances exact in fp32, many exact ties -> identical lists."""
    g = torch.Generator().manual_seed(11)
    N, d, B, r = 7000, 16, 6, 300
    K = torch.randint(-3, 4, (N, d), generator=g).float()
    q = torch.randint(-3, 4, (B, d), generator=g).float()
    dt = synth.torch_dtype(dtype)
    V = torch.randint(0, 50, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, 50, generator=g), dim=1)
    run_and_check(nest, K.to(dt), V, q.to(dt), p_lm, r, 0.25, 0.6, 50, dtype, exact=True)


def test_duplicate_keys_tie_break_by_index(nest):
    g = torch.Generator().manual_seed(12)
    base = torch.randn(50, 32, generator=g)
    K = base.repeat(40, 1)  # every key appears 40 times
    q = base[:4] + 0.01
    V = torch.randint(0, 20, (K.shape[0],), generator=g, dtype=torch.int32)
    p_lm = torch.full((4, 20), 1 / 20)
    out, ref, _ = run_and_check(nest, K, V, q, p_lm, 100, 0.2, 0.5, 20, "f32")
    # copies of the nearest key come first, in index order
    i = out["idx"].cpu().numpy()
    for b in range(4):
        assert i[b, :40].tolist() == list(range(b, 2000, 50))


def test_key_equal_to_query_is_first_with_distance_zero(nest):
    g = torch.Generator().manual_seed(13)
    K = torch.randn(10000, 128, generator=g).to(torch.bfloat16)
    q = K[[17, 9999, 4242]].clone()
    V = torch.randint(0, 100, (10000,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(3, 100, generator=g), dim=1)
    out, _, _ = run_and_check(nest, K, V, q, p_lm, 10, 1 / np.sqrt(128), 0.8, 100, "bf16")
    assert out["idx"][:, 0].cpu().tolist() == [17, 9999, 4242]


@pytest.mark.parametrize("r", [1024, 4096])
def test_narrow_scan_keys_stored_cluster_by_cluster(nest, r):
    """Keys stored cluster after cluster: a query's nearest keys all sit in
    the two or three key ranges that hold its cluster, so those ranges'
    candidate lists hold far more of the r' nearest than their 32-word
    summaries, and the two-phase merge must read them whole (r = 1024: in
    shared memory at once; r = 4096: more than it holds, one list at a time).
    bf16, d=128, N=200,000 in 64 contiguous clusters, B=4."""
    N, d, B, vocab = 200000, 128, 4, 500
    g = torch.Generator().manual_seed(61 + r)
    c = torch.randn(64, d, generator=g)
    assign = torch.arange(N) // (N // 64)
    assign.clamp_(max=63)
    K = (c[assign] + 0.3 * torch.randn(N, d, generator=g)).to(torch.bfloat16)
    q = (c[torch.tensor([5, 5, 40, 63])] + 0.3 * torch.randn(B, d, generator=g)).to(torch.bfloat16)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g), dim=1)
    plan = nest.plan_offline(N, d, "bf16", B, r)
    assert plan["path"] == 1 and plan["parts"] >= 64, plan
    run_and_check(nest, K, V, q, p_lm, r, 1 / np.sqrt(d), 0.7, vocab, "bf16")


def test_margin_check_reports_a_crowded_boundary(nest):
    """Keys whose exact distances are packed closer than the fp32 screening
    error: integer vectors of about 1,000-norm-squared per element (||q||^2 and
    ||k||^2 near 3.7e7, so ||q||^2 + ||k||^2 - 2 q.k carries errors of several
    units), each the query plus a and b in two positions (a, b < 16), so
    D = a^2 + b^2 exactly.  Hundreds of keys lie within the screening error of
    the 16th distance, far more than the 16 extra candidates the re-ranking
    keeps.  The search must either return the oracle's neighbours or report
    NEST_ERR_MARGIN; on this data it reports it."""
    g = torch.Generator().manual_seed(77)
    d, N, r = 1024, 4096, 16
    c = torch.randint(128, 256, (d,), generator=g).float()
    K = c.repeat(N, 1)
    i = torch.arange(N)
    a = torch.randint(0, 16, (N,), generator=g).float()
    b = torch.randint(0, 16, (N,), generator=g).float()
    K[i, i % 1000] += a
    K[i, (7 * i + 3) % 1000 + 1] += b
    K = K.to(torch.bfloat16)
    assert torch.equal(K.float(), K.float().round())  # integers, exact in bf16
    q = c.to(torch.bfloat16).repeat(2, 1)
    V = torch.randint(0, 10, (N,), generator=g, dtype=torch.int32)
    ds = nest.Datastore(K.cuda(), V.cuda(), 10)
    s, idx = ds.search(q.cuda(), r)
    torch.cuda.synchronize()
    st = ds.device_status()
    ds.close()
    K_np, q_np = _np(K), _np(q)
    s_or, i_or = oracle.knn_search(K_np, q_np, r)
    if st == 0:
        check_search(s.cpu().numpy(), idx.cpu().numpy(), s_or, i_or, K_np, q_np, "bf16",
                     np.full(2, N), exact=True)
    else:
        assert st == nest.nest.STATUS_CODE["NEST_ERR_MARGIN"]
        # the rows still hold r distinct keys with exact distances, nearest first
        D = -s.cpu().double().numpy()
        D_ex = oracle.sqdist(K_np[idx.cpu().numpy()[0]], q_np[:1])[0]
        assert np.array_equal(D[0], D_ex) and np.all(np.diff(D[0]) >= 0)
    assert st == nest.nest.STATUS_CODE["NEST_ERR_MARGIN"], "expected the crowded boundary flagged"


def test_ragged_edges(nest):
    """Empty segment, segments shorter than r, unequal lengths, one long segment."""
    g = torch.Generator().manual_seed(14)
    lens = [0, 5, 37, 300, 4000, 0, 64, 1]
    N = sum(lens) + 10
    K = torch.randn(N, 256, generator=g).to(torch.bfloat16)
    B = len(lens)
    q = torch.randn(B, 256, generator=g).to(torch.bfloat16)
    off = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int64) + 3
    V = torch.randint(0, 77, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, 77, generator=g), dim=1)
    out, _, _ = run_and_check(nest, K, V, q, p_lm, 64, 1 / 16, 0.7, 77, "bf16", seg_off=off)
    # an empty segment has no neighbours, so p_M = p_LM there
    p_m = out["p_m"].cpu()
    assert torch.equal(p_m[0], p_lm[0]) and torch.equal(p_m[5], p_lm[5])


def test_mix_rrc_matches_eq4(nest):
    w = synth.WORKLOADS["tiny"]
    x = synth.make_inputs(w)
    dev = torch.device("cuda")
    ds = nest.Datastore(x.K.to(dev), x.V.to(dev), w.vocab)
    s, idx = ds.search(x.q.to(dev), w.r)
    p_lm = x.p_lm.to(dev)
    for alpha, tau in [(0.3, 0.1), (0.2, 0.1), (0.9, 0.5)]:
        p_m, lam, p_knn = ds.mix_rrc(s, idx, p_lm, w.mu, alpha, tau, want_p_knn=True)
        torch.cuda.synchronize()
        s_np, i_np = s.cpu().numpy(), idx.cpu().numpy()
        lam_or = oracle.rrc(s_np.astype(np.float64), i_np, alpha, tau)
        np.testing.assert_allclose(lam.cpu().numpy(), lam_or, rtol=0, atol=1e-6)
        check_mix(p_m.cpu().numpy(), s_np, i_np, x.V.numpy(), x.p_lm.numpy(), w.mu, None,
                  w.vocab, p_knn_gpu=p_knn.cpu().numpy(), lam_gpu=lam.cpu().numpy())
    assert ds.device_status() == 0
    ds.close()


def test_mix_lambda_one_and_zero(nest):
    w = synth.WORKLOADS["tiny"]
    x = synth.make_inputs(w)
    dev = torch.device("cuda")
    ds = nest.Datastore(x.K.to(dev), x.V.to(dev), w.vocab)
    s, idx = ds.search(x.q.to(dev), w.r)
    p_lm = x.p_lm.to(dev)
    p1, k1 = ds.mix(s, idx, p_lm, w.mu, 1.0, want_p_knn=True)
    p0, k0 = ds.mix(s, idx, p_lm, w.mu, 0.0, want_p_knn=True)
    assert torch.equal(p1, p_lm)
    assert torch.equal(p0, k0) and torch.equal(k0, k1)
    np.testing.assert_allclose(k0.double().sum(1).cpu().numpy(), 1.0, atol=1e-5)
    ds.close()


# ---------------------------------------------------------------- device-side errors

def test_bad_segment_offsets_are_reported(nest):
    dev = torch.device("cuda")
    K = torch.randn(100, 16, device=dev)
    V = torch.zeros(100, dtype=torch.int32, device=dev)
    ds = nest.Datastore(K, V, 4)
    q = torch.randn(2, 16, device=dev)
    off = torch.tensor([0, 50, 40], dtype=torch.int64, device=dev)  # decreasing
    s, idx = ds.search(q, 5, seg_off=off)
    assert ds.device_status() == nest.nest.STATUS_CODE["NEST_ERR_INVALID_ARG"]
    assert (idx[1] == -1).all()
    assert ds.device_status() == 0  # cleared
    ds.close()


def test_out_of_range_neighbour_index_is_reported(nest):
    dev = torch.device("cuda")
    K = torch.randn(100, 16, device=dev)
    V = torch.zeros(100, dtype=torch.int32, device=dev)
    ds = nest.Datastore(K, V, 4)
    s = torch.tensor([[-1.0, -2.0]], device=dev)
    idx = torch.tensor([[3, 100]], dtype=torch.int64, device=dev)
    p_lm = torch.full((1, 4), 0.25, device=dev)
    p_m = ds.mix(s, idx, p_lm, 1.0, 0.5)
    assert ds.device_status() == nest.nest.STATUS_CODE["NEST_ERR_VALUE_RANGE"]
    # the bad neighbour carries no weight: token 0 gets all kNN mass
    np.testing.assert_allclose(p_m.cpu().numpy(), [[0.625, 0.125, 0.125, 0.125]], atol=1e-7)
    ds.close()


def test_create_rejects_out_of_range_values(nest):
    dev = torch.device("cuda")
    K = torch.randn(64, 16, device=dev)
    V = torch.arange(64, dtype=torch.int32, device=dev)
    with pytest.raises(nest.NestError) as e:
        nest.Datastore(K, V, 10)
    assert e.value.name == "NEST_ERR_VALUE_RANGE"


def test_host_validation_on_gpu(nest):
    dev = torch.device("cuda")
    K = torch.randn(64, 16, device=dev)
    V = torch.zeros(64, dtype=torch.int32, device=dev)
    ds = nest.Datastore(K, V, 10)
    q = torch.randn(1, 16, device=dev)
    with pytest.raises(nest.NestError) as e:
        ds.search(q, 0)
    assert e.value.name == "NEST_ERR_INVALID_ARG"
    with pytest.raises(nest.NestError) as e:
        ds.search(q, 5000)
    assert e.value.name == "NEST_ERR_INVALID_ARG"
    s, idx = ds.search(q, 3)
    with pytest.raises(nest.NestError) as e:
        ds.mix(s, idx, torch.full((1, 10), 0.1, device=dev), 1.0, 1.5)
    assert e.value.name == "NEST_ERR_INVALID_ARG"
    ds.close()


def test_timing_and_launch_count(nest):
    w = synth.WORKLOADS["tiny"]
    x = synth.make_inputs(w)
    dev = torch.device("cuda")
    ds = nest.Datastore(x.K.to(dev), x.V.to(dev), w.vocab)
    q, p_lm = x.q.to(dev), x.p_lm.to(dev)
    ds.timing_enable(True)
    n0 = ds.launch_count()
    for _ in range(3):
        ds.step(q, w.r, p_lm, w.mu, w.lam)
    ms, n = ds.timing_read()
    assert n == 3 and ms > 0
    assert ds.launch_count() - n0 >= 9  # scan + merge + mix per step
    ds.close()


def test_step_host_matches_device_step(nest):
    """nest_knn_step_host (host buffers in and out, one C call) gives the same
    bytes as nest_knn_step on device copies: pinned and pageable inputs, two
    batch sizes in a row (its device buffers grow), and a ragged batch."""
    dev = torch.device("cuda")
    w = synth.WORKLOADS["tiny"]
    x = synth.make_inputs(w)
    ds = nest.Datastore(x.K.to(dev), x.V.to(dev), w.vocab)
    staging = {}
    for B, pin in ((w.B, True), (3, False), (w.B, True)):
        q, p = x.q[:B].contiguous(), x.p_lm[:B].contiguous()
        if pin:
            q, p = q.pin_memory(), p.pin_memory()
        host = ds.step_host(q, w.r, p, w.mu, w.lam, staging=staging)
        o = ds.step(q.to(dev), w.r, p.to(dev), w.mu, w.lam)
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        assert torch.equal(host["p_m"], o["p_m"].cpu())
        assert torch.equal(host["s"], o["s"].cpu())
        assert torch.equal(host["idx"], o["idx"].cpu())
    ds.close()

    w = synth.WORKLOADS["ragged"]
    x = synth.make_inputs(w, B=5)
    ds = nest.Datastore(x.K.to(dev), x.V.to(dev), w.vocab)
    host = ds.step_host(x.q.pin_memory(), w.r, x.p_lm.pin_memory(), w.mu, w.lam,
                        seg_off_host=x.seg_off.pin_memory())
    o = ds.step(x.q.to(dev), w.r, x.p_lm.to(dev), w.mu, w.lam, seg_off=x.seg_off.to(dev))
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    assert torch.equal(host["p_m"], o["p_m"].cpu())
    assert torch.equal(host["idx"], o["idx"].cpu())
    ds.close()


# ---------------------------------------------------------------- large query batches

def test_wide_batch_with_sampled_thresholds(nest):
    """B=40 queries (more than one CTA keeps lists for at r=256): sample pass,
    thresholded pass, exact selection of the survivors."""
    K, V, q, p_lm = _random_case(200000, 256, 40, 700, "bf16", seed=21, centres=64)
    ds = nest.Datastore(K.cuda(), V.cuda(), 700)
    assert ds.search_path(40, 256) == "tc_wide_kernel"
    assert ds.search_path(4, 256) == "tc_scan_kernel"
    ds.close()
    run_and_check(nest, K, V, q, p_lm, 256, 1 / 16, 0.8, 700, "bf16")


def test_wide_batch_single_pass_over_300_queries(nest):
    """B=300 > 256 (two query groups); the datastore is small enough that the
    sample is every key."""
    K, V, q, p_lm = _random_case(100003, 128, 300, 500, "bf16", seed=22, centres=32)
    run_and_check(nest, K, V, q, p_lm, 64, 1 / np.sqrt(128), 0.8, 500, "bf16")


def _group256_path(pairs):
    return "tc_wide_pair_kernel" if pairs else "tc_wide2_kernel"


@pytest.mark.parametrize("pairs", [True, False], ids=["cta_pairs", "two_tiles"])
@pytest.mark.parametrize("N,d,B,r", [
    (200036, 200, 260, 64),   # two passes; last 256-key tile: part real, part past N
    (70017, 64, 256, 33),     # single pass, one full group, d = one K chunk, 1-row tile
])
def test_group256_wide_kernel_edges(nest, N, d, B, r, pairs):
    """Groups of 256 queries, on CTA pairs (256-key tiles split over two
    SMs) and on single CTAs (two 128-key tiles per pipeline stage): a
    partial last group (padding columns), d not a multiple of 64 (the last
    K chunk half outside the rows), and a last 256-key tile whose second
    half lies wholly past the last key.  On pairs B = 260 is one group of
    512 (252 padding columns) and B = 256 one group of 256."""
    K, V, q, p_lm = _random_case(N, d, B, 900, "bf16", seed=23 + d, centres=48)
    ds = nest.Datastore(K.cuda(), V.cuda(), 900)
    ds.use_cta_pairs(pairs)
    assert ds.search_path(B, r) == _group256_path(pairs)
    ds.close()
    rows = list(range(0, B, 7)) + [B - 1]
    run_and_check(nest, K, V, q, p_lm, r, 1 / np.sqrt(d), 0.7, 900, "bf16", check_rows=rows,
                  pairs=pairs)


@pytest.mark.parametrize("N,r,masked", [
    (119, 4096, True),    # r above N, every list shorter than one warp's stride
    (119, 32, False),
    (8269, 64, False),    # 8269 = 8192 + 77: the last copy trip splits a warp
])
def test_wide_batch_list_lengths_that_split_a_warp(nest, N, r, masked):
    """Batches over a datastore small enough for one pass: each query's list
    holds N words, and when N mod 8192 is below 1024 and not a multiple of 32
    some warp of the selection kernel has lanes with and lanes without a
    word on the last copy trip.  bf16, d=72, B=100."""
    B, d, vocab = 100, 72, 500
    K, V, q, p_lm = _random_case(N, d, B, vocab, "bf16", seed=N + r)
    ds = nest.Datastore(K.cuda(), V.cuda(), vocab)
    assert ds.search_path(B, r) == "tc_wide_kernel"
    if not masked:
        ds.close()
        run_and_check(nest, K, V, q, p_lm, r, 1 / np.sqrt(d), 0.7, vocab, "bf16",
                      check_rows=list(range(0, B, 11)) + [B - 1])
        return
    excl = np.zeros(N, bool)
    excl[30:47] = True
    excl[::7] = True
    words = np.zeros((N + 31) // 32, dtype=np.uint32)
    for k in np.flatnonzero(excl):
        words[k >> 5] |= np.uint32(1 << (k & 31))
    mask = torch.from_numpy(words.view(np.int32)).cuda()
    s, idx = ds.search_masked(q.cuda(), r, mask)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    K_np, q_np = _np(K), _np(q)
    s_or, i_or = oracle.knn_search(K_np, q_np, r, exclude=excl)
    check_search(s.cpu().numpy(), idx.cpu().numpy(), s_or, i_or, K_np, q_np, "bf16",
                 np.full(B, N - int(excl.sum())))
    ds.close()


@pytest.mark.parametrize("pairs", [True, False], ids=["cta_pairs", "two_tiles"])
def test_wide_batch_keys_stored_cluster_by_cluster(nest, pairs):
    """Keys stored cluster after cluster (as a datastore built document by
    document would be): each query's main-pass survivors come from the one or
    two key ranges that hold its cluster, so the epilogue warps there use up
    their reserved list slots and go on one slot at a time.  bf16, d=256,
    N=262,144 in 64 contiguous clusters, B=512, r=256."""
    N, d, B, r, vocab = 262144, 256, 512, 256, 900
    g = torch.Generator().manual_seed(31)
    c = torch.randn(64, d, generator=g)
    assign = torch.arange(N) // (N // 64)
    K = (c[assign] + 0.3 * torch.randn(N, d, generator=g)).to(torch.bfloat16)
    q = (c[torch.randint(0, 64, (B,), generator=g)]
         + 0.3 * torch.randn(B, d, generator=g)).to(torch.bfloat16)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g) * 2, dim=1)
    ds = nest.Datastore(K.cuda(), V.cuda(), vocab)
    ds.use_cta_pairs(pairs)
    assert ds.search_path(B, r) == _group256_path(pairs)
    ds.close()
    rows = list(range(0, B, 37)) + [B - 1]
    run_and_check(nest, K, V, q, p_lm, r, 1 / 16, 0.8, vocab, "bf16", check_rows=rows,
                  pairs=pairs)


@pytest.mark.parametrize("pairs", [True, False], ids=["cta_pairs", "two_tiles"])
def test_wide_batch_massive_exact_ties(nest, pairs):
    """Groups of 256 queries over keys that are exact copies of two integer
    vectors (two of every three keys are the same vector): every query sees
    two distances, the r nearest are the r smallest indices among the nearer
    copies, and the bin of the r-th smallest word holds tens of thousands of
    words, more than the exact selection stages in shared memory.  Integer
    values keep the fp32 distances exact, so the lists must match bit for
    bit.  bf16, d=64, N=100,000 (one pass), B=300, r=64."""
    g = torch.Generator().manual_seed(41)
    N, d, B, r, vocab = 100000, 64, 300, 64, 500
    b0 = torch.randint(-2, 3, (d,), generator=g).float()
    b1 = b0.clone()
    b1[0] += 1
    K = torch.where((torch.arange(N) % 3 == 0)[:, None], b1, b0).to(torch.bfloat16)
    q = (b0 + torch.randint(-1, 2, (B, d), generator=g).float()).to(torch.bfloat16)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g), dim=1)
    ds = nest.Datastore(K.cuda(), V.cuda(), vocab)
    ds.use_cta_pairs(pairs)
    assert ds.search_path(B, r) == _group256_path(pairs)
    ds.close()
    rows = list(range(0, B, 23)) + [B - 1]
    run_and_check(nest, K, V, q, p_lm, r, 1 / 8, 0.7, vocab, "bf16", exact=True, check_rows=rows,
                  pairs=pairs)


@pytest.mark.parametrize("B", [40, 300])
def test_wide_batch_list_overflow_is_recovered(nest, B):
    """50,000 exact copies of one vector among 200,000 keys, and queries next
    to it: the sample's r-th distance is the copies' distance, so the
    thresholded pass admits every copy, far more than a query's list holds.
    The overflowed lists are scanned again with the r-th smallest word each
    holds as the limit (ties broken by key index), and the search returns the
    oracle's exact neighbours -- the copies with the smallest indices -- with
    no error.  B = 40 runs the groups-of-64 kernel, B = 300 one group of 512
    on CTA pairs (recovered as two groups of 256); bf16, d=64, r=16."""
    g = torch.Generator().manual_seed(91)
    N, d, r, vocab, n_copies = 200000, 64, 16, 300, 50000
    K = torch.randn(N, d, generator=g)
    v = torch.randn(d, generator=g)
    pos = torch.randperm(N, generator=g)[:n_copies]
    K[pos] = v
    K = K.to(torch.bfloat16)
    q = torch.randn(B, d, generator=g)
    near = torch.arange(0, B, 2)
    q[near] = v + 0.05 * torch.randn(len(near), d, generator=g)
    q = q.to(torch.bfloat16)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g), dim=1)
    plan = nest.plan_offline(N, d, "bf16", B, r)
    assert plan["path"] in (2, 4) and not plan["single_pass"]
    assert plan["list_capacity"] < n_copies  # every copy is admitted: the lists overflow
    rows = sorted(set(list(range(0, B, max(1, B // 12))) + [1, B - 1, B - 2]))
    out, ref, exact_rows = run_and_check(nest, K, V, q, p_lm, r, 1 / 8, 0.7, vocab, "bf16",
                                         check_rows=rows)
    copies = np.sort(pos.numpy())[:r]
    for j, b in enumerate(rows):
        if b % 2 == 0:
            assert out["idx"][b].cpu().numpy().tolist() == copies.tolist()


def test_wide_batch_threshold_underflow_is_rescanned(nest):
    """The main pass of a large batch admits keys up to the sample's j-th
    distance with j well below r' (here j = 37, r' = 272), expecting about
    4 r' keys of the datastore below it.  Here every key near the queries
    sits at a sampled position (400 of them, one every stride-th key), so
    only 37 keys pass: the list holds fewer than r' words, and the query is
    scanned again up to the sample's r'-th distance, which is safe.  The
    result must be the oracle's.  bf16, d=64, N=2,000,000, B=300 (one group
    of 512 on CTA pairs), r=256."""
    g = torch.Generator().manual_seed(93)
    N, d, B, r, vocab = 2_000_000, 64, 300, 256, 300
    plan = nest.plan_offline(N, d, "bf16", B, r)
    assert plan["path"] == 4 and not plan["single_pass"]
    stride = plan["sample_stride"]
    K = 3.0 + torch.randn(N, d, generator=g)
    near = torch.arange(0, 400 * stride, stride)
    K[near] = 0.5 * torch.randn(len(near), d, generator=g)
    K = K.to(torch.bfloat16)
    q = (0.1 * torch.randn(B, d, generator=g)).to(torch.bfloat16)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g), dim=1)
    rows = sorted(set(list(range(0, B, 23)) + [B - 1]))
    out, _, _ = run_and_check(nest, K, V, q, p_lm, r, 1 / 8, 0.7, vocab, "bf16", check_rows=rows)
    # every neighbour is one of the near keys
    near_set = set(near.tolist())
    for b in rows:
        assert set(out["idx"][b].cpu().numpy().tolist()) <= near_set


@pytest.mark.parametrize("N,d,B,r", [
    (200000, 128, 2048, 64),   # 8 query groups over 19 key ranges, two passes
    (70017, 64, 4000, 33),     # 16 groups (the last one partial), one pass
])
def test_many_query_groups(nest, N, d, B, r):
    """Batches far above 256 queries: many groups of 256 stream each key
    range (adjacent CTAs share its tiles in L2), and every group's lists,
    counters and thresholds stay separate.  Rows sampled across all groups."""
    K, V, q, p_lm = _random_case(N, d, B, 600, "bf16", seed=B + r, centres=40)
    rows = sorted(set(list(range(0, B, B // 12)) + [255, 256, B - 1]))
    run_and_check(nest, K, V, q, p_lm, r, 1 / np.sqrt(d), 0.7, 600, "bf16", check_rows=rows)


def test_large_batch_shape_sampled_rows(nest):
    """Large-batch shape: bf16 d=4096, B=512, r=256, clustered keys (N reduced
    to 524,288); the oracle checks 12 query rows spread over the batch."""
    w = synth.WORKLOADS["large_batch"]
    x = synth.make_inputs(w, device="cuda", N=1 << 19)
    rows = list(range(0, 512, 43))
    run_and_check(nest, x.K, x.V, x.q, x.p_lm, w.r, w.mu, w.lam, w.vocab, w.dtype,
                  check_rows=rows)


# ---------------------------------------------------------------- full-size, sampled rows

def _chunks(K, rows=65536):
    for lo in range(0, K.shape[0], rows):
        yield lo, synth.to_numpy_raw(K[lo:min(K.shape[0], lo + rows)])


def _oracle_rows_parallel(K, q_np, r, workers=16):
    """The oracle's top-r of each row of q_np over all keys of the device tensor K:
    distances chunk by chunk (the oracle's sqdist, OpenMP inside), then each
    row's top-r (the oracle's topr) in a thread pool; the C calls release the
    interpreter lock, so the per-row sorts run side by side."""
    from concurrent.futures import ThreadPoolExecutor
    B = q_np.shape[0]
    D = np.empty((B, K.shape[0]), dtype=np.float64)
    for lo, piece in _chunks(K):
        D[:, lo:lo + piece.shape[0]] = oracle.sqdist(piece, q_np)
    allidx = np.arange(K.shape[0], dtype=np.int64)
    s = np.empty((B, r), dtype=np.float64)
    idx = np.empty((B, r), dtype=np.int64)

    def one(b):
        Db, Ib, _ = oracle.topr(D[b], allidx, r)
        s[b], idx[b] = -Db, Ib
    with ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(one, range(B)))
    return s, idx


def _check_rows_against(out, K, V, q_rows_np, rows, p_lm, w, s_or, i_or, label):
    """Rows ``rows`` of a step's output against the oracle's (s_or, i_or) for
    the same query vectors (row j of s_or belongs to output row rows[j])."""
    s_all, i_all = out["s"].cpu().numpy(), out["idx"].cpu().numpy()
    V_np = V.cpu().numpy()
    p_m = out["p_m"].cpu().numpy()
    for j, b in enumerate(rows):
        i_g = i_all[b]
        # exact distances of the union of both lists, from the rows themselves
        union = np.unique(np.concatenate([i_g, i_or[j]]))
        K_rows = synth.to_numpy_raw(K[torch.as_tensor(union, device=K.device)])
        where = {int(k): n for n, k in enumerate(union)}
        g_loc = np.array([where[int(k)] for k in i_g])[None]
        o_loc = np.array([where[int(k)] for k in i_or[j]])[None]
        matched = check_search(s_all[b:b + 1], g_loc, s_or[j:j + 1], o_loc, K_rows,
                               q_rows_np[j:j + 1], w.dtype, np.array([K.shape[0]]), label=label)
        p_lm_b = p_lm[b:b + 1].cpu().numpy()
        check_mix(p_m[b:b + 1], s_all[b:b + 1], i_all[b:b + 1], V_np, p_lm_b, w.mu, w.lam,
                  w.vocab)
        if matched:
            P, n = oracle.pknn(s_or[j:j + 1], i_or[j:j + 1], V_np, w.mu, w.vocab)
            ref = oracle.mix(p_lm_b, P, w.lam, n)
            check_mix_end_to_end(p_m[b:b + 1], ref, [0])


def _spread_rows(B, n, first=()):
    """n distinct rows of a batch of B: the given first rows, then evenly spread."""
    rows = list(first)
    for v in np.linspace(0, B - 1, n).round().astype(int).tolist():
        if len(rows) >= n:
            break
        if v not in rows:
            rows.append(v)
    k = 0
    while len(rows) < n:
        if k not in rows:
            rows.append(k)
        k += 1
    return sorted(rows)


def test_large_batch_full_size_sampled_rows(nest):
    """bf16 d=4096, N=4,194,304, B=512, r=256 (the benchmarked large-batch launch):
    the oracle checks 32 query rows spread over both query groups, over all keys."""
    w = synth.WORKLOADS["large_batch"]
    x = synth.make_inputs(w, device="cuda")
    ds = nest.Datastore(x.K, x.V, w.vocab)
    out = ds.step(x.q, w.r, x.p_lm, w.mu, w.lam)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    rows = _spread_rows(512, 32, first=(0, 255, 256, 511))
    q_np = synth.to_numpy_raw(x.q[rows])
    s_or, i_or = _oracle_rows_parallel(x.K, q_np, w.r)
    _check_rows_against(out, x.K, x.V, q_np, rows, x.p_lm, w, s_or, i_or,
                        "config 4: large batch, 4M keys, B=512, r=256")
    ds.close()


def test_hidden8192_full_size_B_sweep(nest):
    """bf16 d=8192, N=8,388,608 clustered keys (128 GiB), r=1024, B in {1, 8, 64, 256}:
    four kernel paths on one datastore, each checked against the oracle on the
    rows it shares with a fixed set of 48 rows (0-7, 24 more spread below 64
    and 16 spread to 255), so that B = 64 and B = 256 are checked on at least
    32 rows and B = 1 and 8 on all of theirs; the oracle scans all keys once
    for those rows."""
    w = synth.WORKLOADS["hidden8192"]
    x = synth.make_inputs(w, device="cuda", B=256)
    ds = nest.Datastore(x.K, x.V, w.vocab)
    rows = sorted(set(range(8)) | set(np.linspace(8, 63, 24).round().astype(int).tolist())
                  | set(np.linspace(64, 255, 16).round().astype(int).tolist()))
    assert len(rows) == 48 and sum(b < 64 for b in rows) == 32
    q_np = synth.to_numpy_raw(x.q[rows])
    s_or, i_or = _oracle_rows_parallel(x.K, q_np, w.r)
    for B in (1, 8, 64, 256):
        out = ds.step(x.q[:B].contiguous(), w.r, x.p_lm[:B].contiguous(), w.mu, w.lam)
        torch.cuda.synchronize()
        assert ds.device_status() == 0, f"B={B}"
        sel = [j for j, b in enumerate(rows) if b < B]
        _check_rows_against(out, x.K, x.V, q_np[sel], [rows[j] for j in sel], x.p_lm, w,
                            s_or[sel], i_or[sel],
                            f"config 5: 8M keys, d=8192, r=1024, B={B}")
    ds.close()
