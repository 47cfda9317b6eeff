"""Pins for the fp64 oracle, on CPU, against things other than the oracle itself.

Each test fixes part of the oracle to mathematics it cannot share a bug with:
an independent library routine (scipy's cdist, torch's bf16 decoding), exact
integer arithmetic, brute-force Python sorting, closed forms of Eq. 2 - Eq. 4,
a hand-worked example (tests/golden/hand_2d.json) and invariants the paper's
definitions imply.  A dropped term, a wrong sign, a swapped index or a
transposed operand in the oracle fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.spatial.distance import cdist

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16_bits(x: torch.Tensor) -> np.ndarray:
    return x.to(torch.bfloat16).contiguous().view(torch.int16).numpy().view(np.uint16)


def _closed(expr: str) -> float:
    return float(eval(expr, {"__builtins__": {}}, {"exp": math.exp, "sqrt": math.sqrt}))


# ---------------------------------------------------------------- distances

def test_sqdist_matches_scipy_f32():
    rng = np.random.default_rng(1)
    K = rng.standard_normal((257, 37)).astype(np.float32)
    q = rng.standard_normal((3, 37)).astype(np.float32)
    D = oracle.sqdist(K, q)
    ref = cdist(q.astype(np.float64), K.astype(np.float64), "sqeuclidean")
    assert D.shape == (3, 257)
    np.testing.assert_allclose(D, ref, rtol=1e-12, atol=1e-12)


def test_sqdist_bf16_decoding_matches_torch():
    g = torch.Generator().manual_seed(2)
    K = torch.randn(129, 72, generator=g) * 3
    q = torch.randn(5, 72, generator=g) * 3
    D = oracle.sqdist(_bf16_bits(K), _bf16_bits(q))
    Kd = K.to(torch.bfloat16).double().numpy()
    qd = q.to(torch.bfloat16).double().numpy()
    np.testing.assert_allclose(D, cdist(qd, Kd, "sqeuclidean"), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sqdist_integer_lattice_exact(dtype):
    rng = np.random.default_rng(3)
    Ki = rng.integers(-8, 9, size=(64, 24))
    qi = rng.integers(-8, 9, size=(4, 24))
    if dtype == "f32":
        K, q = Ki.astype(np.float32), qi.astype(np.float32)
    else:
        K, q = _bf16_bits(torch.tensor(Ki, dtype=torch.float32)), _bf16_bits(
            torch.tensor(qi, dtype=torch.float32))
    D = oracle.sqdist(K, q)
    for b in range(4):
        for i in range(64):
            exact = sum(int(qi[b, j] - Ki[i, j]) ** 2 for j in range(24))
            assert D[b, i] == exact


def test_sqdist_key_equal_to_query_is_zero_and_first():
    rng = np.random.default_rng(4)
    K = rng.standard_normal((50, 16)).astype(np.float32)
    q = K[[17, 3]].copy()
    s, idx = oracle.knn_search(K, q, 4)
    assert s[0, 0] == 0.0 and idx[0, 0] == 17
    assert s[1, 0] == 0.0 and idx[1, 0] == 3
    assert np.all(s[:, 1:] < 0)


def test_sqdist_operands_not_transposed():
    # B != n and non-symmetric data: D[b, i] must pair query b with key i.
    K = np.array([[0, 0], [10, 0], [0, 3]], dtype=np.float32)
    q = np.array([[10, 0], [0, 1]], dtype=np.float32)
    D = oracle.sqdist(K, q)
    assert D.tolist() == [[100, 0, 109], [1, 101, 4]]


# ---------------------------------------------------------------- top-r

def _brute_topr(D_row, r):
    pairs = sorted((float(D_row[i]), i) for i in range(len(D_row)))
    return pairs[:r]


@pytest.mark.parametrize("r", [1, 5, 17, 64, 200])
def test_topr_brute_force_with_ties(r):
    rng = np.random.default_rng(5)
    # small integer lattice: many exactly equal distances, so ties matter
    K = rng.integers(-2, 3, size=(150, 3)).astype(np.float32)
    q = rng.integers(-2, 3, size=(4, 3)).astype(np.float32)
    s, idx = oracle.knn_search(K, q, r)
    D = cdist(q.astype(np.float64), K.astype(np.float64), "sqeuclidean")
    for b in range(4):
        want = _brute_topr(D[b], r)
        n = len(want)
        assert idx[b, :n].tolist() == [i for _, i in want]
        assert (-s[b, :n]).tolist() == [dd for dd, _ in want]
        assert np.all(idx[b, n:] == -1) and np.all(np.isneginf(s[b, n:]))


def test_chunked_search_matches_brute_force_in_any_chunk_order():
    """knn_search_chunked (keys delivered in pieces, as the full-size d=8192
    parity test streams them back from the device) against a brute-force
    sort: uneven chunks in shuffled order, integer keys with many ties."""
    rng = np.random.default_rng(21)
    K = rng.integers(-2, 3, size=(257, 5)).astype(np.float32)
    q = rng.integers(-2, 3, size=(3, 5)).astype(np.float32)
    cuts = [0, 1, 64, 65, 200, 257]
    chunks = [(cuts[i], K[cuts[i]:cuts[i + 1]]) for i in range(len(cuts) - 1)]
    order = rng.permutation(len(chunks))
    r = 40
    s, idx = oracle.knn_search_chunked([chunks[i] for i in order], q, r)
    D = cdist(q.astype(np.float64), K.astype(np.float64), "sqeuclidean")
    for b in range(3):
        want = _brute_topr(D[b], r)
        assert idx[b].tolist() == [i for _, i in want]
        assert (-s[b]).tolist() == [dd for dd, _ in want]


def test_topr_r_equals_n_returns_every_key_sorted():
    rng = np.random.default_rng(6)
    K = rng.standard_normal((40, 8)).astype(np.float32)
    q = rng.standard_normal((2, 8)).astype(np.float32)
    s, idx = oracle.knn_search(K, q, 40)
    for b in range(2):
        assert sorted(idx[b].tolist()) == list(range(40))
        assert np.all(np.diff(s[b]) <= 0)


def test_search_permutation_invariance():
    rng = np.random.default_rng(7)
    n, d, B, r, V = 300, 12, 3, 20, 50
    K = rng.standard_normal((n, d)).astype(np.float32)
    vals = rng.integers(0, V, n).astype(np.int32)
    q = rng.standard_normal((B, d)).astype(np.float32)
    p_lm = rng.dirichlet(np.ones(V), B).astype(np.float32)
    perm = rng.permutation(n)
    a = oracle.knn_step(K, vals, q, r, p_lm, 0.3, 0.6, V)
    b = oracle.knn_step(K[perm], vals[perm], q, r, p_lm, 0.3, 0.6, V)
    np.testing.assert_array_equal(a["s"], b["s"])
    np.testing.assert_array_equal(a["idx"], perm[b["idx"]])
    np.testing.assert_allclose(a["p_m"], b["p_m"], rtol=0, atol=1e-15)


def test_ragged_search_matches_per_segment_brute_force():
    rng = np.random.default_rng(8)
    K = rng.standard_normal((100, 6)).astype(np.float32)
    q = rng.standard_normal((4, 6)).astype(np.float32)
    off = np.array([0, 30, 30, 37, 100], dtype=np.int64)  # one empty, one shorter than r
    r = 10
    s, idx = oracle.knn_search(K, q, r, seg_off=off)
    for b in range(4):
        lo, hi = off[b], off[b + 1]
        D = cdist(q[b:b + 1].astype(np.float64), K[lo:hi].astype(np.float64), "sqeuclidean")[0]
        want = _brute_topr(D, r)
        n = len(want)
        assert idx[b, :n].tolist() == [lo + i for _, i in want]
        np.testing.assert_array_equal(-s[b, :n], [dd for dd, _ in want])
        assert np.all(idx[b, n:] == -1)
    assert np.all(idx[1] == -1)


# ---------------------------------------------------------------- Eq. 2

def _rand_neighbours(rng, r, N):
    s = -np.sort(rng.uniform(0, 40, r))[::-1].copy()
    s = np.sort(s)[::-1].copy()
    idx = rng.choice(N, r, replace=False).astype(np.int64)
    return s, idx


def test_pknn_sums_to_one_and_zero_outside_neighbour_values():
    rng = np.random.default_rng(9)
    N, V, r = 500, 40, 64
    vals = rng.integers(0, V, N).astype(np.int32)
    s, idx = _rand_neighbours(rng, r, N)
    P, nreal = oracle.pknn(s, idx, vals, 1 / 8, V)
    assert nreal[0] == r
    assert abs(P[0].sum() - 1) < 1e-14
    outside = np.setdiff1d(np.arange(V), vals[idx])
    assert np.all(P[0, outside] == 0)
    assert np.all(P[0, np.unique(vals[idx])] > 0)


def test_pknn_single_neighbour_is_one_hot():
    vals = np.array([3, 7, 1], dtype=np.int32)
    P, _ = oracle.pknn(np.array([-12.5]), np.array([1]), vals, 0.25, 10)
    assert P[0, 7] == 1.0 and P[0].sum() == 1.0


def test_pknn_all_values_equal_is_one_hot():
    rng = np.random.default_rng(10)
    vals = np.full(100, 4, dtype=np.int32)
    s, idx = _rand_neighbours(rng, 30, 100)
    P, _ = oracle.pknn(s, idx, vals, 0.5, 8)
    assert abs(P[0, 4] - 1) < 1e-15 and P[0].sum() == P[0, 4]


def test_pknn_mu_zero_is_value_histogram():
    rng = np.random.default_rng(11)
    N, V, r = 200, 9, 50
    vals = rng.integers(0, V, N).astype(np.int32)
    s, idx = _rand_neighbours(rng, r, N)
    P, _ = oracle.pknn(s, idx, vals, 0.0, V)
    hist = np.bincount(vals[idx], minlength=V) / r
    np.testing.assert_allclose(P[0], hist, rtol=0, atol=1e-15)


@pytest.mark.parametrize("s1,s2,mu", [(-3.0, -5.0, 0.125), (-100000.0, -100001.0, 1.0),
                                      (-7.0, -7.0, 2.0), (-0.5, -40.0, 1 / 64)])
def test_pknn_two_neighbours_is_logistic(s1, s2, mu):
    # p(v1) = e^{mu s1} / (e^{mu s1} + e^{mu s2}) = 1 / (1 + e^{-mu (s1 - s2)});
    # the second case also shows no underflow at large |s|.
    vals = np.array([0, 1], dtype=np.int32)
    P, _ = oracle.pknn(np.array([s1, s2]), np.array([0, 1]), vals, mu, 2)
    want = 1 / (1 + math.exp(-mu * (s1 - s2)))
    assert abs(P[0, 0] - want) < 1e-15 and abs(P[0, 1] - (1 - want)) < 1e-15


def test_pknn_ignores_padding_and_order():
    rng = np.random.default_rng(12)
    vals = rng.integers(0, 20, 100).astype(np.int32)
    s, idx = _rand_neighbours(rng, 10, 100)
    P1, n1 = oracle.pknn(s, idx, vals, 0.2, 20)
    order = rng.permutation(10)
    s2 = np.concatenate([s[order], [-np.inf] * 3])
    i2 = np.concatenate([idx[order], [-1] * 3])
    P2, n2 = oracle.pknn(s2, i2, vals, 0.2, 20)
    assert n1[0] == 10 and n2[0] == 10
    np.testing.assert_allclose(P1, P2, rtol=0, atol=1e-16)


# ---------------------------------------------------------------- Eq. 3

def _mix_case(seed=13, V=30):
    rng = np.random.default_rng(seed)
    p_lm = rng.dirichlet(np.ones(V)).astype(np.float32)[None]
    vals = rng.integers(0, V, 80).astype(np.int32)
    s, idx = _rand_neighbours(rng, 12, 80)
    P, nreal = oracle.pknn(s, idx, vals, 0.3, V)
    return p_lm, P, nreal


def test_mix_lambda_one_is_p_lm_and_zero_is_p_knn():
    p_lm, P, nreal = _mix_case()
    np.testing.assert_array_equal(oracle.mix(p_lm, P, 1.0, nreal), p_lm.astype(np.float64))
    np.testing.assert_array_equal(oracle.mix(p_lm, P, 0.0, nreal), P)


def test_mix_is_linear_in_lambda_and_sums_to_one():
    p_lm, P, nreal = _mix_case()
    m0, m1 = oracle.mix(p_lm, P, 0.0, nreal), oracle.mix(p_lm, P, 1.0, nreal)
    for lam in (0.25, 0.7, 0.9):
        m = oracle.mix(p_lm, P, lam, nreal)
        np.testing.assert_allclose(m, lam * m1 + (1 - lam) * m0, rtol=0, atol=1e-16)
        assert abs(m.sum() - (lam * p_lm.astype(np.float64).sum() + (1 - lam))) < 1e-14


def test_mix_with_no_neighbours_returns_p_lm():
    p_lm, _, _ = _mix_case()
    P, nreal = oracle.pknn(np.full(4, -np.inf), np.full(4, -1), np.zeros(3, np.int32), 0.1, 30)
    assert nreal[0] == 0 and not P.any()
    np.testing.assert_array_equal(oracle.mix(p_lm, P, 0.3, nreal), p_lm.astype(np.float64))


# ---------------------------------------------------------------- Eq. 4

@pytest.mark.parametrize("alpha,tau", [(0.3, 0.1), (0.2, 0.1), (0.5, 1.0)])
def test_rrc_closed_form(alpha, tau):
    s = np.array([-2.0, -3.0, -8.0])
    lam = oracle.rrc(s, np.array([0, 1, 2]), alpha, tau)[0]
    assert abs(lam - 1 / (1 + math.exp(-(2.0 / 8.0 - alpha) / tau))) < 1e-15


def test_rrc_uses_absolute_values_and_skips_padding():
    s = np.array([-4.0, -16.0, -np.inf])
    lam = oracle.rrc(s, np.array([5, 6, -1]), 0.3, 0.1)[0]
    assert abs(lam - 1 / (1 + math.exp(-(0.25 - 0.3) / 0.1))) < 1e-15


# ---------------------------------------------------------------- hand-worked example

def test_golden_hand_worked_2d_example():
    with open(os.path.join(GOLDEN, "hand_2d.json")) as f:
        g = json.load(f)
    K = np.array(g["K"], dtype=np.float32)
    q = np.array(g["q"], dtype=np.float32)
    vals = np.array(g["values"], dtype=np.int32)
    mu = _closed(g["mu"])
    p_lm = np.array([g["p_lm"]], dtype=np.float32)
    out = oracle.knn_step(K, vals, q, g["r"], p_lm, mu, g["lambda"], g["vocab"])
    assert out["idx"][0].tolist() == g["expect_idx"]
    assert (-out["s"][0]).tolist() == g["expect_sqdist"]
    s_all, i_all = oracle.knn_search(K, q, len(K))
    assert i_all[0].tolist() == g["expect_order_all"]
    assert (-s_all[0]).tolist() == g["expect_sqdist_all"]
    np.testing.assert_allclose(out["p_knn"][0], [_closed(e) for e in g["expect_p_knn"]],
                               rtol=0, atol=1e-15)
    np.testing.assert_allclose(out["p_m"][0], [_closed(e) for e in g["expect_p_m"]],
                               rtol=0, atol=1e-15)
    lam_t = oracle.rrc(out["s"], out["idx"], g["rrc_alpha"], g["rrc_tau"])[0]
    assert abs(lam_t - _closed(g["expect_rrc"])) < 1e-15


# ---------------------------------------------------------------- inputs

def test_tiny_workload_inputs_are_seeded_and_shaped():
    w = synth.WORKLOADS["tiny"]
    a = synth.make_inputs(w)
    b = synth.make_inputs(w)
    assert a.K.shape == (4096, 64) and a.K.dtype == torch.float32
    assert a.q.shape == (8, 64) and a.V.dtype == torch.int32
    assert torch.equal(a.K, b.K) and torch.equal(a.V, b.V) and torch.equal(a.p_lm, b.p_lm)
    assert int(a.V.min()) >= 0 and int(a.V.max()) < w.vocab
    assert torch.allclose(a.p_lm.double().sum(1), torch.ones(8, dtype=torch.float64), atol=1e-5)
    # Zipf(1.1): token 0 is the most frequent value
    counts = torch.bincount(a.V.long(), minlength=w.vocab)
    assert int(counts.argmax()) == 0


# ---------------------------------------------------------------- Eq. 5 / Eq. 6

def _brute_decide(p_m, s, idx, values, lam, delta):
    token = int(np.argmax(p_m))  # numpy: first maximum = smaller token id
    cands = sorted((-float(s[i]), int(idx[i])) for i in range(len(idx))
                   if idx[i] >= 0 and values[idx[i]] == token)
    key = cands[0][1] if cands else -1
    return token, float(p_m[token]), key, int(lam <= delta and key >= 0)


def test_decide_matches_brute_force_with_ties():
    rng = np.random.default_rng(30)
    N, V, r = 300, 12, 40
    values = rng.integers(0, V, N).astype(np.int32)
    for trial in range(40):
        p_m = rng.dirichlet(np.ones(V))
        if trial % 3 == 0:  # planted tie on the maximum
            j, k = rng.choice(V, 2, replace=False)
            p_m[j] = p_m[k] = p_m.max() + 0.01
        s = -np.round(rng.uniform(0, 5, r), 1)  # rounded: ties in s
        idx = rng.choice(N, r, replace=False).astype(np.int64)
        idx[rng.random(r) < 0.1] = -1
        lam = float(rng.uniform())
        got = oracle.decide(p_m, s, idx, values, lam, 0.5)
        want = _brute_decide(p_m, s, idx, values, lam, 0.5)
        assert (int(got[0][0]), float(got[1][0]), int(got[2][0]), int(got[3][0])) == want


def test_decide_without_matching_neighbour_emits_the_token():
    values = np.array([1, 1, 2], dtype=np.int32)
    p_m = np.array([0.7, 0.2, 0.1])
    tok, pmax, key, use = oracle.decide(p_m, np.array([-1.0, -2.0]), np.array([0, 2]), values,
                                        0.1, 0.5)
    assert tok[0] == 0 and pmax[0] == 0.7 and key[0] == -1 and use[0] == 0


@pytest.mark.parametrize("lam,delta,want", [(0.2, 0.5, 1), (0.5, 0.5, 1), (0.51, 0.5, 0)])
def test_decide_span_rule_of_eq6(lam, delta, want):
    values = np.array([3, 0, 3], dtype=np.int32)
    p_m = np.array([0.1, 0.1, 0.1, 0.7])
    _, _, key, use = oracle.decide(p_m, np.array([-4.0, -1.0, -3.0]), np.array([0, 1, 2]),
                                   values, lam, delta)
    assert key[0] == 2 and use[0] == want  # nearest neighbour with token 3 is key 2


# ---------------------------------------------------------------- Eq. 7

def _frac(e):
    return float(eval(e, {"__builtins__": {}}, {}))


def test_verify_hand_worked_example():
    with open(os.path.join(GOLDEN, "verify_hand.json")) as f:
        g = json.load(f)
    ratio, acc, n_acc = oracle.verify(np.array(g["p_m"]), np.array(g["draft"]),
                                      np.array(g["span_off"]), g["gamma"])
    np.testing.assert_allclose(ratio, [_frac(e) for e in g["expect_ratio"]], rtol=1e-15)
    assert acc.tolist() == g["expect_accept"]
    assert n_acc.tolist() == g["expect_n_accept"]


def test_verify_closed_forms():
    rng = np.random.default_rng(31)
    V = 50
    p = rng.dirichlet(np.ones(V), 6)
    draft = p.argmax(1).astype(np.int32)  # drafting the argmax: ratio = 1/gamma
    ratio, acc, n = oracle.verify(p, draft, np.array([0, 6]), 0.05)
    np.testing.assert_allclose(ratio, 20.0, rtol=1e-14)
    assert acc.all() and n[0] == 6
    # a token with zero probability is always rejected and cuts the span there
    p2 = p.copy()
    p2[3, draft[3]] = 0.0
    _, acc2, n2 = oracle.verify(p2, draft, np.array([0, 6]), 0.05)
    assert acc2[3] == 0 and n2[0] == 3
    # gamma = 1: accept iff the draft has more than half the top probability
    q = np.array([[0.4, 0.3, 0.3], [0.4, 0.21, 0.39], [0.4, 0.2, 0.4]])
    _, acc3, _ = oracle.verify(q, np.array([1, 1, 1]), np.array([0, 3]), 1.0)
    assert acc3.tolist() == [1, 1, 0]


# ---------------------------------------------------------------- masked keys

def test_search_with_excluded_keys_is_search_of_the_rest():
    rng = np.random.default_rng(32)
    K = rng.standard_normal((400, 10)).astype(np.float32)
    q = rng.standard_normal((3, 10)).astype(np.float32)
    excl = rng.random(400) < 0.3
    s, I = oracle.knn_search(K, q, 25, exclude=excl)
    keep = np.flatnonzero(~excl)
    D = cdist(q.astype(np.float64), K[keep].astype(np.float64), "sqeuclidean")
    for b in range(3):
        want = sorted((float(D[b, j]), int(keep[j])) for j in range(len(keep)))[:25]
        assert I[b].tolist() == [i for _, i in want]
        np.testing.assert_array_equal(-s[b], [dd for dd, _ in want])
    # ragged: the exclusion applies inside segments too
    off = np.array([0, 150, 150, 400])
    s2, I2 = oracle.knn_search(K, q, 10, seg_off=off, exclude=excl)
    assert not np.isin(I2[I2 >= 0], np.flatnonzero(excl)).any()
    assert (I2[1] == -1).all()
