"""Comparison of the CUDA path with the fp64 oracle.

Rules (the tolerances the kNN-LM step is held to):

* Neighbour sets: the GPU's top-r key set must equal the oracle's, except
  for keys whose oracle distance lies within ``tie_rel`` (1e-4) relative of
  the oracle's r-th distance: with near-equal distances either key is a
  correct r-th neighbour.  Integer-exact inputs are compared bit-exactly.
* Distances of the keys both sides returned:
  |D_gpu - D_exact| <= rel * D_exact, with rel = 1e-3 for bf16 keys and
  1e-5 for fp32 keys, and D_gpu = 0 exactly where D_exact = 0.  The GPU
  re-ranks its screened candidates by distances recomputed as sums of
  squared differences in fp32, whose error is relative to D itself (a few
  units in the last place), so no allowance in terms of the norms is made.
* Order: the GPU row is nearest first by its own distances, ties by the
  smaller key index, then padding (s = -inf, idx = -1); the number of real
  entries is min(r, number of candidate keys).
* p_M and p_kNN: fed the GPU's own neighbours, the oracle's Eq. 2 / Eq. 3
  must agree with the GPU within 1e-5 per entry and total variation < 1e-4;
  for rows whose neighbour sets match exactly the oracle's end-to-end p_M
  must agree to the same tolerance.

``STATS`` collects, per label, the largest relative distance error and the
largest relative gap between a swapped key's distance and the oracle's r-th
distance seen by ``check_search``; the test session prints them at the end.
"""
from __future__ import annotations

import numpy as np

import oracle

P_ABS_TOL = 1e-5
TV_TOL = 1e-4
TIE_REL = 1e-4

STATS: dict[str, dict] = {}


def _record(label, dist_rel, gap_rel, swaps):
    label = label or "edge, shape and sweep cases"
    st = STATS.setdefault(label, {"rows": 0, "max_dist_rel": 0.0, "max_gap_rel": 0.0,
                                  "swaps": 0})
    st["rows"] += 1
    st["max_dist_rel"] = max(st["max_dist_rel"], float(dist_rel))
    st["max_gap_rel"] = max(st["max_gap_rel"], float(gap_rel))
    st["swaps"] += int(swaps)


def dist_rel_tol(dtype: str) -> float:
    return 1e-3 if dtype == "bf16" else 1e-5


def _exact_sqdist_rows(K_np, q_np, b, keys):
    """Exact fp64 squared distances of query b to the given key indices."""
    keys = np.asarray(keys, dtype=np.int64)
    if keys.size == 0:
        return np.zeros(0)
    return oracle.sqdist(K_np[keys], q_np[b:b + 1])[0]


def check_search(s_gpu, idx_gpu, s_or, idx_or, K_np, q_np, dtype, cand_count,
                 exact=False, tie_rel=TIE_REL, label=None):
    """Assert the GPU search matches the oracle's under the rules above.

    Returns the list of rows whose index sets match the oracle exactly.
    """
    s_gpu = np.asarray(s_gpu, dtype=np.float64)
    idx_gpu = np.asarray(idx_gpu, dtype=np.int64)
    B, r = s_gpu.shape
    rel = dist_rel_tol(dtype)
    exact_rows = []
    for b in range(B):
        n_real = min(r, int(cand_count[b]))
        g_idx = idx_gpu[b, :n_real]
        g_D = -s_gpu[b, :n_real]
        assert np.all(idx_gpu[b, n_real:] == -1), f"row {b}: padding idx"
        assert np.all(np.isneginf(s_gpu[b, n_real:])), f"row {b}: padding s"
        assert np.all(g_idx >= 0), f"row {b}: missing neighbours"
        assert len(set(g_idx.tolist())) == n_real, f"row {b}: duplicate neighbours"
        # nearest first by the GPU's own distances, ties by smaller index
        order = np.lexsort((g_idx, g_D))
        assert np.array_equal(order, np.arange(n_real)), f"row {b}: GPU row not sorted"
        o_idx = idx_or[b, :n_real]
        o_D = -s_or[b, :n_real]
        if exact:
            np.testing.assert_array_equal(g_idx, o_idx, err_msg=f"row {b}: idx (exact inputs)")
            np.testing.assert_array_equal(g_D, o_D, err_msg=f"row {b}: D (exact inputs)")
            exact_rows.append(b)
            _record(label, 0.0, 0.0, 0)
            continue
        gs, os_ = set(g_idx.tolist()), set(o_idx.tolist())
        gap = 0.0
        extra = []
        if gs == os_:
            exact_rows.append(b)
        else:
            D_r = o_D[-1]
            extra = sorted(gs - os_)
            missing = sorted(os_ - gs)
            D_extra = _exact_sqdist_rows(K_np, q_np, b, extra)
            D_missing = _exact_sqdist_rows(K_np, q_np, b, missing)
            band = tie_rel * D_r
            gaps = np.abs(np.concatenate([D_extra, D_missing]) - D_r)
            gap = gaps.max() / D_r if D_r > 0 else (0.0 if gaps.max() == 0 else np.inf)
            assert np.all(np.abs(D_extra - D_r) <= band), \
                f"row {b}: GPU-only neighbours {extra[:5]} not at the r-th distance {D_r}"
            assert np.all(np.abs(D_missing - D_r) <= band), \
                f"row {b}: oracle-only neighbours {missing[:5]} not at the r-th distance {D_r}"
        # distances of every GPU neighbour against the exact value
        D_ex = _exact_sqdist_rows(K_np, q_np, b, g_idx)
        err = np.abs(g_D - D_ex)
        zero = D_ex == 0
        assert np.all(g_D[zero] == 0), f"row {b}: a key equal to the query has D != 0"
        dist_rel = (err[~zero] / D_ex[~zero]).max() if np.any(~zero) else 0.0
        assert dist_rel <= rel, f"row {b}: distance error {dist_rel:.3g} relative > {rel}"
        _record(label, dist_rel, gap, len(extra))
    return exact_rows


def check_mix(p_m_gpu, s_gpu, idx_gpu, V_np, p_lm_np, mu, lam, vocab, p_knn_gpu=None,
              lam_gpu=None):
    """Oracle Eq. 2 / Eq. 3 on the GPU's own neighbours vs the GPU's p_M (and p_kNN)."""
    s64 = np.asarray(s_gpu, dtype=np.float64)
    P, nreal = oracle.pknn(s64, idx_gpu, V_np, mu, vocab)
    lam_rows = lam if lam_gpu is None else np.asarray(lam_gpu, dtype=np.float64)
    M = oracle.mix(p_lm_np, P, lam_rows, nreal)
    p_m_gpu = np.asarray(p_m_gpu, dtype=np.float64)
    err = np.abs(p_m_gpu - M)
    assert err.max() <= P_ABS_TOL, f"p_M max error {err.max():.3g}"
    tv = 0.5 * err.sum(axis=1)
    assert tv.max() < TV_TOL, f"p_M total variation {tv.max():.3g}"
    if p_knn_gpu is not None:
        ek = np.abs(np.asarray(p_knn_gpu, dtype=np.float64) - P)
        assert ek.max() <= P_ABS_TOL, f"p_kNN max error {ek.max():.3g}"
        assert (0.5 * ek.sum(axis=1)).max() < TV_TOL
    return M


def check_mix_end_to_end(p_m_gpu, p_m_oracle, rows):
    """Full p_M comparison for the rows whose neighbour sets match the oracle's."""
    if not rows:
        return
    a = np.asarray(p_m_gpu, dtype=np.float64)[rows]
    b = np.asarray(p_m_oracle, dtype=np.float64)[rows]
    err = np.abs(a - b)
    assert err.max() <= P_ABS_TOL, f"end-to-end p_M max error {err.max():.3g}"
    assert (0.5 * err.sum(axis=1)).max() < TV_TOL
