"""fp64 CPU oracle for the kNN-LM step of NEST (arXiv 2405.19325).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import this package; the product path never
does.  It shares no code with the CUDA library.  The arithmetic lives in
``nest_oracle.c`` (plain C, double precision); this module compiles it with
gcc on first use and marshals numpy arrays into it.

Inputs are numpy arrays holding the exact stored values: ``float32`` arrays
for fp32 data, ``uint16`` arrays holding raw bf16 bit patterns for bf16 data.

Functions and the passages they restate:

* ``sqdist``   -- ||q - k||^2; the similarity is s = -||q - k||^2 (Sec. 2.2, App. A)
* ``topr``     -- the r nearest neighbours pi, ties to the smaller key index
                  (Sec. 2.2; search step of Algorithm 1)
* ``knn_search`` -- sqdist + topr over all keys or over per-query candidate
                  segments (second-stage search over K', Sec. 3.1)
* ``pknn``     -- Eq. 2
* ``mix``      -- Eq. 3
* ``rrc``      -- Eq. 4
* ``decide``   -- greedy token and span start (Eq. 5), span decision (Eq. 6)
* ``verify``   -- relaxed speculative decoding of drafted spans (Eq. 7)

``knn_search`` also takes ``exclude`` (a boolean per key): excluded keys are
left out of the candidate set, as accepted spans are masked out of the
datastore for the rest of a generation (Sec. 3.4).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

F32 = 0
BF16 = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "nest_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libnest_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into ``oracle/libnest_oracle.so`` (gcc, OpenMP)."""
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC",
                        "-shared", "-std=c11", _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        # NEST_ORACLE_LIB points the tests at a deliberately broken copy of the
        # oracle (tests/test_oracle_mutants.py) to show the pins catch it.
        path = os.environ.get("NEST_ORACLE_LIB") or build()
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        lib.nest_oracle_sqdist.argtypes = [P, ctypes.c_int, ctypes.c_int64, ctypes.c_int32,
                                           P, ctypes.c_int32, P, ctypes.c_int]
        lib.nest_oracle_sqdist.restype = ctypes.c_int
        lib.nest_oracle_topr.argtypes = [P, P, ctypes.c_int64, ctypes.c_int32, P, P]
        lib.nest_oracle_topr.restype = ctypes.c_int64
        lib.nest_oracle_pknn.argtypes = [P, P, P, ctypes.c_int64, ctypes.c_int32,
                                         ctypes.c_double, ctypes.c_int32, P]
        lib.nest_oracle_pknn.restype = ctypes.c_int32
        lib.nest_oracle_mix.argtypes = [P, P, ctypes.c_int32, ctypes.c_double,
                                        ctypes.c_int32, P]
        lib.nest_oracle_mix.restype = ctypes.c_int
        lib.nest_oracle_rrc.argtypes = [P, P, ctypes.c_int32, ctypes.c_double, ctypes.c_double]
        lib.nest_oracle_rrc.restype = ctypes.c_double
        lib.nest_oracle_decide.argtypes = [P, ctypes.c_int32, P, P, P, ctypes.c_int64,
                                           ctypes.c_int32, ctypes.c_double, ctypes.c_double,
                                           P, P, P, P]
        lib.nest_oracle_decide.restype = ctypes.c_int
        lib.nest_oracle_verify.argtypes = [P, ctypes.c_int32, P, ctypes.c_int32, P, ctypes.c_int32,
                                           ctypes.c_double, P, P, P]
        lib.nest_oracle_verify.restype = ctypes.c_int
        _lib = lib
    return _lib


def default_threads() -> int:
    return max(1, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity")
               else (os.cpu_count() or 1))


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _vec_dtype(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle inputs must be float32 or uint16 (bf16 bits), got {a.dtype}")


def sqdist(K: np.ndarray, q: np.ndarray, nthreads: int | None = None) -> np.ndarray:
    """D[b, i] = sum_j (q[b, j] - K[i, j])^2 in fp64 (distance behind s, Sec. 2.2)."""
    K = np.ascontiguousarray(K)
    q = np.ascontiguousarray(q)
    dt = _vec_dtype(K)
    if _vec_dtype(q) != dt:
        raise TypeError("K and q must have the same element type")
    if K.ndim != 2 or q.ndim != 2 or K.shape[1] != q.shape[1]:
        raise ValueError("K must be n x d and q must be B x d")
    n, d = K.shape
    B = q.shape[0]
    D = np.empty((B, n), dtype=np.float64)
    rc = _load().nest_oracle_sqdist(_ptr(K), dt, n, d, _ptr(q), B, _ptr(D),
                                    nthreads or default_threads())
    if rc != 0:
        raise ValueError("nest_oracle_sqdist rejected its arguments")
    return D


def topr(D: np.ndarray, idx: np.ndarray, r: int) -> tuple[np.ndarray, np.ndarray, int]:
    """r nearest of one query: (D_sorted[r], idx[r], n_real); pads D=+inf, idx=-1."""
    D = np.ascontiguousarray(D, dtype=np.float64)
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    if D.shape != idx.shape or D.ndim != 1:
        raise ValueError("D and idx must be equal-length vectors")
    Dout = np.empty(r, dtype=np.float64)
    Iout = np.empty(r, dtype=np.int64)
    keep = _load().nest_oracle_topr(_ptr(D), _ptr(idx), D.shape[0], r, _ptr(Dout), _ptr(Iout))
    if keep < 0:
        raise ValueError("nest_oracle_topr rejected its arguments")
    return Dout, Iout, int(keep)


def knn_search(K: np.ndarray, q: np.ndarray, r: int, seg_off: np.ndarray | None = None,
               nthreads: int | None = None,
               exclude: np.ndarray | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Top-r search of every query.

    Returns (s, idx), each B x r: s = -||q - k||^2 in fp64, nearest first
    (ties to the smaller key index), padded with s = -inf, idx = -1.  With
    ``seg_off`` (B + 1 offsets) query b searches only keys
    [seg_off[b], seg_off[b+1]) and idx stays a global key index.  Keys with
    ``exclude[i]`` true are not candidates.
    """
    B = q.shape[0]
    s = np.empty((B, r), dtype=np.float64)
    I = np.empty((B, r), dtype=np.int64)
    keep_all = None if exclude is None else ~np.asarray(exclude, dtype=bool)
    if seg_off is None:
        D = sqdist(K, q, nthreads)
        allidx = np.arange(K.shape[0], dtype=np.int64)
        for b in range(B):
            Db, Ib = D[b], allidx
            if keep_all is not None:
                Db, Ib = Db[keep_all], Ib[keep_all]
            Db, Ib, _ = topr(Db, Ib, r)
            s[b], I[b] = -Db, Ib
    else:
        seg_off = np.asarray(seg_off, dtype=np.int64)
        for b in range(B):
            lo, hi = int(seg_off[b]), int(seg_off[b + 1])
            D = sqdist(K[lo:hi], q[b:b + 1], nthreads)[0]
            Ib = np.arange(lo, hi, dtype=np.int64)
            if keep_all is not None:
                D, Ib = D[keep_all[lo:hi]], Ib[keep_all[lo:hi]]
            Db, Ib, _ = topr(D, Ib, r)
            s[b], I[b] = -Db, Ib
    return s, I


def knn_search_chunked(chunks, q: np.ndarray, r: int,
                       nthreads: int | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Full-scan top-r search over keys delivered in pieces.

    ``chunks`` yields (start, K_piece) in any order covering every key once;
    distances of all pieces are kept (fp64, B x N) and the top-r taken over
    all of them, exactly as ``knn_search`` does over one array.
    """
    parts_D, parts_I = [], []
    for start, piece in chunks:
        parts_D.append(sqdist(piece, q, nthreads))
        parts_I.append(np.arange(start, start + piece.shape[0], dtype=np.int64))
    D = np.concatenate(parts_D, axis=1)
    allidx = np.concatenate(parts_I)
    B = q.shape[0]
    s = np.empty((B, r), dtype=np.float64)
    I = np.empty((B, r), dtype=np.int64)
    for b in range(B):
        Db, Ib, _ = topr(D[b], allidx, r)
        s[b], I[b] = -Db, Ib
    return s, I


def pknn(s: np.ndarray, idx: np.ndarray, values: np.ndarray, mu: float,
         vocab: int) -> tuple[np.ndarray, np.ndarray]:
    """Eq. 2 for each query row: (p_knn B x vocab fp64, n_real B)."""
    s = np.ascontiguousarray(np.atleast_2d(s), dtype=np.float64)
    idx = np.ascontiguousarray(np.atleast_2d(idx), dtype=np.int64)
    values = np.ascontiguousarray(values, dtype=np.int32)
    B, r = s.shape
    P = np.empty((B, vocab), dtype=np.float64)
    nreal = np.empty(B, dtype=np.int32)
    lib = _load()
    for b in range(B):
        n = lib.nest_oracle_pknn(_ptr(s[b]), _ptr(idx[b]), _ptr(values), values.shape[0],
                                 r, float(mu), vocab, _ptr(P[b]))
        if n < 0:
            raise ValueError("nest_oracle_pknn rejected its arguments")
        nreal[b] = n
    return P, nreal


def mix(p_lm: np.ndarray, p_knn: np.ndarray, lam, n_real: np.ndarray) -> np.ndarray:
    """Eq. 3 for each query row; ``lam`` is a scalar or one lambda per row."""
    p_lm = np.ascontiguousarray(np.atleast_2d(p_lm), dtype=np.float32)
    p_knn = np.ascontiguousarray(np.atleast_2d(p_knn), dtype=np.float64)
    B, V = p_lm.shape
    lams = np.broadcast_to(np.asarray(lam, dtype=np.float64), (B,))
    out = np.empty((B, V), dtype=np.float64)
    lib = _load()
    for b in range(B):
        if lib.nest_oracle_mix(_ptr(p_lm[b]), _ptr(p_knn[b]), V, float(lams[b]),
                               int(n_real[b]), _ptr(out[b])) != 0:
            raise ValueError("nest_oracle_mix rejected its arguments")
    return out


def rrc(s: np.ndarray, idx: np.ndarray, alpha: float, tau: float) -> np.ndarray:
    """Eq. 4 for each query row."""
    s = np.ascontiguousarray(np.atleast_2d(s), dtype=np.float64)
    idx = np.ascontiguousarray(np.atleast_2d(idx), dtype=np.int64)
    lib = _load()
    return np.array([lib.nest_oracle_rrc(_ptr(s[b]), _ptr(idx[b]), s.shape[1],
                                         float(alpha), float(tau))
                     for b in range(s.shape[0])], dtype=np.float64)


def decide(p_m: np.ndarray, s: np.ndarray, idx: np.ndarray, values: np.ndarray, lam,
           delta: float):
    """Eq. 5 / Eq. 6 per row: (token, p_max, span_key, use_span)."""
    p_m = np.ascontiguousarray(np.atleast_2d(p_m), dtype=np.float64)
    s = np.ascontiguousarray(np.atleast_2d(s), dtype=np.float64)
    idx = np.ascontiguousarray(np.atleast_2d(idx), dtype=np.int64)
    values = np.ascontiguousarray(values, dtype=np.int32)
    B, V = p_m.shape
    lams = np.broadcast_to(np.asarray(lam, dtype=np.float64), (B,))
    tok = np.empty(B, np.int32)
    pmax = np.empty(B, np.float64)
    key = np.empty(B, np.int64)
    use = np.empty(B, np.int32)
    lib = _load()
    for b in range(B):
        t, pm = ctypes.c_int32(), ctypes.c_double()
        k, u = ctypes.c_int64(), ctypes.c_int32()
        if lib.nest_oracle_decide(_ptr(p_m[b]), V, _ptr(s[b]), _ptr(idx[b]), _ptr(values),
                                  values.shape[0], s.shape[1], float(lams[b]), float(delta),
                                  ctypes.byref(t), ctypes.byref(pm), ctypes.byref(k),
                                  ctypes.byref(u)) != 0:
            raise ValueError("nest_oracle_decide rejected its arguments")
        tok[b], pmax[b], key[b], use[b] = t.value, pm.value, k.value, u.value
    return tok, pmax, key, use


def verify(p_m: np.ndarray, draft: np.ndarray, span_off: np.ndarray, gamma: float):
    """Eq. 7 over drafted spans: (ratio[rows], accept[rows], n_accept[spans])."""
    p_m = np.ascontiguousarray(np.atleast_2d(p_m), dtype=np.float64)
    draft = np.ascontiguousarray(draft, dtype=np.int32)
    span_off = np.ascontiguousarray(span_off, dtype=np.int32)
    rows, V = p_m.shape
    spans = span_off.shape[0] - 1
    ratio = np.empty(rows, np.float64)
    acc = np.empty(rows, np.int32)
    n_acc = np.empty(max(spans, 0), np.int32)
    if _load().nest_oracle_verify(_ptr(p_m), V, _ptr(draft), rows, _ptr(span_off), spans,
                                  float(gamma), _ptr(ratio), _ptr(acc), _ptr(n_acc)) != 0:
        raise ValueError("nest_oracle_verify rejected its arguments")
    return ratio, acc, n_acc


def knn_step(K, values, q, r, p_lm, mu, lam, vocab, seg_off=None, nthreads=None):
    """Search then Eq. 2 then Eq. 3; returns dict(s, idx, p_knn, p_m, n_real)."""
    s, I = knn_search(K, q, r, seg_off, nthreads)
    P, nreal = pknn(s, I, values, mu, vocab)
    return dict(s=s, idx=I, p_knn=P, p_m=mix(p_lm, P, lam, nreal), n_real=nreal)
