"""ctypes binding of the C ABI in include/nest.h (argument marshalling only).

Every step of the kNN-LM path runs in the CUDA kernels of ``libnest.so``;
this module only checks tensor properties, passes device pointers and the
current torch stream, and raises on a non-zero status.  There is no CPU
fallback: if the library is missing or no GPU is present, calls raise.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libnest.so")

F32 = 0
BF16 = 1

STATUS = {
    0: "NEST_OK", 1: "NEST_ERR_INVALID_ARG", 2: "NEST_ERR_DTYPE", 3: "NEST_ERR_ALIGN",
    4: "NEST_ERR_OOM", 5: "NEST_ERR_CUDA", 6: "NEST_ERR_VALUE_RANGE", 7: "NEST_ERR_OVERFLOW",
    8: "NEST_ERR_TIMEOUT", 9: "NEST_ERR_UNSUPPORTED", 10: "NEST_ERR_MARGIN",
}
STATUS_CODE = {v: k for k, v in STATUS.items()}

# Every entry point of include/nest.h: (name, restype, argtypes).
_P = ctypes.c_void_p
_I32, _I64, _F = ctypes.c_int32, ctypes.c_int64, ctypes.c_float
SIGNATURES = {
    "nest_datastore_create": (ctypes.c_int, [_P, _P, _I64, _I32, ctypes.c_int, _I32, _P,
                                             ctypes.POINTER(_P)]),
    "nest_datastore_destroy": (ctypes.c_int, [_P]),
    "nest_datastore_reserve": (ctypes.c_int, [_P, _I32, _I32, _I32]),
    "nest_datastore_use_cta_pairs": (ctypes.c_int, [_P, _I32]),
    "nest_selftest_bounded_wait": (ctypes.c_int, [_P, ctypes.POINTER(_I64), _P]),
    "nest_plan_offline": (ctypes.c_int, [_I64, _I32, _I32, _I32, _I32, _I32, _I32, _I64, _I32,
                                         _P]),
    "nest_knn_search": (ctypes.c_int, [_P, _P, _I32, _I32, _P, _P, _P, _P]),
    "nest_knn_search_static": (ctypes.c_int, [_P, _P, _I32, _I32, _P, _P, _P, _P]),
    "nest_knn_search_masked": (ctypes.c_int, [_P, _P, _I32, _I32, _P, _P, _P, _P, _P]),
    "nest_mask_keys": (ctypes.c_int, [_P, _P, _I64, _I64, _P]),
    "nest_knn_decide": (ctypes.c_int, [_P, _P, _P, _P, _P, _I32, _I32, _F, _P, _P, _P, _P, _P]),
    "nest_verify_spans": (ctypes.c_int, [_P, _P, _P, _I32, _P, _I32, _F, _P, _P, _P, _P]),
    "nest_knn_mix": (ctypes.c_int, [_P, _P, _P, _P, _I32, _I32, _F, _F, _P, _P, _P]),
    "nest_knn_mix_rrc": (ctypes.c_int, [_P, _P, _P, _P, _I32, _I32, _F, _F, _F, _P, _P, _P, _P]),
    "nest_knn_step": (ctypes.c_int, [_P, _P, _I32, _I32, _P, _P, _F, _F, _P, _P, _P, _P, _P]),
    "nest_knn_step_host": (ctypes.c_int, [_P, _P, _I32, _I32, _P, _P, _F, _F, _P, _P, _P, _P]),
    "nest_device_status": (ctypes.c_int, [_P, _P]),
    "nest_timing_enable": (ctypes.c_int, [_P, _I32]),
    "nest_timing_read": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_double),
                                        ctypes.POINTER(_I64)]),
    "nest_launch_count": (_I64, [_P]),
    "nest_search_path": (_I32, [_P, _I32, _I32, _I32]),
    "nest_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "nest_version": (_I32, []),
}

_lib = None


class Plan(ctypes.Structure):
    """nest_plan_t (include/nest.h)."""
    _fields_ = [("path", ctypes.c_int32), ("queries_per_group", ctypes.c_int32),
                ("groups", ctypes.c_int32), ("parts", ctypes.c_int32),
                ("stages", ctypes.c_int32), ("single_pass", ctypes.c_int32),
                ("sample_stride", ctypes.c_int64), ("list_capacity", ctypes.c_int64),
                ("scratch_bytes", ctypes.c_int64)]


class NestError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        self.name = STATUS.get(code, f"status {code}")
        super().__init__(f"{where}: {self.name}")


def load_library(path: str | None = None):
    """Load libnest.so (raises if it has not been built)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build it with paper_2405_19325_gb300.build.build()")
    lib = ctypes.CDLL(p)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def _pair_mode(on: bool | None) -> int:
    """nest_datastore_use_cta_pairs mode: 1 (pairs), 0 (single CTAs), -1 (automatic)."""
    return -1 if on is None else int(bool(on))


def plan_offline(N: int, d: int, dtype: str, B: int, r: int, ragged: bool = False,
                 num_sms: int = 152, smem_per_block: int = 232448,
                 cta_pairs: bool | None = None) -> dict:
    """The plan a search of this shape would run (nest_plan_offline): host
    only, no GPU.  The defaults are a GB300's 152 SMs and 227 KiB of opt-in
    shared memory per block.  ``dtype`` is "f32" or "bf16".  ``cta_pairs``
    as in Datastore.use_cta_pairs (None: the handle's automatic default)."""
    lib = load_library()
    p = Plan()
    code = BF16 if dtype == "bf16" else F32 if dtype == "f32" else -1
    if code < 0:
        raise ValueError("dtype must be 'f32' or 'bf16'")
    _check(lib.nest_plan_offline(int(N), int(d), code, int(B), int(r), int(bool(ragged)),
                                 int(num_sms), int(smem_per_block), _pair_mode(cta_pairs),
                                 ctypes.byref(p)), "nest_plan_offline")
    out = {name: getattr(p, name) for name, _ in Plan._fields_}
    out["kernel"] = Datastore.SEARCH_PATHS[p.path]
    return out


def _check(code: int, where: str) -> None:
    if code != 0:
        raise NestError(code, where)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"keys/queries must be float32 or bfloat16, got {t.dtype}")


def _dev(t: torch.Tensor, name: str, dtype=None) -> int:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _host(t: torch.Tensor, name: str, dtype=None) -> int:
    if not isinstance(t, torch.Tensor) or t.is_cuda:
        raise TypeError(f"{name} must be a host tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


class Datastore:
    """A key-value datastore (K, V) registered with the CUDA library (Eq. 1)."""

    def __init__(self, K: torch.Tensor, V: torch.Tensor, vocab: int, stream=None):
        lib = load_library()
        if K.dim() != 2:
            raise ValueError("K must be N x d")
        self.N, self.d = K.shape
        self.dtype = K.dtype
        self.vocab = int(vocab)
        if V.shape != (self.N,):
            raise ValueError("V must hold one token id per key")
        kp = _dev(K, "K")
        vp = _dev(V, "V", torch.int32)
        self._K, self._V = K, V  # borrowed by the library: keep them alive
        h = ctypes.c_void_p()
        _check(lib.nest_datastore_create(kp, vp, self.N, self.d, _dtype_code(K), self.vocab,
                                         _stream(stream), ctypes.byref(h)),
               "nest_datastore_create")
        self._h = h
        self._lib = lib

    @property
    def handle(self) -> int:
        return self._h.value

    def close(self) -> None:
        if getattr(self, "_h", None) is not None and self._h.value:
            self._lib.nest_datastore_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reserve(self, max_B: int, max_r: int, ragged: bool = False) -> None:
        _check(self._lib.nest_datastore_reserve(self._h, max_B, max_r, int(ragged)),
               "nest_datastore_reserve")

    def use_cta_pairs(self, on: bool | None) -> None:
        """Batches of more than 128 queries on CTA pairs (True), on single
        CTAs with two key tiles per stage (False), or automatically (None,
        the default): pairs when the batch is one group (up to 512)."""
        _check(self._lib.nest_datastore_use_cta_pairs(self._h, _pair_mode(on)),
               "nest_datastore_use_cta_pairs")

    # ------------------------------------------------------------ search / mix / step
    def search(self, q: torch.Tensor, r: int, seg_off: torch.Tensor | None = None,
               s_out: torch.Tensor | None = None, idx_out: torch.Tensor | None = None,
               stream=None):
        """r nearest neighbours of each query: (s [B, r] fp32, idx [B, r] int64)."""
        B = q.shape[0]
        if q.dtype != self.dtype or q.dim() != 2 or q.shape[1] != self.d:
            raise ValueError("q must be B x d with the datastore's dtype")
        s_out = torch.empty(B, r, dtype=torch.float32, device=q.device) if s_out is None else s_out
        idx_out = torch.empty(B, r, dtype=torch.int64, device=q.device) if idx_out is None else idx_out
        sp = _dev(seg_off, "seg_off", torch.int64) if seg_off is not None else None
        _check(self._lib.nest_knn_search(self._h, _dev(q, "q"), B, r, sp,
                                         _dev(s_out, "s_out", torch.float32),
                                         _dev(idx_out, "idx_out", torch.int64), _stream(stream)),
               "nest_knn_search")
        return s_out, idx_out

    def new_key_mask(self) -> torch.Tensor:
        """All-clear key mask (one bit per key, int32 words) on the current device."""
        return torch.zeros((self.N + 31) // 32, dtype=torch.int32, device="cuda")

    def mask_keys(self, key_mask: torch.Tensor, first_key: int, count: int, stream=None) -> None:
        """Mark keys [first_key, first_key + count) as used (Sec. 3.4 masking)."""
        _check(self._lib.nest_mask_keys(self._h, _dev(key_mask, "key_mask", torch.int32),
                                        int(first_key), int(count), _stream(stream)),
               "nest_mask_keys")

    def search_masked(self, q: torch.Tensor, r: int, key_mask: torch.Tensor,
                      seg_off: torch.Tensor | None = None, stream=None):
        """search() over the keys whose bit in key_mask is clear."""
        B = q.shape[0]
        if q.dtype != self.dtype or q.dim() != 2 or q.shape[1] != self.d:
            raise ValueError("q must be B x d with the datastore's dtype")
        if key_mask.numel() < (self.N + 31) // 32:
            raise ValueError("key_mask needs one bit per key")
        s_out = torch.empty(B, r, dtype=torch.float32, device=q.device)
        idx_out = torch.empty(B, r, dtype=torch.int64, device=q.device)
        sp = _dev(seg_off, "seg_off", torch.int64) if seg_off is not None else None
        _check(self._lib.nest_knn_search_masked(self._h, _dev(q, "q"), B, r, sp,
                                                _dev(key_mask, "key_mask", torch.int32),
                                                s_out.data_ptr(), idx_out.data_ptr(),
                                                _stream(stream)),
               "nest_knn_search_masked")
        return s_out, idx_out

    def decide(self, p_m: torch.Tensor, s: torch.Tensor, idx: torch.Tensor, lam: torch.Tensor,
               delta: float, stream=None) -> dict:
        """Eq. 5 / Eq. 6: greedy token, its probability, span start key, span choice."""
        B, r = s.shape
        self._check_rows(p_m, B)
        dev = p_m.device
        o = {"token": torch.empty(B, dtype=torch.int32, device=dev),
             "p_max": torch.empty(B, dtype=torch.float32, device=dev),
             "span_key": torch.empty(B, dtype=torch.int64, device=dev),
             "use_span": torch.empty(B, dtype=torch.int32, device=dev)}
        _check(self._lib.nest_knn_decide(self._h, _dev(p_m, "p_m", torch.float32),
                                         _dev(s, "s", torch.float32), _dev(idx, "idx", torch.int64),
                                         _dev(lam, "lambda", torch.float32), B, r, float(delta),
                                         o["token"].data_ptr(), o["p_max"].data_ptr(),
                                         o["span_key"].data_ptr(), o["use_span"].data_ptr(),
                                         _stream(stream)),
               "nest_knn_decide")
        return o

    def verify(self, p_m: torch.Tensor, draft: torch.Tensor, span_off: torch.Tensor, gamma: float,
               stream=None) -> dict:
        """Eq. 7 over drafted spans: per-row ratio and acceptance, accepted prefix per span."""
        rows = p_m.shape[0]
        spans = span_off.numel() - 1
        dev = p_m.device
        o = {"ratio": torch.empty(rows, dtype=torch.float32, device=dev),
             "accept": torch.empty(rows, dtype=torch.int32, device=dev),
             "n_accept": torch.empty(spans, dtype=torch.int32, device=dev)}
        _check(self._lib.nest_verify_spans(self._h, _dev(p_m, "p_m", torch.float32),
                                           _dev(draft, "draft", torch.int32), rows,
                                           _dev(span_off, "span_off", torch.int32), spans,
                                           float(gamma), o["ratio"].data_ptr(),
                                           o["accept"].data_ptr(), o["n_accept"].data_ptr(),
                                           _stream(stream)),
               "nest_verify_spans")
        return o

    def mix(self, s: torch.Tensor, idx: torch.Tensor, p_lm: torch.Tensor, mu: float, lam: float,
            want_p_knn: bool = False, p_m_out=None, p_knn_out=None, stream=None):
        """Eq. 2 + Eq. 3: p_M (and p_kNN when asked)."""
        B, r = s.shape
        p_m_out = torch.empty_like(p_lm) if p_m_out is None else p_m_out
        if want_p_knn and p_knn_out is None:
            p_knn_out = torch.empty_like(p_lm)
        self._check_rows(p_lm, B)
        _check(self._lib.nest_knn_mix(self._h, _dev(s, "s", torch.float32),
                                      _dev(idx, "idx", torch.int64),
                                      _dev(p_lm, "p_lm", torch.float32), B, r, float(mu), float(lam),
                                      _dev(p_knn_out, "p_knn_out", torch.float32)
                                      if p_knn_out is not None else None,
                                      _dev(p_m_out, "p_m_out", torch.float32), _stream(stream)),
               "nest_knn_mix")
        return (p_m_out, p_knn_out) if want_p_knn else p_m_out

    def mix_rrc(self, s: torch.Tensor, idx: torch.Tensor, p_lm: torch.Tensor, mu: float,
                alpha: float, tau: float, want_p_knn: bool = False, stream=None):
        """Eq. 2 + Eq. 4: (p_M, lambda_t[B]) (+ p_kNN when asked)."""
        B, r = s.shape
        self._check_rows(p_lm, B)
        p_m = torch.empty_like(p_lm)
        lam = torch.empty(B, dtype=torch.float32, device=p_lm.device)
        p_knn = torch.empty_like(p_lm) if want_p_knn else None
        _check(self._lib.nest_knn_mix_rrc(self._h, _dev(s, "s", torch.float32),
                                          _dev(idx, "idx", torch.int64),
                                          _dev(p_lm, "p_lm", torch.float32), B, r, float(mu),
                                          float(alpha), float(tau), lam.data_ptr(),
                                          p_knn.data_ptr() if p_knn is not None else None,
                                          p_m.data_ptr(), _stream(stream)),
               "nest_knn_mix_rrc")
        return (p_m, lam, p_knn) if want_p_knn else (p_m, lam)

    def step(self, q: torch.Tensor, r: int, p_lm: torch.Tensor, mu: float, lam: float,
             seg_off: torch.Tensor | None = None, want_p_knn: bool = False, out: dict | None = None,
             stream=None) -> dict:
        """One kNN-LM step (search + Eq. 2 + Eq. 3) in one C call."""
        B = q.shape[0]
        if q.dtype != self.dtype or q.dim() != 2 or q.shape[1] != self.d:
            raise ValueError("q must be B x d with the datastore's dtype")
        self._check_rows(p_lm, B)
        o = out if out is not None else {}
        dev = q.device
        if "s" not in o:
            o["s"] = torch.empty(B, r, dtype=torch.float32, device=dev)
            o["idx"] = torch.empty(B, r, dtype=torch.int64, device=dev)
            o["p_m"] = torch.empty(B, self.vocab, dtype=torch.float32, device=dev)
            if want_p_knn:
                o["p_knn"] = torch.empty(B, self.vocab, dtype=torch.float32, device=dev)
        pk = o.get("p_knn")
        sp = _dev(seg_off, "seg_off", torch.int64) if seg_off is not None else None
        _check(self._lib.nest_knn_step(self._h, _dev(q, "q"), B, r, sp,
                                       _dev(p_lm, "p_lm", torch.float32), float(mu), float(lam),
                                       _dev(o["s"], "s_out", torch.float32),
                                       _dev(o["idx"], "idx_out", torch.int64),
                                       _dev(pk, "p_knn_out", torch.float32) if pk is not None else None,
                                       _dev(o["p_m"], "p_m_out", torch.float32), _stream(stream)),
               "nest_knn_step")
        return o

    def step_host(self, q_host: torch.Tensor, r: int, p_lm_host: torch.Tensor, mu: float,
                  lam: float, seg_off_host: torch.Tensor | None = None, staging: dict | None = None,
                  stream=None) -> dict:
        """One step from host inputs to host outputs in one C call (nest_knn_step_host).

        The library copies the query batch, p_LM and the segment offsets to
        device buffers of its own, runs the step on ``stream`` and copies p_M,
        s and idx back before returning.  Page-locked host tensors let the
        copies run asynchronously.  ``staging`` caches the page-locked output
        tensors between calls (they are overwritten by the next call).
        """
        B = q_host.shape[0]
        if q_host.dtype != self.dtype or q_host.dim() != 2 or q_host.shape[1] != self.d:
            raise ValueError("q must be B x d with the datastore's dtype")
        if p_lm_host.dim() != 2 or p_lm_host.shape[0] != B or p_lm_host.shape[1] != self.vocab:
            raise ValueError(f"p_lm must be {B} x {self.vocab}")
        st = staging if staging is not None else {}
        if st.get("shape") != (B, r):
            st["shape"] = (B, r)
            st["p_m"] = torch.empty(B, self.vocab, dtype=torch.float32).pin_memory()
            st["s"] = torch.empty(B, r, dtype=torch.float32).pin_memory()
            st["idx"] = torch.empty(B, r, dtype=torch.int64).pin_memory()
        sp = _host(seg_off_host, "seg_off", torch.int64) if seg_off_host is not None else None
        _check(self._lib.nest_knn_step_host(self._h, _host(q_host, "q"), B, r, sp,
                                            _host(p_lm_host, "p_lm", torch.float32), float(mu),
                                            float(lam), st["s"].data_ptr(), st["idx"].data_ptr(),
                                            st["p_m"].data_ptr(), _stream(stream)),
               "nest_knn_step_host")
        return {"p_m": st["p_m"], "s": st["s"], "idx": st["idx"]}

    # ------------------------------------------------------------ status / timing
    def selftest_bounded_wait(self, stream=None) -> int:
        """Runs a kernel whose bounded wait runs out (nothing arrives); the
        device status then holds NEST_ERR_TIMEOUT.  Returns the nanoseconds
        the kernel waited."""
        ns = ctypes.c_int64()
        _check(self._lib.nest_selftest_bounded_wait(self._h, ctypes.byref(ns), _stream(stream)),
               "nest_selftest_bounded_wait")
        return ns.value
    def device_status(self, stream=None) -> int:
        """Synchronize and return (and clear) the device status code."""
        return int(self._lib.nest_device_status(self._h, _stream(stream)))

    def check(self, stream=None) -> None:
        _check(self.device_status(stream), "device status")

    def timing_enable(self, on: bool = True) -> None:
        _check(self._lib.nest_timing_enable(self._h, int(on)), "nest_timing_enable")

    def timing_read(self) -> tuple[float, int]:
        ms = ctypes.c_double()
        n = ctypes.c_int64()
        _check(self._lib.nest_timing_read(self._h, ctypes.byref(ms), ctypes.byref(n)),
               "nest_timing_read")
        return ms.value, n.value

    def launch_count(self) -> int:
        return int(self._lib.nest_launch_count(self._h))

    SEARCH_PATHS = {0: "scan_topr_kernel", 1: "tc_scan_kernel", 2: "tc_wide_kernel",
                    3: "tc_wide2_kernel", 4: "tc_wide_pair_kernel", 5: "scan_rows_kernel"}

    def search_path(self, B: int, r: int, ragged: bool = False) -> str:
        """Name of the distance-scan kernel a search of this shape runs."""
        code = int(self._lib.nest_search_path(self._h, B, r, int(ragged)))
        if code < 0:
            raise NestError(-code, "nest_search_path")
        return self.SEARCH_PATHS[code]

    def _check_rows(self, p_lm: torch.Tensor, B: int) -> None:
        if p_lm.dim() != 2 or p_lm.shape[0] != B or p_lm.shape[1] != self.vocab:
            raise ValueError(f"p_lm must be {B} x {self.vocab}")
