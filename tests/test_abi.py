"""The C ABI on a machine without a GPU: the library builds for sm_103a,
loads, exports every entry point include/nest.h declares, and rejects bad
arguments on the host before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "nest.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2405_19325_gb300 import build as nest_build
    from paper_2405_19325_gb300 import nest
    nest_build.build()
    return nest.load_library()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^NEST_API\s+[\w\s\*]+?\b(nest_\w+)\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for required in ["nest_datastore_create", "nest_knn_search", "nest_knn_mix", "nest_knn_step"]:
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2405_19325_gb300 import nest
    for name in declared_symbols():
        assert hasattr(lib, name), name
        assert name in nest.SIGNATURES, f"binding lacks {name}"


def test_status_strings(lib):
    from paper_2405_19325_gb300.nest import STATUS
    for code in STATUS:
        assert lib.nest_status_string(code)
    assert lib.nest_version() >= 100


FAKE = 0x10000  # a 16-byte aligned non-null address that is never dereferenced


def test_create_validation(lib):
    h = ctypes.c_void_p()
    P = ctypes.c_void_p
    assert lib.nest_datastore_create(None, P(FAKE), 10, 64, 0, 100, None, ctypes.byref(h)) == 1
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 64, 7, 100, None, ctypes.byref(h)) == 2
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 0, 64, 0, 100, None, ctypes.byref(h)) == 1
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 64, 0, 0, None, ctypes.byref(h)) == 1
    # fp32 row of 12 bytes, bf16 row of 14 bytes: not a multiple of 16
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 3, 0, 100, None, ctypes.byref(h)) == 3
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 7, 1, 100, None, ctypes.byref(h)) == 3
    # misaligned K
    assert lib.nest_datastore_create(P(FAKE + 4), P(FAKE), 10, 64, 0, 100, None,
                                     ctypes.byref(h)) == 3
    # row larger than 16 KiB
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 8200, 1, 100, None,
                                     ctypes.byref(h)) == 9
    assert lib.nest_datastore_create(P(FAKE), P(FAKE), 10, 64, 0, 100, None, None) == 1
    assert h.value is None


def test_search_and_mix_validation(lib):
    P = ctypes.c_void_p
    ds, q, s, i = P(FAKE), P(FAKE), P(FAKE), P(FAKE)
    assert lib.nest_knn_search(None, q, 1, 1, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, None, 1, 1, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, q, 0, 1, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, q, 1, 0, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, q, 1, 4097, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, q, 70000, 1, None, s, i, None) == 1
    assert lib.nest_knn_search(ds, P(FAKE + 8), 1, 1, None, s, i, None) == 3
    assert lib.nest_knn_search(ds, q, 1, 1, P(FAKE + 4), s, i, None) == 3
    assert lib.nest_knn_search(ds, q, 1, 1, None, s, P(FAKE + 4), None) == 3
    # the allocation-free search makes the same checks first, before its size check
    assert lib.nest_knn_search_static(None, q, 1, 1, None, s, i, None) == 1
    assert lib.nest_knn_search_static(ds, q, 65536, 1, None, s, i, None) == 1
    assert lib.nest_knn_search_static(ds, q, 1, 4097, None, s, i, None) == 1
    assert lib.nest_knn_search_static(ds, P(FAKE + 8), 1, 1, None, s, i, None) == 3
    assert lib.nest_knn_search_static(ds, q, 1, 1, P(FAKE + 4), s, i, None) == 3
    p = P(FAKE)
    assert lib.nest_knn_mix(ds, s, i, p, 1, 1, 1.0, 1.5, None, p, None) == 1
    assert lib.nest_knn_mix(ds, s, i, p, 1, 1, 1.0, -0.1, None, p, None) == 1
    assert lib.nest_knn_mix(ds, s, i, None, 1, 1, 1.0, 0.5, None, p, None) == 1
    assert lib.nest_knn_mix(ds, s, i, p, 1, 1, 1.0, float("nan"), None, p, None) == 1
    assert lib.nest_knn_mix_rrc(ds, s, i, p, 1, 1, 1.0, 0.3, 0.0, None, None, p, None) == 1
    assert lib.nest_knn_mix_rrc(ds, s, i, p, 1, 1, 1.0, 0.3, -1.0, None, None, p, None) == 1
    assert lib.nest_knn_step(ds, q, 1, 1, None, p, 1.0, 2.0, s, i, None, p, None) == 1
    h = P(FAKE)  # host-pointer entry point: checks run before any device work
    assert lib.nest_knn_step_host(None, h, 1, 1, None, h, 1.0, 0.5, h, h, h, None) == 1
    assert lib.nest_knn_step_host(ds, None, 1, 1, None, h, 1.0, 0.5, h, h, h, None) == 1
    assert lib.nest_knn_step_host(ds, h, 0, 1, None, h, 1.0, 0.5, h, h, h, None) == 1
    assert lib.nest_knn_step_host(ds, h, 1, 4097, None, h, 1.0, 0.5, h, h, h, None) == 1
    assert lib.nest_knn_step_host(ds, h, 1, 1, None, h, 1.0, 2.0, h, h, h, None) == 1
    assert lib.nest_knn_step_host(ds, h, 1, 1, None, h, 1.0, 0.5, h, h, None, None) == 1
    assert lib.nest_knn_step(ds, q, 1, 1, None, p, 1.0, 0.5, None, i, None, p, None) == 1


def test_nest_step_calls_validation(lib):
    """The decision, verification, masking and diagnostic calls refuse bad
    arguments on the host, before they touch the handle or the device."""
    P = ctypes.c_void_p
    ds, a = P(FAKE), P(FAKE)
    # masked search: the mask is required and 4-byte aligned
    assert lib.nest_knn_search_masked(None, a, 1, 1, None, None, a, a, None) == 1
    assert lib.nest_knn_search_masked(ds, a, 1, 1, None, None, a, a, None) == 1
    assert lib.nest_knn_search_masked(ds, a, 1, 1, None, P(FAKE + 2), a, a, None) == 3
    # masking: a negative start or count
    assert lib.nest_mask_keys(None, a, 0, 1, None) == 1
    assert lib.nest_mask_keys(ds, a, -1, 1, None) == 1
    assert lib.nest_mask_keys(ds, a, 0, -1, None) == 1
    # Eq. 5 / Eq. 6
    args = [a] * 4
    assert lib.nest_knn_decide(None, a, a, a, a, 1, 1, 0.5, *args, None) == 1
    assert lib.nest_knn_decide(ds, a, a, a, a, 0, 1, 0.5, *args, None) == 1
    assert lib.nest_knn_decide(ds, a, a, a, a, 1, 4097, 0.5, *args, None) == 1
    assert lib.nest_knn_decide(ds, a, a, a, a, 1, 1, float("nan"), *args, None) == 1
    assert lib.nest_knn_decide(ds, a, a, P(FAKE + 4), a, 1, 1, 0.5, *args, None) == 3
    # Eq. 7: rows, spans and gamma
    assert lib.nest_verify_spans(None, a, a, 1, a, 1, 0.5, a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, a, a, 0, a, 1, 0.5, a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, a, a, 1, a, 0, 0.5, a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, a, a, 70000, a, 1, 0.5, a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, a, a, 1, a, 1, 0.0, a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, a, a, 1, a, 1, float("nan"), a, a, a, None) == 1
    assert lib.nest_verify_spans(ds, P(FAKE + 2), a, 1, a, 1, 0.5, a, a, a, None) == 3
    # handle-level calls
    assert lib.nest_datastore_use_cta_pairs(None, 1) == 1
    # modes are 1, 0 and -1 (checked before the handle is read)
    assert lib.nest_datastore_use_cta_pairs(ds, 2) == 1
    assert lib.nest_datastore_use_cta_pairs(ds, -2) == 1
    assert lib.nest_selftest_bounded_wait(None, None, None) == 1
    assert lib.nest_datastore_reserve(None, 1, 1, 0) == 1
    assert lib.nest_search_path(None, 1, 1, 0) == -1
    assert lib.nest_datastore_destroy(None) == 0


def test_no_cpu_fallback_when_library_missing():
    from paper_2405_19325_gb300 import nest
    with pytest.raises(RuntimeError):
        nest.load_library("/nonexistent/libnest.so")
