"""Seeded random sweep of search shapes against the fp64 oracle.

The hand-picked cases elsewhere pin each edge on purpose; this sweep draws
shapes at random to reach combinations nobody picked: any element type, row
width, batch, r, datastore size, key layout, ragged segments and key masks,
with the search path following from the shape.  The cases are drawn once
from a fixed seed, so every run sees the same shapes and a failure names
its case.  Each case is held to the same rules as the other parity tests
(neighbour sets up to ties at the r-th distance, distances within the fp32
bound, Eq. 2 / Eq. 3 on the GPU's own neighbours); integer layouts must
match bit for bit.

A second set draws every size from values next to the ones the kernels
branch on (tile and warp multiples, the 8,192-word copy stride of the
selection, the 65,536-key threshold sample, the query-group sizes, list
lengths around 1,024) and goes through each public entry point in turn:
the device step, the host-buffer step, search + Eq. 4 + the Eq. 5 / Eq. 6
decision, and the masked search.  In both sets, half of the bf16 shapes (by
seed) run groups of 256 queries on CTA pairs.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from parity import check_mix, check_mix_end_to_end, check_search

pytestmark = pytest.mark.gpu

N_CASES = 100
# keep the oracle's work per case bounded: checked rows x N x d
MAX_ORACLE_WORK = 2.0e9
BATCHES = [1, 2, 3, 4, 5, 8, 13, 16, 17, 33, 40, 64, 100, 200, 255, 256, 257, 300, 511, 512, 600]
RS = [1, 2, 7, 32, 64, 100, 255, 256, 257, 1000, 1024, 2048, 4096]
WIDTHS = [8, 16, 24, 40, 64, 72, 128, 136, 256, 520, 1024, 2048, 4096]
LAYOUTS = ["clustered", "sorted_clusters", "uniform", "integer"]


def _draw_cases():
    rng = np.random.default_rng(2405_19325)
    cases = []
    while len(cases) < N_CASES:
        dtype = "bf16" if rng.random() < 0.75 else "f32"
        esize = 2 if dtype == "bf16" else 4
        d = int(rng.choice([w for w in WIDTHS if w * esize <= 16384 and (w * esize) % 16 == 0]))
        B = int(rng.choice(BATCHES))
        r = int(rng.choice(RS))
        ragged = bool(rng.random() < 0.25)
        masked = bool(rng.random() < 0.3)
        layout = str(rng.choice(LAYOUTS))
        # log-uniform datastore size; three draws in ten above the threshold
        # sample (65,536 keys or more) so that batched searches take two passes
        lo, hi = (60000, 700000) if rng.random() < 0.3 else (1, 400000)
        N = int(np.exp(rng.uniform(np.log(lo), np.log(hi))))
        rows = min(B, 10)
        if rows * N * d > MAX_ORACLE_WORK or N * d > 2.5e8:
            continue
        cases.append(dict(dtype=dtype, d=d, B=B, r=r, N=N, ragged=ragged, masked=masked,
                          layout=layout, seed=int(rng.integers(1 << 30))))
    return cases


CASES = _draw_cases()

EDGE_N = [1, 2, 31, 33, 127, 128, 129, 255, 257, 1023, 1024, 1025, 1057, 8191, 8192, 8193,
          8269, 9215, 16447, 65535, 65536, 65537, 65599, 131071, 131073, 196705, 262145]
EDGE_B = [1, 2, 3, 4, 5, 15, 16, 17, 31, 33, 63, 64, 65, 127, 128, 129, 255, 256, 257, 383,
          384, 511, 512, 513]
EDGE_R = [1, 2, 31, 32, 33, 255, 256, 257, 511, 512, 513, 1023, 1024, 1025, 2047, 2048, 4095, 4096]
EDGE_D = {"bf16": [8, 56, 64, 72, 120, 128, 136, 1016, 4096, 8192],
          "f32": [4, 60, 64, 68, 1020, 4096]}
ENTRIES = ["step", "host", "rrc_decide", "masked"]
N_EDGE = 100


def _draw_edge_cases():
    rng = np.random.default_rng(7_2405)
    cases = []
    while len(cases) < N_EDGE:
        dtype = "bf16" if rng.random() < 0.75 else "f32"
        d = int(rng.choice(EDGE_D[dtype]))
        B = int(rng.choice(EDGE_B))
        r = int(rng.choice(EDGE_R))
        N = int(rng.choice(EDGE_N))
        entry = ENTRIES[len(cases) % len(ENTRIES)]
        ragged = entry != "rrc_decide" and bool(rng.random() < 0.2)
        layout = str(rng.choice(LAYOUTS))
        rows = B if ragged else min(B, 10)
        if rows * N * d > MAX_ORACLE_WORK or N * d > 2.5e8:
            continue
        cases.append(dict(dtype=dtype, d=d, B=B, r=r, N=N, ragged=ragged,
                          masked=entry == "masked", layout=layout, entry=entry,
                          seed=int(rng.integers(1 << 30))))
    return cases


EDGE_CASES = _draw_edge_cases()


def _pairs(c):
    """Half of the bf16 shapes (by seed) run groups of 256 queries on CTA pairs
    whatever the number of groups (True); the others keep the handle's
    automatic choice (None): pairs for one group, single CTAs for more."""
    return True if c["dtype"] == "bf16" and c["seed"] % 2 == 1 else None


def _case_id(c):
    entry = c.get("entry")
    return (f"{c['dtype']}-N{c['N']}-d{c['d']}-B{c['B']}-r{c['r']}-{c['layout']}"
            + ("-ragged" if c["ragged"] else "")
            + (f"-{entry}" if entry else ("-masked" if c["masked"] else ""))
            + ("-pairs" if _pairs(c) else ""))


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _inputs(c, vocab):
    """Keys, values, queries, p_LM, segment offsets and excluded keys of a case."""
    N, d, B = c["N"], c["d"], c["B"]
    g = torch.Generator().manual_seed(c["seed"])
    nc = int(torch.randint(2, 65, (1,), generator=g))
    if c["layout"] == "integer":
        # a few integer base vectors plus small integer offsets: fp32 distances exact,
        # many exact ties
        base = torch.randint(-2, 3, (nc, d), generator=g).float()
        K = base[torch.randint(0, nc, (N,), generator=g)] \
            + (torch.rand(N, d, generator=g) < 0.05).float()
        q = base[torch.randint(0, nc, (B,), generator=g)] \
            + torch.randint(-1, 2, (B, d), generator=g).float()
    else:
        cen = torch.randn(nc, d, generator=g)
        if c["layout"] == "uniform":
            K = torch.randn(N, d, generator=g)
        elif c["layout"] == "sorted_clusters":
            K = cen[torch.arange(N) * nc // max(N, 1)] + 0.3 * torch.randn(N, d, generator=g)
        else:
            K = cen[torch.randint(0, nc, (N,), generator=g)] + 0.3 * torch.randn(N, d, generator=g)
        q = cen[torch.randint(0, nc, (B,), generator=g)] + 0.3 * torch.randn(B, d, generator=g)
    dt = synth.torch_dtype(c["dtype"])
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g) * 2, dim=1)
    seg_off = None
    if c["ragged"]:
        cuts = torch.sort(torch.randint(0, N + 1, (B - 1,), generator=g)).values
        seg_off = torch.cat([torch.zeros(1, dtype=torch.int64), cuts.to(torch.int64),
                             torch.full((1,), N, dtype=torch.int64)])
        if B > 2:  # one empty segment in the middle
            seg_off[B // 2 + 1] = seg_off[B // 2]
            seg_off = torch.cummax(seg_off, 0).values
    excl = None
    if c["masked"]:
        excl = (torch.rand(N, generator=g) < 0.15).numpy()
        a = int(torch.randint(0, N, (1,), generator=g))
        excl[a:a + max(1, N // 7)] = True          # one used span of keys
    return K.to(dt), V, q.to(dt), p_lm, seg_off, excl


def _mask_words(excl):
    N = excl.size
    words = np.zeros((N + 31) // 32, dtype=np.uint32)
    k = np.flatnonzero(excl)
    np.bitwise_or.at(words, k >> 5, (np.uint32(1) << (k & 31).astype(np.uint32)))
    return torch.from_numpy(words.view(np.int32))


@pytest.mark.parametrize("c", CASES, ids=[_case_id(c) for c in CASES])
def test_random_shape(nest, c):
    _run_case(nest, c)


@pytest.mark.parametrize("c", EDGE_CASES, ids=[_case_id(c) for c in EDGE_CASES])
def test_boundary_shape(nest, c):
    _run_case(nest, c)


def _run_case(nest, c):
    vocab = 700
    N, d, B, r, dtype = c["N"], c["d"], c["B"], c["r"], c["dtype"]
    K, V, q, p_lm, seg_off, excl = _inputs(c, vocab)
    dev = torch.device("cuda")
    ds = nest.Datastore(K.to(dev), V.to(dev), vocab)
    if _pairs(c):
        ds.use_cta_pairs(True)
    qd = q.to(dev)
    so_d = seg_off.to(dev) if seg_off is not None else None
    mu, lam = 1 / np.sqrt(d), 0.75
    # full scans: a spread of rows; ragged: every row (each scans only its segment)
    rows = list(range(B)) if c["ragged"] else sorted(set(range(0, B, max(1, B // 9))) | {B - 1})
    K_np, V_np = synth.to_numpy_raw(K), V.numpy()
    q_np = synth.to_numpy_raw(q)[rows]
    p_lm_np = p_lm.numpy()[rows]
    so_np = seg_off.numpy() if seg_off is not None else None
    exact = c["layout"] == "integer"
    entry = c.get("entry", "masked" if excl is not None else "step")
    counts = (np.full(B, N) if so_np is None else so_np[1:] - so_np[:-1])[rows]
    if entry in ("step", "host"):
        if entry == "step":
            out = ds.step(qd, r, p_lm.to(dev), mu, lam, seg_off=so_d, want_p_knn=True)
            torch.cuda.synchronize()
            p_knn = out["p_knn"].cpu().numpy()[rows]
        else:
            out = ds.step_host(q.pin_memory(), r, p_lm.pin_memory(), mu, lam,
                               seg_off_host=seg_off)
            p_knn = None
        assert ds.device_status() == 0
        s_g, i_g = out["s"].cpu().numpy()[rows], out["idx"].cpu().numpy()[rows]
        ref = oracle.knn_step(K_np, V_np, q_np, r, p_lm_np, mu, lam, vocab, seg_off=so_np)
        matched = check_search(s_g, i_g, ref["s"], ref["idx"], K_np, q_np, dtype, counts,
                               exact=exact)
        p_m = out["p_m"].cpu().numpy()[rows]
        check_mix(p_m, s_g, i_g, V_np, p_lm_np, mu, lam, vocab, p_knn_gpu=p_knn)
        check_mix_end_to_end(p_m, ref["p_m"], matched)
    elif entry == "rrc_decide":
        alpha, tau, delta = 0.3, 0.1, 0.5
        s, idx = ds.search(qd, r, seg_off=so_d)
        p_m, lam_t = ds.mix_rrc(s, idx, p_lm.to(dev), mu, alpha, tau)
        o = ds.decide(p_m, s, idx, lam_t, delta)
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        s_g, i_g = s.cpu().numpy()[rows], idx.cpu().numpy()[rows]
        s_or, i_or = oracle.knn_search(K_np, q_np, r, seg_off=so_np)
        check_search(s_g, i_g, s_or, i_or, K_np, q_np, dtype, counts, exact=exact)
        lam_g = lam_t.cpu().numpy()[rows]
        np.testing.assert_allclose(lam_g, oracle.rrc(s_g.astype(np.float64), i_g, alpha, tau),
                                   rtol=0, atol=1e-6)
        p_m_g = p_m.cpu().numpy()[rows]
        check_mix(p_m_g, s_g, i_g, V_np, p_lm_np, mu, None, vocab, lam_gpu=lam_g)
        tok, pmax, key, use = oracle.decide(p_m_g.astype(np.float64), s_g, i_g, V_np,
                                            lam_g.astype(np.float64), delta)
        assert o["token"].cpu().numpy()[rows].tolist() == tok.tolist()
        np.testing.assert_array_equal(o["p_max"].cpu().numpy()[rows].astype(np.float64), pmax)
        assert o["span_key"].cpu().numpy()[rows].tolist() == key.tolist()
        assert o["use_span"].cpu().numpy()[rows].tolist() == use.tolist()
    else:
        mask = _mask_words(excl).to(dev)
        s, idx = ds.search_masked(qd, r, mask, seg_off=so_d)
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        i_all = idx.cpu().numpy()
        assert not excl[i_all[i_all >= 0]].any(), "a masked key was returned"
        s_or, i_or = oracle.knn_search(K_np, q_np, r, seg_off=so_np, exclude=excl)
        if so_np is None:
            counts = np.full(len(rows), N - int(excl.sum()))
        else:
            counts = np.array([int(so_np[b + 1] - so_np[b] - excl[so_np[b]:so_np[b + 1]].sum())
                               for b in range(B)])[rows]
        check_search(s.cpu().numpy()[rows], i_all[rows], s_or, i_or, K_np, q_np, dtype, counts,
                     exact=exact)
    ds.close()


def test_sweep_reaches_every_search_path(nest):
    """The drawn shapes run every distance-scan kernel the library has, and a
    handle on this device picks the kernel nest_plan_offline predicts from
    the device's SM count and shared memory per block."""
    seen = set()
    props = torch.cuda.get_device_properties(0)
    smem = getattr(props, "shared_memory_per_block_optin", None)
    V = torch.zeros(64, dtype=torch.int32, device="cuda")
    for c in CASES + EDGE_CASES:
        K = torch.zeros(64, c["d"], dtype=synth.torch_dtype(c["dtype"]), device="cuda")
        ds = nest.Datastore(K, V, 10)
        if _pairs(c):
            ds.use_cta_pairs(True)
        path = ds.search_path(c["B"], c["r"], ragged=c["ragged"])
        seen.add(path)
        ds.close()
        if smem:
            plan = nest.plan_offline(64, c["d"], c["dtype"], c["B"], c["r"], ragged=c["ragged"],
                                     num_sms=props.multi_processor_count, smem_per_block=smem,
                                     cta_pairs=_pairs(c))
            assert plan["kernel"] == path, (c, plan)
    assert seen >= {"tc_scan_kernel", "tc_wide_kernel", "tc_wide2_kernel",
                    "tc_wide_pair_kernel", "scan_topr_kernel", "scan_rows_kernel"}, seen


# ---------------------------------------------------------------- Eq. 7 verification and masking

VOCABS = [1, 2, 3, 7, 31, 1000, 4097, 32000, 50257, 128256]
P_KINDS = ["peaked", "flat", "one_hot", "tied_max", "with_zero_rows"]
GAMMAS = [1.0, 0.5, 0.1, 1e-3, 1e-6]


def _draw_verify_cases(n=40):
    rng = np.random.default_rng(7_7)
    cases = []
    while len(cases) < n:
        vocab = int(rng.choice(VOCABS))
        rows = int(np.exp(rng.uniform(0, np.log(3000))))
        if rows * vocab > 3e7:
            continue
        cases.append(dict(vocab=vocab, rows=rows, kind=str(rng.choice(P_KINDS)),
                          gamma=float(rng.choice(GAMMAS)), spans=int(rng.integers(1, 65)),
                          seed=int(rng.integers(1 << 30))))
    return cases


VERIFY_CASES = _draw_verify_cases()


def _verify_inputs(c):
    g = torch.Generator().manual_seed(c["seed"])
    rows, vocab = c["rows"], c["vocab"]
    kind = c["kind"]
    if kind == "flat":
        p = torch.softmax(torch.randn(rows, vocab, generator=g) * 0.1, dim=1)
    elif kind == "one_hot":
        p = torch.zeros(rows, vocab)
        p[torch.arange(rows), torch.randint(0, vocab, (rows,), generator=g)] = 1.0
    else:
        p = torch.softmax(torch.randn(rows, vocab, generator=g) * 8, dim=1)
    if kind == "tied_max" and vocab > 1:
        # the two largest entries of every row set equal
        top2 = torch.topk(p, 2, dim=1)
        p[torch.arange(rows), top2.indices[:, 1]] = top2.values[:, 0]
    if kind == "with_zero_rows":
        p[torch.rand(rows, generator=g) < 0.2] = 0.0
    top = p.argmax(1).to(torch.int32)
    other = torch.randint(0, vocab, (rows,), generator=g, dtype=torch.int32)
    if vocab > 1:
        second = torch.topk(p, 2, dim=1).indices[:, 1].to(torch.int32)
    else:
        second = top
    u = torch.rand(rows, generator=g)
    draft = torch.where(u < 0.6, top, torch.where(u < 0.8, second, other))
    cuts = torch.sort(torch.randint(0, rows + 1, (c["spans"] - 1,), generator=g)).values
    off = torch.cat([torch.zeros(1, dtype=torch.int32), cuts.to(torch.int32),
                     torch.full((1,), rows, dtype=torch.int32)])
    return p.contiguous(), draft, off


def _verify_id(c):
    return f"V{c['vocab']}-rows{c['rows']}-spans{c['spans']}-{c['kind']}-g{c['gamma']:g}"


@pytest.mark.parametrize("c", VERIFY_CASES, ids=[_verify_id(c) for c in VERIFY_CASES])
def test_verify_random(nest, c):
    """Eq. 7 on random spans (empty spans included) against the oracle: the
    ratio within fp32 rounding, the acceptance flags exactly except where
    min(1, ratio) lies within rounding of 1/2, and each span's accepted
    prefix following the GPU's own flags."""
    p, draft, off = _verify_inputs(c)
    dev = torch.device("cuda")
    K = torch.randn(64, 16, device=dev)
    ds = nest.Datastore(K, torch.zeros(64, dtype=torch.int32, device=dev), c["vocab"])
    o = ds.verify(p.to(dev), draft.to(dev), off.to(dev), c["gamma"])
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    ratio, acc, n_acc = oracle.verify(p.numpy().astype(np.float64), draft.numpy(), off.numpy(),
                                      c["gamma"])
    g_ratio = o["ratio"].cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(g_ratio, ratio, rtol=2e-6, atol=0)
    g_acc = o["accept"].cpu().numpy()
    near = np.abs(np.minimum(ratio, 1.0) - 0.5) <= 1e-6
    assert np.array_equal(g_acc[~near], acc[~near])
    g_n = o["n_accept"].cpu().numpy()
    so = off.numpy()
    for j in range(len(so) - 1):
        run = 0
        while so[j] + run < so[j + 1] and g_acc[so[j] + run]:
            run += 1
        assert g_n[j] == run, f"span {j}"
    if not near.any():
        assert g_n.tolist() == n_acc.tolist()
    ds.close()


def _draw_mask_cases(n=30):
    rng = np.random.default_rng(7_31)
    cases = []
    for _ in range(n):
        N = int(np.exp(rng.uniform(0, np.log(2_000_000))))
        spans = []
        for _ in range(int(rng.integers(1, 9))):
            kind = rng.integers(0, 4)
            if kind == 0:      # empty span
                first, count = int(rng.integers(0, N + 1)), 0
            elif kind == 1:    # ends at the last key
                count = int(rng.integers(1, N + 1))
                first = N - count
            elif kind == 2:    # starts on a word boundary
                first = int(rng.integers(0, N // 32 + 1)) * 32
                first = min(first, N - 1)
                count = int(rng.integers(1, min(N - first, 200) + 1))
            else:
                first = int(rng.integers(0, N))
                count = int(rng.integers(1, min(N - first, 5000) + 1))
            spans.append((first, count))
        cases.append(dict(N=N, spans=spans))
    return cases


MASK_CASES = _draw_mask_cases()


@pytest.mark.parametrize("c", MASK_CASES, ids=[f"N{c['N']}-{len(c['spans'])}spans" for c in MASK_CASES])
def test_mask_keys_random(nest, c):
    """Sec. 3.4 masking: the bits nest_mask_keys sets over random runs of
    keys (empty runs, runs ending at the last key, runs on and off word
    boundaries, overlapping runs) equal the union of the runs."""
    N = c["N"]
    dev = torch.device("cuda")
    K = torch.zeros(N, 4, device=dev)
    ds = nest.Datastore(K, torch.zeros(N, dtype=torch.int32, device=dev), 10)
    mask = ds.new_key_mask()
    want = np.zeros(N, bool)
    for first, count in c["spans"]:
        ds.mask_keys(mask, first, count)
        want[first:first + count] = True
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    words = mask.cpu().numpy().view(np.uint32)
    got = ((words[np.arange(N) >> 5] >> (np.arange(N) & 31)) & 1).astype(bool)
    assert np.array_equal(got, want)
    tail = N % 32
    if tail:
        assert words[-1] >> np.uint32(tail) == 0, "bits past the last key"
    ds.close()
