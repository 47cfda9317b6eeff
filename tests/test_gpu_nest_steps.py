"""GPU parity of the NEST decisions that follow p_M, through the C ABI:
Eq. 4 interpolation (RRC), Eq. 5 / Eq. 6 greedy token, span start and span
choice, Eq. 7 relaxed speculative verification, and the masking of accepted
spans out of the datastore (Sec. 3.4).  Integer results (tokens, key
indices, decisions) must equal the oracle's run on the GPU's own fp32 p_M
and neighbours; where an fp32 ratio sits within rounding of the 1/2 cut,
either decision is accepted and the span counts must follow the flags."""
import numpy as np
import pytest
import torch

import oracle
import synth
from parity import check_mix, check_search

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _case(N, d, B, vocab, seed, dtype="bf16", centres=16):
    g = torch.Generator().manual_seed(seed)
    c = torch.randn(centres, d, generator=g)
    K = c[torch.randint(0, centres, (N,), generator=g)] + 0.3 * torch.randn(N, d, generator=g)
    q = c[torch.randint(0, centres, (B,), generator=g)] + 0.3 * torch.randn(B, d, generator=g)
    # Zipf-like values so that the greedy token often has neighbours
    V = torch.multinomial(torch.arange(1, vocab + 1, dtype=torch.float64).pow(-1.1), N,
                          replacement=True, generator=g).to(torch.int32)
    p_lm = torch.softmax(torch.randn(B, vocab, generator=g) * 3, dim=1)
    dt = synth.torch_dtype(dtype)
    return K.to(dt).cuda(), V.cuda(), q.to(dt).cuda(), p_lm.cuda()


@pytest.mark.parametrize("alpha,tau,delta", [(0.3, 0.1, 0.5), (0.2, 0.1, 0.5), (0.9, 0.05, 0.3)])
def test_nest_decision_step_matches_oracle(nest, alpha, tau, delta):
    K, V, q, p_lm = _case(30000, 512, 12, 400, seed=40)
    ds = nest.Datastore(K, V, 400)
    s, idx = ds.search(q, 128)
    p_m, lam = ds.mix_rrc(s, idx, p_lm, 1 / np.sqrt(512), alpha, tau)
    o = ds.decide(p_m, s, idx, lam, delta)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    s_np, i_np = s.cpu().numpy(), idx.cpu().numpy()
    check_mix(p_m.cpu().numpy(), s_np, i_np, V.cpu().numpy(), p_lm.cpu().numpy(),
              1 / np.sqrt(512), None, 400, lam_gpu=lam.cpu().numpy())
    tok, pmax, key, use = oracle.decide(p_m.cpu().numpy().astype(np.float64), s_np, i_np,
                                        V.cpu().numpy(), lam.cpu().numpy().astype(np.float64),
                                        delta)
    assert o["token"].cpu().numpy().tolist() == tok.tolist()
    np.testing.assert_array_equal(o["p_max"].cpu().numpy().astype(np.float64), pmax)
    assert o["span_key"].cpu().numpy().tolist() == key.tolist()
    assert o["use_span"].cpu().numpy().tolist() == use.tolist()
    assert (key >= 0).any(), "the case should exercise span starts"
    ds.close()


def test_verify_spans_matches_oracle(nest):
    g = torch.Generator().manual_seed(41)
    vocab, rows = 3000, 150
    p = torch.softmax(torch.randn(rows, vocab, generator=g) * 4, dim=1)
    draft = torch.randint(0, vocab, (rows,), generator=g, dtype=torch.int32)
    top = p.argmax(1).to(torch.int32)
    pick = torch.rand(rows, generator=g) < 0.7
    draft = torch.where(pick, top, draft)  # mostly confident drafts
    lens = [1, 5, 17, 64, 40, 23]
    off = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32)
    assert int(off[-1]) == rows
    dev = torch.device("cuda")
    K = torch.randn(64, 16, device=dev)
    ds = nest.Datastore(K, torch.zeros(64, dtype=torch.int32, device=dev), vocab)
    for gamma in (5e-1, 5e-2, 5e-4):
        o = ds.verify(p.to(dev), draft.to(dev), off.to(dev), gamma)
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        ratio, acc, n_acc = oracle.verify(p.numpy().astype(np.float64), draft.numpy(),
                                          off.numpy(), gamma)
        g_ratio = o["ratio"].cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(g_ratio, ratio, rtol=2e-6, atol=0)
        g_acc = o["accept"].cpu().numpy()
        near = np.abs(np.minimum(ratio, 1.0) - 0.5) <= 1e-6
        assert np.array_equal(g_acc[~near], acc[~near])
        g_n = o["n_accept"].cpu().numpy()
        for j in range(len(lens)):  # counts follow the GPU's own flags
            lo = int(off[j])
            run = 0
            while run < lens[j] and g_acc[lo + run]:
                run += 1
            assert g_n[j] == run
        if not near.any():
            assert g_n.tolist() == n_acc.tolist()
    ds.close()


@pytest.mark.parametrize("path,B,r,dtype,N", [("tc_scan_kernel", 4, 64, "bf16", 60000),
                                               ("tc_wide_kernel", 40, 128, "bf16", 60000),
                                               ("scan_rows_kernel", 3, 50, "f32", 60000),
                                               # groups of 256: one pass, then two passes,
                                               # on CTA pairs and on single CTAs
                                               ("tc_wide_pair_kernel", 300, 128, "bf16", 60000),
                                               ("tc_wide_pair_kernel", 260, 64, "bf16", 140000),
                                               ("tc_wide2_kernel", 300, 128, "bf16", 60000),
                                               ("tc_wide2_kernel", 260, 64, "bf16", 140000)])
def test_masked_search_skips_used_keys(nest, path, B, r, dtype, N):
    K, V, q, p_lm = _case(N, 256, B, 300, seed=42, dtype=dtype)
    ds = nest.Datastore(K, V, 300)
    if path in ("tc_wide_pair_kernel", "tc_wide2_kernel"):
        ds.use_cta_pairs(path == "tc_wide_pair_kernel")
    assert ds.search_path(B, r) == path
    mask = ds.new_key_mask()
    g = torch.Generator().manual_seed(43)
    # mask the current neighbours of query 0 (an accepted span would be consecutive)
    s0, i0 = ds.search(q, r)
    first = int(i0[0, 0])
    ds.mask_keys(mask, max(0, first - 20), 64)
    bits = torch.rand(N, generator=g) < 0.2
    ds.mask_keys(mask, 1000, 4000)
    words = mask.cpu().numpy().view(np.uint32)
    for k in np.flatnonzero(bits.numpy()):
        words[k >> 5] |= np.uint32(1 << (k & 31))
    mask.copy_(torch.from_numpy(words.view(np.int32)))
    s, idx = ds.search_masked(q, r, mask)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    excl = ((words[np.arange(N) >> 5] >> (np.arange(N) & 31)) & 1).astype(bool)
    K_np, q_np = synth.to_numpy_raw(K), synth.to_numpy_raw(q)
    rows = list(range(0, B, max(1, B // 12))) + [B - 1]
    s_or, i_or = oracle.knn_search(K_np, q_np[rows], r, exclude=excl)
    i_np = idx.cpu().numpy()
    assert not excl[i_np[i_np >= 0]].any()
    check_search(s.cpu().numpy()[rows], i_np[rows], s_or, i_or, K_np, q_np[rows], dtype,
                 np.full(len(rows), N))
    ds.close()


def test_masked_ragged_search(nest):
    K, V, q, p_lm = _case(20000, 256, 6, 300, seed=44)
    ds = nest.Datastore(K, V, 300)
    off = torch.tensor([0, 3000, 3000, 9000, 9100, 15000, 20000], dtype=torch.int64, device="cuda")
    mask = ds.new_key_mask()
    ds.mask_keys(mask, 2500, 700)     # crosses the first segment's end
    ds.mask_keys(mask, 9000, 100)     # a whole segment
    s, idx = ds.search_masked(q, 32, mask, seg_off=off)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    excl = np.zeros(20000, bool)
    excl[2500:3200] = True
    excl[9000:9100] = True
    K_np, q_np = synth.to_numpy_raw(K), synth.to_numpy_raw(q)
    so = off.cpu().numpy()
    s_or, i_or = oracle.knn_search(K_np, q_np, 32, seg_off=so, exclude=excl)
    counts = np.array([max(0, int(so[b + 1] - so[b] - excl[so[b]:so[b + 1]].sum()))
                       for b in range(6)])
    check_search(s.cpu().numpy(), idx.cpu().numpy(), s_or, i_or, K_np, q_np, "bf16", counts)
    assert (idx[3] == -1).all()
    ds.close()


def test_bounded_wait_gives_up_and_the_context_stays_usable(nest):
    """Failure detection without a fault: a kernel waits, through the scan
    kernels' bounded mbarrier wait, on a barrier nothing arrives on.  It must
    give up after about 2 s, the device status must read NEST_ERR_TIMEOUT
    (and be cleared by reading it), and a search afterwards must still run
    and match the oracle."""
    K, V, q, p_lm = _case(20000, 256, 4, 300, seed=45)
    ds = nest.Datastore(K, V, 300)
    waited = ds.selftest_bounded_wait()
    assert 1.9e9 <= waited <= 4e9, waited
    assert ds.device_status() == 8  # NEST_ERR_TIMEOUT
    assert ds.device_status() == 0
    s, idx = ds.search(q, 64)
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    K_np, q_np = synth.to_numpy_raw(K), synth.to_numpy_raw(q)
    s_or, i_or = oracle.knn_search(K_np, q_np, 64)
    check_search(s.cpu().numpy(), idx.cpu().numpy(), s_or, i_or, K_np, q_np, "bf16",
                 np.full(4, 20000))
    ds.close()
