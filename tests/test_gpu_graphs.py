"""CUDA-graph capture of the step.

A serving loop that runs the same shapes every step can capture the step
once and replay it, which removes the host's launch work and the gaps
between the step's kernels.  After nest_datastore_reserve no call of the
step allocates or synchronizes, so torch.cuda.graph captures it.  Replays
read the input buffers the capture saw: new queries are copied into them,
and the replayed outputs must equal, bit for bit, an eager step on the same
inputs (the kernels are deterministic for a fixed batch)."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def _case(N, d, B, vocab, seed):
    g = torch.Generator().manual_seed(seed)
    c = torch.randn(16, d, generator=g)
    K = c[torch.randint(0, 16, (N,), generator=g)] + 0.3 * torch.randn(N, d, generator=g)
    V = torch.randint(0, vocab, (N,), generator=g, dtype=torch.int32)

    def batch(s):
        gg = torch.Generator().manual_seed(s)
        q = c[torch.randint(0, 16, (B,), generator=gg)] + 0.3 * torch.randn(B, d, generator=gg)
        p = torch.softmax(torch.randn(B, vocab, generator=gg) * 2, dim=1)
        return q.to(torch.bfloat16).cuda(), p.cuda()
    return K.to(torch.bfloat16).cuda(), V.cuda(), batch


@pytest.mark.parametrize("N,d,B,r,path", [
    (200000, 1024, 4, 256, "tc_scan_kernel"),      # decode-shaped: scan + merge + mix
    (100000, 256, 40, 128, "tc_wide_kernel"),      # large batch: sample, main pass, selections
    (140000, 128, 300, 64, "tc_wide_pair_kernel"),  # one group of 512 on CTA pairs (clusters)
])
def test_captured_step_replays_match_eager(nest, N, d, B, r, path):
    vocab = 1000
    K, V, batch = _case(N, d, B, vocab, seed=N + B)
    ds = nest.Datastore(K, V, vocab)
    assert ds.search_path(B, r) == path
    ds.reserve(B, r)
    q, p_lm = batch(1)
    out = {}
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(2):
            ds.step(q, r, p_lm, 0.03, 0.7, out=out)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        ds.step(q, r, p_lm, 0.03, 0.7, out=out)
    for s in (2, 3, 4):
        q2, p2 = batch(s)
        q.copy_(q2)
        p_lm.copy_(p2)
        g.replay()
        torch.cuda.synchronize()
        got = {k: v.clone() for k, v in out.items()}
        ref = ds.step(q2, r, p2, 0.03, 0.7)
        torch.cuda.synchronize()
        assert ds.device_status() == 0
        for k in ("s", "idx", "p_m"):
            assert torch.equal(got[k], ref[k]), f"replay {s}: {k} differs from the eager step"
    ds.close()


def test_captured_nest_verification_replays_match_eager(nest):
    """search -> Eq. 4 mix -> Eq. 7 verification of one drafted span, captured once."""
    N, d, B, r, vocab = 20000, 512, 16, 128, 700
    K, V, batch = _case(N, d, B, vocab, seed=5)
    ds = nest.Datastore(K, V, vocab)
    ds.reserve(B, r)
    q, p_lm = batch(1)
    draft = torch.randint(0, vocab, (B,), dtype=torch.int32, device="cuda")
    off = torch.tensor([0, B // 2, B], dtype=torch.int32, device="cuda")

    def run():
        s, idx = ds.search(q, r)
        p_m, lam = ds.mix_rrc(s, idx, p_lm, 0.05, 0.3, 0.1)
        return ds.verify(p_m, draft, off, 0.5)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        o = run()
    q2, p2 = batch(7)
    q.copy_(q2)
    p_lm.copy_(p2)
    g.replay()
    torch.cuda.synchronize()
    got = {k: v.clone() for k, v in o.items()}
    ref = run()
    torch.cuda.synchronize()
    assert ds.device_status() == 0
    for k in ("ratio", "accept", "n_accept"):
        assert torch.equal(got[k], ref[k]), k
    ds.close()
