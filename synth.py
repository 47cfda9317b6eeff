"""Seeded synthetic inputs shaped like the paper's kNN-LM workloads.

Shared by the tests and ``bench.py`` (for both the CUDA path and the oracle).
This module draws random numbers only; it holds none of the method's
arithmetic (no distance, selection, softmax over neighbours or mixing).

The paper's datastores are Llama-2 hidden states over Wikipedia / Pile of Law
passages, which are not available here.  These generators stand in for them
with the same shapes: hidden size d (4096 for 7B, 8192 for 70B), clustered
keys (a Gaussian mixture, like hidden states of related contexts), values
drawn from a Zipf(1.1) law over the vocabulary (like token frequencies),
r = 1024 neighbours (App. A), b = 40 passages per query for the second-stage
search (Sec. 4 setup), and p_LM a softmax over Gaussian logits.
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: datastore shape, query batch and step settings."""
    name: str
    dtype: str            # "f32" or "bf16": element type of keys and queries
    d: int                # hidden size
    N: int                # datastore keys (for ragged: total keys of all segments)
    B: int                # queries per step
    r: int                # neighbours per query
    vocab: int
    mu: float             # inverse temperature of Eq. 2
    lam: float            # lambda of Eq. 3
    logit_std: float      # std of the Gaussian logits behind p_LM
    centres: int = 0      # 0: keys iid N(0,1); else Gaussian mixture with this many centres
    centre_std: float = 1.0
    within_std: float = 0.3
    passages: int = 0     # >0: ragged second-stage search, passages per query
    passage_len: int = 0
    seed: int = 0

    @property
    def ragged(self) -> bool:
        return self.passages > 0


WORKLOADS = {
    # fp32 d=64, N=4096 iid N(0,1) keys, Zipf values over 1000, B=8, r=16
    "tiny": Workload("tiny", "f32", 64, 4096, 8, 16, 1000, 1 / 8, 0.75, 2.0),
    # 7B hidden size, 1M keys from 256 centres, decode batch 4, r=1024
    "decode": Workload("decode", "bf16", 4096, 1 << 20, 4, 1024, 32000, 1 / 64, 0.8, 3.0,
                       centres=256),
    # second-stage search: 32 queries x 40 passages x 256 tokens each
    "ragged": Workload("ragged", "bf16", 4096, 32 * 40 * 256, 32, 64, 32000, 1 / 64, 0.7, 3.0,
                       passages=40, passage_len=256),
    # large query batch over 4M keys
    "large_batch": Workload("large_batch", "bf16", 4096, 1 << 22, 512, 256, 32000, 1 / 64, 0.8,
                            3.0, centres=256),
    # NEST verification of one drafted span: the on-the-fly datastore K' of one
    # query (40 passages x 256 tokens around 40 passage centres) searched by the
    # n = 64 drafted positions at once (App. A: n-gram length 64, top-1024)
    "nest_span": Workload("nest_span", "bf16", 4096, 40 * 256, 64, 1024, 32000, 1 / 64, 0.8, 3.0,
                          centres=40),
    # 70B hidden size over 8M keys (128 GiB); B is swept over 1, 8, 64, 256
    "hidden8192": Workload("hidden8192", "bf16", 8192, 1 << 23, 1, 1024, 32000,
                           1 / math.sqrt(8192), 0.8, 3.0, centres=256),
}


def torch_dtype(name: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[name]


def generator(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def zipf_values(n: int, vocab: int, s: float, gen: torch.Generator, device) -> torch.Tensor:
    """n token ids with P(id = k - 1) proportional to k^-s, k = 1..vocab (int32).

    Inverse-CDF sampling over the fp64 cumulative table.
    """
    ranks = torch.arange(1, vocab + 1, dtype=torch.float64, device=device)
    cdf = torch.cumsum(ranks.pow(-s), 0)
    cdf = cdf / cdf[-1]
    out = torch.empty(n, dtype=torch.int32, device=device)
    step = 1 << 22
    for lo in range(0, n, step):
        hi = min(n, lo + step)
        u = torch.rand(hi - lo, dtype=torch.float64, generator=gen, device=device)
        ids = torch.searchsorted(cdf, u, right=True).clamp_(max=vocab - 1)
        out[lo:hi] = ids.to(torch.int32)
    return out


def p_lm(B: int, vocab: int, logit_std: float, gen: torch.Generator, device) -> torch.Tensor:
    """B x vocab fp32 rows: softmax of N(0, logit_std^2) logits (stand-in LM output)."""
    logits = torch.randn(B, vocab, generator=gen, device=device, dtype=torch.float32)
    return torch.softmax(logits * logit_std, dim=1).contiguous()


def _fill_rows(out: torch.Tensor, centre_of_row, centres: torch.Tensor | None,
               within_std: float, gen: torch.Generator, chunk: int = 1 << 17) -> None:
    """out[i] = centres[centre_of_row[i]] + within_std * N(0, I), rounded to out.dtype."""
    n, d = out.shape
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        noise = torch.randn(hi - lo, d, generator=gen, device=out.device, dtype=torch.float32)
        if centres is None:
            out[lo:hi] = noise.to(out.dtype)
        else:
            rows = centres.index_select(0, centre_of_row[lo:hi].to(torch.int64))
            out[lo:hi] = (rows + within_std * noise).to(out.dtype)
        del noise


@dataclasses.dataclass
class Inputs:
    K: torch.Tensor          # N x d keys (dtype of the workload)
    V: torch.Tensor          # N int32 token ids
    q: torch.Tensor          # B x d queries
    p_lm: torch.Tensor       # B x vocab fp32
    seg_off: torch.Tensor | None  # B + 1 int64 offsets (ragged) or None


def make_inputs(w: Workload, device="cpu", B: int | None = None, N: int | None = None,
                seed: int | None = None) -> Inputs:
    """Materialise workload ``w`` on ``device`` (B and N may be overridden).

    Full-scan workloads: keys are iid N(0, I) (centres == 0) or a Gaussian
    mixture (centre c_m ~ N(0, centre_std^2 I), key = c_m + within_std N(0, I)
    with m uniform), and each query is drawn the same way around a random
    centre.  Ragged workloads: query b owns passages*passage_len consecutive
    keys, each passage around its own centre, and the query is drawn around
    one of its own passages' centres.
    """
    seed = w.seed if seed is None else seed
    B = w.B if B is None else B
    gen = generator(device, seed)
    dt = torch_dtype(w.dtype)
    d = w.d
    if w.ragged:
        per_q = w.passages * w.passage_len
        N = B * per_q if N is None else N
        n_pass = B * w.passages
        centres = w.centre_std * torch.randn(n_pass, d, generator=gen, device=device)
        centre_of_row = torch.arange(N, device=device, dtype=torch.int64) // w.passage_len
        centre_of_row.clamp_(max=n_pass - 1)
        K = torch.empty(N, d, dtype=dt, device=device)
        _fill_rows(K, centre_of_row, centres, w.within_std, gen)
        pick = torch.randint(0, w.passages, (B,), generator=gen, device=device)
        qc = torch.arange(B, device=device) * w.passages + pick
        q = torch.empty(B, d, dtype=dt, device=device)
        _fill_rows(q, qc, centres, w.within_std, gen)
        seg_off = torch.arange(B + 1, dtype=torch.int64, device=device) * per_q
        seg_off.clamp_(max=N)
    else:
        N = w.N if N is None else N
        K = torch.empty(N, d, dtype=dt, device=device)
        q = torch.empty(B, d, dtype=dt, device=device)
        if w.centres:
            centres = w.centre_std * torch.randn(w.centres, d, generator=gen, device=device)
            assign = torch.randint(0, w.centres, (N,), generator=gen, device=device)
            _fill_rows(K, assign, centres, w.within_std, gen)
            qc = torch.randint(0, w.centres, (B,), generator=gen, device=device)
            _fill_rows(q, qc, centres, w.within_std, gen)
        else:
            _fill_rows(K, None, None, 1.0, gen)
            _fill_rows(q, None, None, 1.0, gen)
        seg_off = None
    V = zipf_values(N, w.vocab, 1.1, gen, device)
    P = p_lm(B, w.vocab, w.logit_std, gen, device)
    return Inputs(K=K, V=V, q=q, p_lm=P, seg_off=seg_off)


def to_numpy_raw(t: torch.Tensor):
    """Host numpy copy of a tensor's exact bytes: bf16 as uint16 bit patterns."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view("uint16")
    return t.numpy()
