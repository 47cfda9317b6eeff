"""Benchmark of the kNN-LM step (search + top-r + Eq. 2 + Eq. 3) on GB300.

Default (headline) workload: the 70B-scale hidden size, bf16 keys d=8192,
N=8,388,608 (128 GiB) from a 256-centre Gaussian mixture, values Zipf(1.1)
over 32000 tokens, B=256 queries, r=1024, mu=1/sqrt(8192), lambda=0.8 -- the
largest workload that fits one GPU, and the batch at which the HBM and the
tensor-core rooflines meet.  A step is one ``nest_knn_step`` over one batch.

Prints ONE JSON line (rank 0): queries/s over all ranks, the dominant
kernel's roofline fraction (CUDA events around that kernel, inside the timed
region), the oracle timed on the host cores on a bounded sample, an
end-to-end number through the public API with host buffers, and the SM
clocks sampled during the timed region.  Its ``suite`` entry holds the other
workloads measured in the same run, each with its own roofline and clocks:
the same datastore at B = 1, 8 and 64, the decode batch (d=4096, 1M keys,
B=4), the second-stage ragged search (32 x 10,240 keys) and the large batch
(4M keys, B=512).

``--impl reference`` times the fp64 CPU oracle instead (the only reference
implementation this method has here), on a bounded sample of the same
workload per step.

Multi-GPU: each rank runs an independent decoding stream (its own datastore
replica and query batches); nothing is exchanged, so ``scaling`` is weak.
"""
from __future__ import annotations

import argparse
import json
import os
import platform
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402

FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=None, choices=sorted(synth.WORKLOADS),
                   help="one workload instead of the default headline + suite")
    p.add_argument("--B", type=int, default=None, help="override the query batch")
    p.add_argument("--N", type=int, default=None,
                   help="override the datastore size (small cases for profiling)")
    p.add_argument("--oracle-queries", type=int, default=2,
                   help="queries in the oracle's bounded sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--e2e-steps", type=int, default=200)
    p.add_argument("--pipeline", choices=["knnlm", "nest", "verify"], default="knnlm",
                   help="knnlm: search + Eq. 2 + Eq. 3 (default); nest: masked search + Eq. 2 + "
                        "Eq. 4 + Eq. 5/6 decision; verify: a batch of drafted positions "
                        "searched, mixed (Eq. 4) and verified (Eq. 7)")
    p.add_argument("--cta-pairs", choices=["auto", "on", "off"], default="auto",
                   help="groups of 256 queries on CTA pairs (nest_datastore_use_cta_pairs): "
                        "auto (the default: pairs for one group), on, or off (single CTAs "
                        "with two key tiles per stage)")
    p.add_argument("--sweep", default=None,
                   help="comma-separated query batch sizes measured on one datastore, one JSON "
                        "line each (e.g. 1,8,64,256 for the d=8192 workload)")
    p.add_argument("--no-suite", action="store_true",
                   help="headline workload only (no other workloads in the line)")
    return p.parse_args()


# The headline workload and batch, and the other workloads measured with it.
HEADLINE = ("hidden8192", 256)
SUITE_SAME_DATASTORE = (64, 8, 1)  # further batches on the headline's datastore
SUITE_OTHERS = (("decode", None), ("ragged", None), ("large_batch", None))


FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0


def peaks():
    """(HBM GB/s, sustained dense bf16 TFLOP/s, 'measured' | 'fallback')."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m["bf16_tflops_sustained"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(device_index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64,
                     device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(world: int, per_rank_units: int, steps: int, max_ms: float) -> float:
    """Whole-job throughput: units processed by all ranks over the slowest rank's time."""
    return world * per_rank_units * steps / (max_ms / 1e3)


def host_keys(K: torch.Tensor, rows: int | None = None):
    """Exact bytes of the first ``rows`` keys on the host (bf16 as uint16), ~1 GiB pieces."""
    import numpy as np
    n = K.shape[0] if rows is None else rows
    step = max(1, (1 << 30) // (K.shape[1] * K.element_size()))
    parts = []
    for lo in range(0, n, step):
        parts.append(synth.to_numpy_raw(K[lo:min(n, lo + step)]))
    return np.concatenate(parts) if len(parts) > 1 else parts[0]


class OracleSampler:
    """Times the fp64 oracle, as it stands, on a bounded sample of the workload.

    Full-scan workloads: ``nq`` queries against the first ``n`` keys (search,
    top-r, Eq. 2, Eq. 3); the oracle's cost grows linearly with the keys
    scanned, so queries/s over the whole datastore is (n / N) * nq / seconds.
    Ragged workloads: ``nq`` queries, each over its own segment.
    """

    def __init__(self, w, x, nq: int):
        import oracle
        oracle.build()
        self.oracle = oracle
        self.w, self.nq = w, nq
        self.x = x
        self.N = x.K.shape[0]
        self.ragged = x.seg_off is not None
        self.V = x.V.cpu().numpy()
        self.q = synth.to_numpy_raw(x.q[:nq])
        self.p_lm = x.p_lm[:nq].cpu().numpy()
        self.K = None  # host copy of the first rows, grown on demand
        if self.ragged:
            so = x.seg_off[:nq + 1].cpu().numpy()
            self.seg = so
            self._host_rows(int(so[-1]))
            self.n = int((so[1:] - so[:-1]).sum())
        else:
            self.n = self.N
        self.threads = oracle.default_threads()

    def _host_rows(self, n: int):
        import numpy as np
        have = 0 if self.K is None else self.K.shape[0]
        if n > have:
            more = host_keys(self.x.K[have:n])
            self.K = more if self.K is None else np.concatenate([self.K, more])
        return self.K[:n]

    def run(self, n: int | None = None) -> float:
        """Seconds for one sample over the first n keys (all sampled keys by default)."""
        w = self.w
        if self.ragged:
            K = self.K
            t0 = time.perf_counter()
            self.oracle.knn_step(K, self.V, self.q, w.r, self.p_lm, w.mu, w.lam, w.vocab,
                                 seg_off=self.seg, nthreads=self.threads)
        else:
            n = self.n if n is None else n
            K = self._host_rows(n)
            t0 = time.perf_counter()
            self.oracle.knn_step(K, self.V[:n], self.q, w.r, self.p_lm, w.mu, w.lam,
                                 w.vocab, nthreads=self.threads)
        return time.perf_counter() - t0

    def fit(self, budget_s: float, max_bytes: int = 4 << 30) -> int:
        """Largest key count (from a short calibration) whose sample fits the
        budget, at most ``max_bytes`` of keys copied to the host."""
        if self.ragged:
            return self.n
        row = self.x.K.shape[1] * self.x.K.element_size()
        cap = max(1024, max_bytes // row)
        probe = min(self.n, 16384, cap)
        t = self.run(probe)
        n = int(probe * budget_s / max(t, 1e-6))
        return max(min(self.n, n, cap), min(self.n, 1024))

    def queries_per_s(self, n: int, seconds: float) -> float:
        if self.ragged:
            return self.nq / seconds
        return self.nq * (n / self.N) / seconds

    def keys_per_s(self, n: int, seconds: float) -> float:
        """(query, key) distance evaluations per second of the sample."""
        return (self.n if self.ragged else self.nq * n) / seconds

    def describe(self, n: int) -> str:
        w = self.w
        if self.ragged:
            return (f"{self.nq} queries, each over its own candidate segment ({self.n} key "
                    f"scans in all), top-{w.r}, Eq. 2 + Eq. 3 over {w.vocab} tokens")
        return (f"{self.nq} queries against the first {n} of {self.N} keys, top-{w.r}, Eq. 2 + "
                f"Eq. 3 over {w.vocab} tokens; queries/s scaled by {n}/{self.N} (cost is "
                f"linear in the keys scanned)")


def cpu_model() -> str:
    """The host CPU's model name (or architecture) from /proc/cpuinfo."""
    try:
        with open("/proc/cpuinfo") as f:
            text = f.read()
    except OSError:
        return platform.machine()
    for key in ("model name", "Model Name", "CPU part"):
        for line in text.splitlines():
            if line.split(":")[0].strip() == key:
                val = line.split(":", 1)[1].strip()
                if key != "CPU part":
                    return val
                names = {"0xd4f": "Arm Neoverse V2", "0xd40": "Arm Neoverse V1",
                         "0xd0c": "Arm Neoverse N1", "0xd49": "Arm Neoverse N2"}
                return f"{platform.machine()} {names.get(val, 'CPU part ' + val)}"
    return platform.machine()


def oracle_queries_for(w, x, nq: int, budget_s: float) -> int:
    """Queries of the oracle sample: more of them when the key sample is
    capped by its size on the host, so that the sample still takes about
    budget_s of CPU time (d=8192: 4 GiB are 262,144 keys)."""
    if w.ragged:
        return nq
    row = x.K.shape[1] * x.K.element_size()
    keys = min(x.K.shape[0], (4 << 30) // row)
    # the oracle evaluates about 1.4e10 / d (query, key) distances per second on 16 cores
    per_s = 1.4e10 / w.d * max(1, os.cpu_count() or 1) / 16
    want = int(budget_s * per_s / keys)
    return max(nq, min(x.q.shape[0], want))


def cpu_baseline(w, x, nq: int, budget_s: float = 15.0):
    """The oracle on the host cores: one bounded sample of ~budget_s seconds."""
    nq = oracle_queries_for(w, x, nq, budget_s)
    smp = OracleSampler(w, x, nq)
    n = smp.fit(budget_s)
    sec = smp.run(n)
    return {"value": smp.queries_per_s(n, sec), "unit": "queries/s", "cores": smp.threads,
            "kind": "oracle", "sample": smp.describe(n), "seconds": sec,
            "keys_per_s": smp.keys_per_s(n, sec), "cpu": cpu_model()}


def run_reference(args, w, B, world, rank):
    """``--impl reference``: the oracle on the host cores, each step a bounded sample."""
    if rank != 0:
        return
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    x = synth.make_inputs(w, device=dev, B=B, N=args.N)
    total_steps = args.steps + args.warmup
    per_step = max(0.05, min(10.0, 150.0 / max(1, total_steps)))
    nq = oracle_queries_for(w, x, min(args.oracle_queries, x.q.shape[0]), per_step)
    smp = OracleSampler(w, x, nq)
    n = smp.fit(per_step)
    times = []
    for i in range(total_steps):
        t = smp.run(n)
        if i >= args.warmup:
            times.append(t)
    total = sum(times)
    value = smp.queries_per_s(n, total / len(times))
    line = {
        "impl": "reference", "metric": "queries/s for fused kNN search+top-r+p_M mix",
        "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(w, x),
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": smp.threads,
                         "kind": "oracle", "sample": smp.describe(n),
                         "keys_per_s": smp.keys_per_s(n, total / len(times)),
                         "cpu": cpu_model()},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# DRAM bytes (read + write) per launch of the dominant kernel, from ncu
# captures (dram__bytes_read.sum + dram__bytes_write.sum) of that kernel on a
# smaller case of the same workload, scaled to the full launch by the keys it
# streams; only valid for the kernel versions captured.  None: not captured
# for the current kernel.
TRAFFIC = {
    # tc_wide_pair_kernel main pass, d=8192, B=256 (the default for one group): a 557,056-key
    # capture; reads x N / 557,056, survivor writes as they are (about 4 r' per query at any N)
    ("hidden8192", "tc_wide_pair_kernel", 256): 9239347456 * 8388608 / 557056 + 79070208,
    # tc_wide2_kernel main pass, same workload on single CTAs (--cta-pairs off)
    ("hidden8192", "tc_wide2_kernel", 256): 9177019648 * 8388608 / 557056 + 35045632,
    # tc_wide_pair_kernel<1> main pass, large batch (one group of 512 on CTA pairs, the
    # default): a 262,144-key capture; reads x16, writes (mostly reservation padding) as they are
    ("large_batch", "tc_wide_pair_kernel", 512): 2237294848 * 16 + 38704128,
    # tc_wide2_kernel main pass, large batch on single CTAs (--cta-pairs off): same capture size
    ("large_batch", "tc_wide2_kernel", 512): 2363021056 * 16 + 33024256,
    # tc_scan_kernel<4>, decode: a 65,536-key capture; reads x16, per-CTA list writes as they are
    ("decode", "tc_scan_kernel", 4): 537274880 * 16 + 2926080,
    # tc_scan_kernel<1>, ragged: captured at full size
    ("ragged", "tc_scan_kernel", 32): 2686010112 + 2874880,
}


def dram_traffic(w, args, kernel, B):
    if args.N is not None:
        return None
    return TRAFFIC.get((w.name, kernel, B))


DESCRIPTIONS = {
    "tiny": "tiny exact kNN-LM step (fp32, d=64, 4,096 keys)",
    "decode": "decode-batch full-datastore search (7B hidden size d=4096, 1,048,576 keys)",
    "ragged": "two-stage ragged search (NEST second stage, 40 passages x 256 keys per query)",
    "large_batch": "large-batch prefill-style search (d=4096, 4,194,304 keys)",
    "nest_span": "span verification batch over one query's K' (40 passages x 256 keys)",
    "hidden8192": "70B-scale hidden size (d=8192, 8,388,608 keys, 128 GiB)",
}


def config_of(w, x, pipeline="knnlm"):
    B = x.q.shape[0]
    return {"workload": w.name, "description": DESCRIPTIONS.get(w.name, w.name),
            "pipeline": pipeline, "N": int(x.K.shape[0]), "d": w.d, "B": int(B), "r": w.r,
            "vocab": w.vocab, "key_dtype": w.dtype, "accumulate": "f32",
            "mu": w.mu, "lambda": w.lam,
            "ragged": bool(w.ragged),
            "l2": "no flush: the keys streamed every step exceed the 129 MB L2"}


def main():
    args = parse()
    world, rank, local = dist_setup()
    if args.workload is None:
        name, B_head = HEADLINE
        suite = (not args.no_suite and args.sweep is None and args.pipeline == "knnlm"
                 and args.N is None and args.B is None)
    else:
        name, B_head = args.workload, None
        suite = False
    if args.B is not None:
        B_head = args.B
    w = synth.WORKLOADS[name]
    if args.impl == "reference":
        run_reference(args, w, B_head, world, rank)
        return
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU for the CUDA path")
    torch.cuda.set_device(local)
    import paper_2405_19325_gb300 as nest
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()

    dev = torch.device("cuda", local)
    sweep = [int(v) for v in args.sweep.split(",")] if args.sweep else [B_head]
    B_gen = max(b for b in sweep if b is not None) if any(b is not None for b in sweep) else None
    x = synth.make_inputs(w, device=dev, B=B_gen, N=args.N, seed=w.seed + rank)
    ds = nest.Datastore(x.K, x.V, w.vocab)
    ds.use_cta_pairs({"auto": None, "on": True, "off": False}[args.cta_pairs])
    lines = []
    for B in sweep:
        lines.append(measure(args, w, x, ds, B if B is not None else x.q.shape[0], world, rank,
                             local))
        if rank == 0 and not suite:
            print(json.dumps(lines[-1]), flush=True)
    if suite:
        extras = {}
        for B in SUITE_SAME_DATASTORE:
            extras[f"{w.name}_B{B}"] = measure(args, w, x, ds, B, world, rank, local, light=True)
        ds.close()
        del ds, x
        torch.cuda.empty_cache()
        for oname, oB in SUITE_OTHERS:
            ow = synth.WORKLOADS[oname]
            ox = synth.make_inputs(ow, device=dev, B=oB, seed=ow.seed + rank)
            ods = nest.Datastore(ox.K, ox.V, ow.vocab)
            extras[oname] = measure(args, ow, ox, ods, ox.q.shape[0], world, rank, local,
                                    light=True)
            ods.close()
            del ods, ox
            torch.cuda.empty_cache()
        if rank == 0:
            lines[0]["suite"] = extras
            print(json.dumps(lines[0]), flush=True)
    else:
        ds.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


NEST_ALPHA, NEST_TAU, NEST_DELTA, NEST_GAMMA = 0.3, 0.1, 0.5, 5e-2  # App. A (Wikipedia, 70B)


def make_step(args, w, x, ds):
    """(step, metric) for the pipeline: step() runs one pass of the hot path."""
    if args.pipeline == "knnlm":
        out = {}

        def step():
            ds.step(x.q, w.r, x.p_lm, w.mu, w.lam, seg_off=x.seg_off, out=out)
            return out["p_m"]
        return step, "queries/s for fused kNN search+top-r+p_M mix"
    B = x.q.shape[0]
    mask = ds.new_key_mask()
    # keys of previously accepted spans: every 64th run of 64 keys is used
    words = mask.cpu().numpy().view(np.uint32)
    words[::64] = np.uint32(0xFFFFFFFF)
    words[1::64] = np.uint32(0xFFFFFFFF)
    mask.copy_(torch.from_numpy(words.view(np.int32)))
    if args.pipeline == "nest":
        def step():
            s, idx = ds.search_masked(x.q, w.r, mask, seg_off=x.seg_off)
            p_m, lam = ds.mix_rrc(s, idx, x.p_lm, w.mu, NEST_ALPHA, NEST_TAU)
            return ds.decide(p_m, s, idx, lam, NEST_DELTA)["token"]
        return step, ("queries/s for NEST step (masked kNN search+top-r+p_M with RRC lambda_t+"
                      "greedy token/span decision)")
    draft = torch.randint(0, w.vocab, (B,), dtype=torch.int32, device=x.q.device)
    span_off = torch.tensor([0, B], dtype=torch.int32, device=x.q.device)

    def step():
        s, idx = ds.search_masked(x.q, w.r, mask, seg_off=x.seg_off)
        p_m, lam = ds.mix_rrc(s, idx, x.p_lm, w.mu, NEST_ALPHA, NEST_TAU)
        return ds.verify(p_m, draft, span_off, NEST_GAMMA)["n_accept"]
    return step, ("draft positions/s for NEST span verification (kNN search+top-r+p_M with RRC "
                  "lambda_t+relaxed speculative acceptance) of one drafted span")


def graph_replay(step, stream, args, world, B):
    """Times the step replayed from a CUDA graph (captured once, after the
    warm-up has sized the scratch, so that nothing allocates during capture);
    this removes the host's launch work and most gaps between kernels."""
    n = max(1, min(args.steps, 200))
    try:
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            step()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            step()
        for _ in range(3):
            g.replay()
        barrier(world)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n):
            g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
    except RuntimeError as err:
        return {"error": str(err).splitlines()[0][:200]}
    ms = max_over_ranks(e0.elapsed_time(e1), world) / n
    return {"ms_per_step": ms, "value": world * B / (ms / 1e3), "steps": n}


def measure(args, w, x_all, ds, B, world, rank, local, light=False):
    """Time one batch size on an existing datastore; returns the JSON line (rank 0).

    ``light``: a suite entry (value, roofline, clocks, e2e, launches), without
    the CPU baseline, the CUDA-graph replays and the search-only timing."""
    x = synth.Inputs(K=x_all.K, V=x_all.V, q=x_all.q[:B].contiguous(),
                     p_lm=x_all.p_lm[:B].contiguous(),
                     seg_off=x_all.seg_off[:B + 1].contiguous() if x_all.seg_off is not None else None)
    step, metric = make_step(args, w, x, ds)
    step()  # allocates scratch once
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    if ds.device_status() != 0:
        raise SystemExit("device status error during warm-up")

    # ---- timed region: K steps, CUDA events on the launching stream
    ds.timing_enable(True)
    ds.timing_read()
    launches0 = ds.launch_count()
    barrier(world)
    torch.cuda.synchronize()
    clocks = Clocks(local)
    time.sleep(0.3)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step()
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(world)
    ms_local = t0.elapsed_time(t1)
    launches = ds.launch_count() - launches0
    scan_ms, scan_n = ds.timing_read()
    ds.timing_enable(False)
    if ds.device_status() != 0:
        raise SystemExit("device status error during the timed steps")
    ms = max_over_ranks(ms_local, world)
    value = aggregate(world, B, args.steps, ms)
    step_ms = ms / args.steps

    # ---- roofline of the dominant kernel (the key scan)
    esize = 2 if w.dtype == "bf16" else 4
    if x.seg_off is not None:
        keys_scanned = int((x.seg_off[1:] - x.seg_off[:-1]).sum().item())
        pairs = keys_scanned            # each key is compared with its own query only
    else:
        keys_scanned = x.K.shape[0]
        pairs = keys_scanned * B
    alg_bytes = keys_scanned * (w.d * esize + 4) + B * w.d * esize
    alg_flops = 2 * pairs * w.d
    scan_avg_ms = scan_ms / max(1, scan_n)
    hbm_peak, tc_peak, peak_kind = peaks()
    t_hbm = alg_bytes / (hbm_peak * 1e9)
    t_tc = alg_flops / (tc_peak * 1e12)
    kernel = ds.search_path(B, w.r, ragged=x.seg_off is not None)
    hbm_frac = alg_bytes / (scan_avg_ms / 1e3) / 1e9 / hbm_peak
    tensor_frac = alg_flops / (scan_avg_ms / 1e3) / 1e12 / tc_peak
    common = {"traffic": dram_traffic(w, args, kernel, B), "kernel": kernel,
              "alg_flops_per_launch": alg_flops, "alg_bytes_per_launch": alg_bytes,
              "hbm_frac": hbm_frac, "tensor_frac": tensor_frac,
              "launch_ms": scan_avg_ms, "share_of_step": scan_ms / ms_local}
    if clk and clk.get("sm_mhz"):
        # the power cap moves the SM clock in tensor-bound runs: time x clock
        common["launch_ms_x_sm_ghz"] = scan_avg_ms * clk["sm_mhz"] / 1e3
    if t_tc > t_hbm:
        achieved = alg_flops / (scan_avg_ms / 1e3) / 1e12
        roofline = {"bound": "tensor", "achieved": achieved, "peak": tc_peak, "unit": "TFLOP/s",
                    "frac": achieved / tc_peak,
                    "peak_kind": peak_kind + " (bf16 dense, sustained)", **common}
    else:
        achieved = alg_bytes / (scan_avg_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                    "frac": achieved / hbm_peak, "peak_kind": peak_kind, **common}

    graph = search = None
    if not light:
        # ---- the same step captured once in a CUDA graph and replayed
        graph = graph_replay(step, stream, args, world, B)
        if ds.device_status() != 0:
            raise SystemExit("device status error during the graph replays")

        # ---- the search alone (scan, merge or selection, re-ranking; no mix), same batch
        s_buf = torch.empty(B, w.r, dtype=torch.float32, device=x.q.device)
        i_buf = torch.empty(B, w.r, dtype=torch.int64, device=x.q.device)
        n_search = max(1, min(args.steps, 200))
        for _ in range(3):
            ds.search(x.q, w.r, seg_off=x.seg_off, s_out=s_buf, idx_out=i_buf)
        barrier(world)
        torch.cuda.synchronize()
        u0 = torch.cuda.Event(enable_timing=True)
        u1 = torch.cuda.Event(enable_timing=True)
        u0.record(stream)
        for _ in range(n_search):
            ds.search(x.q, w.r, seg_off=x.seg_off, s_out=s_buf, idx_out=i_buf)
        u1.record(stream)
        torch.cuda.synchronize()
        search_ms = max_over_ranks(u0.elapsed_time(u1), world) / n_search
        if ds.device_status() != 0:
            raise SystemExit("device status error during the search-only steps")
        search = {"call": "nest_knn_search", "ms": search_ms,
                  "queries_per_s": world * B / (search_ms / 1e3), "steps": n_search}

    # ---- end to end through the public API with pinned host buffers
    q_h = x.q.cpu().pin_memory()
    p_h = x.p_lm.cpu().pin_memory()
    so_h = x.seg_off.cpu().pin_memory() if x.seg_off is not None else None
    h2d = q_h.numel() * q_h.element_size() + p_h.numel() * 4 + (
        so_h.numel() * 8 if so_h is not None else 0)
    if args.pipeline == "knnlm":
        staging = {}

        def e2e_step():
            ds.step_host(q_h, w.r, p_h, w.mu, w.lam, seg_off_host=so_h, staging=staging)
        d2h = B * w.vocab * 4 + B * w.r * 4 + B * w.r * 8
    else:
        # inputs copied into the tensors the step reads, the step's decision read back
        res = step()
        res_h = torch.empty(res.shape, dtype=res.dtype).pin_memory()

        def e2e_step():
            x.q.copy_(q_h, non_blocking=True)
            x.p_lm.copy_(p_h, non_blocking=True)
            if so_h is not None:
                x.seg_off.copy_(so_h, non_blocking=True)
            res_h.copy_(step(), non_blocking=True)
            stream.synchronize()
        d2h = res_h.numel() * res_h.element_size()
    # about three seconds of end-to-end steps at most (and at least five)
    n_e2e = max(5, min(args.e2e_steps, int(3000.0 / max(step_ms, 1e-3))))
    # clocks of this loop too: it runs seconds after the timed region, and
    # where the power cap sets the clock the two can differ by a few per cent
    e2e_clocks = Clocks(local)
    for _ in range(3):
        e2e_step()
    barrier(world)
    te = time.perf_counter()
    for _ in range(n_e2e):
        e2e_step()
    e2e_s = max_over_ranks(time.perf_counter() - te, world)
    e2e = {"value": world * B * n_e2e / e2e_s,
           "unit": "positions/s" if args.pipeline == "verify" else "queries/s",
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n_e2e,
           "clocks": e2e_clocks.stop()}

    unit = "positions/s" if args.pipeline == "verify" else "queries/s"
    if light:
        if rank != 0:
            return None
        return {"value": value, "unit": unit, "ms_per_step": step_ms,
                "config": config_of(w, x, args.pipeline),
                "keys_scanned_per_s": world * keys_scanned * args.steps / (ms / 1e3),
                "roofline": roofline, "e2e": e2e, "gpu_launches": launches, "clocks": clk}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, x, min(args.oracle_queries, B))
        cpu.pop("seconds", None)

    line = None
    if rank == 0:
        line = {
            "metric": metric, "value": value, "unit": unit, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32",
            "data": "synthetic", "config": config_of(w, x, args.pipeline),
            "keys_scanned_per_s": world * keys_scanned * args.steps / (ms / 1e3),
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "search": search,
            "graph": graph,
            "gpu_launches": launches, "clocks": clk,
        }
    return line


if __name__ == "__main__":
    main()
