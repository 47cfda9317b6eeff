"""The search planner on a machine without a GPU (nest_plan_offline).

nest_plan_offline runs the planning code of nest_knn_search for a given
datastore shape and device (SM count, shared memory per block), so the host
logic that picks the kernel, splits the work and sizes the scratch is
checked here without a GPU:
  * the benchmarked workloads get the plans their descriptions state (one
    wave of CTAs on 152 SMs, the 65,536-key threshold sample, the static
    array's 8 MiB budget for the decode search);
  * every shape of the GPU sweeps satisfies the planner's invariants (all
    queries covered, lists with room for a tile of appends, samples of at
    least 65,536 keys, scratch for every list);
  * arguments are checked as nest_datastore_create / nest_knn_search check
    them.
"""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

SMS, SMEM = 152, 232448  # a GB300: 152 SMs, 227 KiB opt-in shared memory per block


@pytest.fixture(scope="module")
def nest():
    from paper_2405_19325_gb300 import build as nest_build
    nest_build.build()
    import paper_2405_19325_gb300 as pkg
    pkg.load_library()
    return pkg


def test_decode_plan(nest):
    """B=4, 1M bf16 keys of 4096, r=1024: the narrow tensor-core scan, one
    group of 4 queries over 152 key ranges (one CTA per SM), scratch within
    the allocation-free entry point's 2^20 words."""
    p = nest.plan_offline(1 << 20, 4096, "bf16", 4, 1024, num_sms=SMS, smem_per_block=SMEM)
    assert p["kernel"] == "tc_scan_kernel"
    assert (p["queries_per_group"], p["groups"], p["parts"]) == (4, 1, SMS)
    assert p["list_capacity"] >= 1024 + 128
    assert p["scratch_bytes"] <= (1 << 20) * 8


def test_large_batch_plan(nest):
    """B=512, 4M keys, r=256: two groups of 256 queries, every key range once
    per group in one wave (2 x 76 CTAs), thresholds from every 64th key
    (max(65,536, 64 r') sampled keys, r' = 256 + 16 screened candidates kept
    for the exact re-ranking).  The main pass admits keys up to the sample's
    32nd distance: about 32 x 64 = 2,048 survivors per query, and the lists
    hold 8x that."""
    p = nest.plan_offline(1 << 22, 4096, "bf16", 512, 256, num_sms=SMS, smem_per_block=SMEM,
                          cta_pairs=False)
    assert p["kernel"] == "tc_wide2_kernel"
    assert (p["queries_per_group"], p["groups"], p["parts"]) == (256, 2, SMS // 2)
    assert p["single_pass"] == 0 and p["sample_stride"] == (1 << 22) // 65536
    assert p["list_capacity"] >= 8 * 32 * 64  # 8x the expected survivors
    # by default (and when forced) the 512 queries are one group on 76 CTA pairs,
    # each pair streaming its key range once for all of them
    for mode in (None, True):
        q = nest.plan_offline(1 << 22, 4096, "bf16", 512, 256, num_sms=SMS, smem_per_block=SMEM,
                              cta_pairs=mode)
        assert q["kernel"] == "tc_wide_pair_kernel"
        assert (q["queries_per_group"], q["groups"], q["parts"], q["stages"]) == (512, 1, SMS // 2, 4)
        assert q["sample_stride"] == p["sample_stride"]


def test_hidden8192_plan_runs_one_group_on_cta_pairs(nest):
    """B=256 at d=8192 over 8M keys is one group of 256 queries: by default
    it runs on 76 CTA pairs (two 256-key tiles per 48 KiB stage, four
    stages); forced off, on 152 single CTAs with three 64 KiB stages."""
    p = nest.plan_offline(1 << 23, 8192, "bf16", 256, 1024, num_sms=SMS, smem_per_block=SMEM)
    assert p["kernel"] == "tc_wide_pair_kernel"
    assert (p["groups"], p["parts"], p["stages"]) == (1, SMS // 2, 4)
    q = nest.plan_offline(1 << 23, 8192, "bf16", 256, 1024, num_sms=SMS, smem_per_block=SMEM,
                          cta_pairs=False)
    assert q["kernel"] == "tc_wide2_kernel"
    assert (q["groups"], q["parts"], q["stages"]) == (1, SMS, 3)
    # batches of 129 to 512 queries are one group on pairs; more are groups of
    # 256 on single CTAs
    for B, kernel in ((129, "tc_wide_pair_kernel"), (128, "tc_wide_kernel"),
                      (257, "tc_wide_pair_kernel"), (513, "tc_wide2_kernel")):
        assert nest.plan_offline(1 << 23, 8192, "bf16", B, 1024, num_sms=SMS,
                                 smem_per_block=SMEM)["kernel"] == kernel, B


def test_ragged_and_fp32_plans(nest):
    p = nest.plan_offline(32 * 10240, 4096, "bf16", 32, 64, ragged=True, num_sms=SMS,
                          smem_per_block=SMEM)
    assert p["kernel"] == "tc_scan_kernel"
    assert (p["queries_per_group"], p["groups"]) == (1, 32)  # one query per CTA, own segment
    # fp32 keys: narrow rows one per thread (the tiny workload: 256-byte rows,
    # all 8 queries in one CTA), wide rows on the column-chunk scan
    p = nest.plan_offline(4096, 64, "f32", 8, 16, num_sms=SMS, smem_per_block=SMEM)
    assert p["kernel"] == "scan_rows_kernel"
    assert (p["queries_per_group"], p["groups"], p["stages"]) == (8, 1, 1)
    assert p["list_capacity"] >= (16 + 16) + 128  # r' plus a tile of appends
    assert nest.plan_offline(1 << 20, 512, "f32", 8, 16, num_sms=SMS,
                             smem_per_block=SMEM)["kernel"] == "scan_rows_kernel"
    assert nest.plan_offline(1 << 20, 516, "f32", 8, 16, num_sms=SMS,
                             smem_per_block=SMEM)["kernel"] == "scan_topr_kernel"
    # ragged fp32 segments: one query per CTA group on either fp32 scan
    for d, kernel in ((64, "scan_rows_kernel"), (1024, "scan_topr_kernel")):
        p = nest.plan_offline(32 * 2560, d, "f32", 32, 16, ragged=True, num_sms=SMS,
                              smem_per_block=SMEM)
        assert p["kernel"] == kernel
        assert (p["queries_per_group"], p["groups"]) == (1, 32)


def test_large_batch_single_pass_when_the_sample_is_every_key(nest):
    p = nest.plan_offline(60000, 256, "bf16", 300, 64, num_sms=SMS, smem_per_block=SMEM)
    assert p["single_pass"] == 1 and p["sample_stride"] == 1
    assert p["list_capacity"] == 60000  # every key's word at its row position


def _sweep_shapes():
    import test_gpu_random_sweep as sweep
    return sweep.CASES + sweep.EDGE_CASES, sweep._pairs


def test_plans_of_every_sweep_shape_keep_the_invariants(nest):
    cases, pairs_of = _sweep_shapes()
    seen = set()
    for c in cases:
        N, d, B, r = c["N"], c["d"], c["B"], c["r"]
        p = nest.plan_offline(N, d, c["dtype"], B, r, ragged=c["ragged"], num_sms=SMS,
                              smem_per_block=SMEM, cta_pairs=pairs_of(c))
        seen.add(p["kernel"])
        tag = f"{c}: {p}"
        qpg, groups = p["queries_per_group"], p["groups"]
        # the smallest ring each kernel is planned with
        assert p["parts"] >= 1 and p["stages"] >= {0: 2, 1: 4, 2: 3, 3: 3, 4: 4, 5: 1}[p["path"]], tag
        assert (c["dtype"] == "f32") == (p["path"] in (0, 5)), tag
        assert (p["path"] == 5) == (c["dtype"] == "f32" and d * 4 <= 2048), tag
        if c["ragged"]:
            assert qpg == 1 and groups == B, tag
        else:
            assert groups * qpg >= B > (groups - 1) * qpg, tag
        if p["path"] in (0, 1, 5):
            # room for a list of r plus the appends of at least one block of keys
            assert p["list_capacity"] > r, tag
            assert p["scratch_bytes"] >= groups * p["parts"] * qpg * r * 8, tag
        else:
            assert not c["ragged"] and c["dtype"] == "bf16", tag
            # pairs when forced, or automatically for one group of up to 512
            assert (p["path"] == 4) == (qpg >= 256 and (pairs_of(c) is True or B <= 512)), tag
            # groups of 512 only on pairs, and only for 257 to 512 queries
            assert (qpg == 512) == (p["path"] == 4 and 256 < B <= 512), tag
            if p["single_pass"]:
                assert p["sample_stride"] == 1 and p["list_capacity"] == N, tag
            else:
                # r' = r + m screened candidates, m = r / 16 within [16, 128]
                rp = r + min(128, max(16, r // 16))
                target = max(65536, 64 * rp)
                assert p["sample_stride"] == N // target >= 2, tag
                assert N // p["sample_stride"] >= target, tag
                assert p["list_capacity"] >= min(N, 8 * rp), tag
            assert p["scratch_bytes"] >= B * p["list_capacity"] * 8, tag
    assert seen >= {"scan_topr_kernel", "scan_rows_kernel", "tc_scan_kernel", "tc_wide_kernel",
                    "tc_wide2_kernel",
                    "tc_wide_pair_kernel"}, seen


def test_plan_argument_checks(nest):
    from paper_2405_19325_gb300 import NestError
    bad = [
        (dict(N=0, d=64, dtype="f32", B=1, r=1), 1),
        (dict(N=10, d=3, dtype="f32", B=1, r=1), 3),        # 12-byte rows
        (dict(N=10, d=8200, dtype="bf16", B=1, r=1), 9),    # row above NEST_MAX_ROW_BYTES
        (dict(N=10, d=64, dtype="f32", B=0, r=1), 1),
        (dict(N=10, d=64, dtype="f32", B=65536, r=1), 1),
        (dict(N=10, d=64, dtype="f32", B=1, r=4097), 1),
    ]
    for kw, code in bad:
        with pytest.raises(NestError) as e:
            nest.plan_offline(**kw, num_sms=SMS, smem_per_block=SMEM)
        assert e.value.code == code, kw
    with pytest.raises(ValueError):
        nest.plan_offline(10, 64, "f16", 1, 1)


def test_largest_tensor_core_datastore_keeps_32_bit_lists(nest):
    """At the largest bf16 datastore the tensor-core paths take (0x7FFFFF00
    keys), every list the large-batch kernels index with 32-bit positions
    stays below 2^31 words: samples hold at least 64 r keys, so a query's
    survivors are at most about N / 8 plus the reservation blocks."""
    N = 0x7FFFFF00
    for B, r in [(17, 1), (64, 1024), (512, 4096)]:
        p = nest.plan_offline(N, 8, "bf16", B, r, num_sms=SMS, smem_per_block=SMEM)
        assert p["path"] in (2, 3, 4), p
        assert p["list_capacity"] < 2 ** 31, p
        # each part has up to 8 reserving warps per column (16 on a pair with
        # two 256-key tiles per step), each holding a block of at most 1024 slots
        warps = 16 if p["path"] == 4 else 8
        assert p["list_capacity"] <= N // 8 + p["parts"] * warps * 1024, p
