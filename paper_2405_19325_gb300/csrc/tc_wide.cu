// tc_wide.cu -- the search for large query batches (Sec. 2.2 / App. A: the
// r nearest keys of each query, s = -||q - k||^2), where per-query candidate
// lists no longer fit in one CTA's shared memory.  "r" below is the number
// of screened candidates the search keeps for the exact re-ranking
// (refine.cu), r' = r + margin of the caller.
//
//   0. wide_qnorm_kernel computes ||q||^2 of every query once.
//   1. A sampling pre-pass: the scan kernel over a tensor map that reads
//      every stride-th key, admitting every sampled key (each list holds the
//      sample in row order), then gselect_kernel sorts each query's r
//      nearest sampled keys.  The sample's r-th distance bounds the query's
//      true r-th distance from above.
//   2. The main pass streams every key once per group of queries with
//      tcgen05.mma (M = 128 keys, N = up to 256 queries, K = 16):
//      tc_wide_kernel keeps one key tile per stage and two TMEM accumulators
//      of N columns; groups of 256 run on tc_wide2_kernel (two key tiles per
//      stage, one accumulator each) or on CTA pairs (tc_wide_pair_kernel:
//      M = 256 keys over the pair, groups of 256 or 512; the default when the
//      batch is one group).  The epilogue warps form ||q||^2 + ||k||^2 -
//      2 q.k, admit the keys up to the sample's j-th distance (an optimistic
//      threshold, j = max(32, 4 r / stride), that lets about 4 r keys
//      through) and append them to that query's global list through
//      per-warp slot reservations.
//   3. Recovery, up to three rounds of two kernels that return at once when
//      nothing needs them: gselect_kernel in preparation mode flags a list
//      with fewer than r real words (scanned again up to the sample's r-th
//      distance) or one that overflowed its capacity (scanned again up to
//      the r-th smallest word it holds), and tc_wide_kernel<NM, true>
//      rescans the flagged groups.
//   4. gselect_kernel takes the exact r smallest words of each list (three
//      streaming passes, then a select in shared memory) for the exact
//      re-ranking.
#include <cmath>
#include <cuda.h>

#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kTileM = 128;
constexpr int kChunkK = 64;
constexpr int kABytes = kTileM * kChunkK * 2;
constexpr int kMaxStagesW = 12;
constexpr int kEpiThreads = 128;
constexpr int kSelThreads = 1024;

constexpr int kMaxEpiWarps = 16;
constexpr int kStageK = 4;  // admitted keys a lane stages per 32-column block

template <int NM>
struct WideShared {
    float qn[NM];      // ||q||^2 of the group's queries
    uint32_t thr[NM];  // a key is admitted iff the fp32 bits of its distance, as signed
                       // integers, are <= thr (0xFFFFFFFF = -1 for padding columns)
    // Slots [x, y) of query column c's global list reserved by an epilogue
    // warp and not yet written (used when WideArgs::resv > 0); x passes y
    // once the block is used up.  Each warp has one entry per column it
    // drains (NM / 2 or NM columns; 128 in each of a CTA pair's sixteen
    // epilogue warps for groups of 512).
    int2 resv[NM <= 256 ? 8 * NM : 16 * 128];
    // Distance bits of the keys a lane admitted in one 32-column block, in
    // column order: [warp][k][lane].
    uint32_t stage[kMaxEpiWarps][kStageK][32];
    uint64_t full[kMaxStagesW];
    uint64_t empty[kMaxStagesW];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    int issued;
};

template <int NM>
constexpr int stage_bytes() { return kABytes + NM * kChunkK * 2; }

template <int NM>
constexpr uint32_t tmem_cols()
{
    return (2 * NM) <= 32 ? 32u : (2 * NM) <= 64 ? 64u : (2 * NM) <= 128 ? 128u : (2 * NM) <= 256 ? 256u : 512u;
}

__device__ __forceinline__ void wait_or_abort_w(uint64_t* bar, uint32_t parity, int* abort_flag,
                                                int* status)
{
    if (*reinterpret_cast<volatile int*>(abort_flag)) return;
    if (!mbar_wait_bounded(bar, parity)) {
        record_status(status, NEST_ERR_TIMEOUT);
        *reinterpret_cast<volatile int*>(abort_flag) = 1;
    }
}

// Pads slots [from, to) of list `col` with kNoCandidate (reserved, never written).
// Slot numbers are taken as unsigned: a count that has passed 2^31 (far
// beyond any list) writes nothing.
__device__ __forceinline__ void wide_pad(const WideArgs& a, int64_t col, int from, int to)
{
    uint64_t* list = a.cand + col * a.cap;
    const uint64_t end = (uint32_t)to < (uint64_t)a.cap ? (uint32_t)to : (uint64_t)a.cap;
    for (uint64_t p = (uint32_t)from; p < end; ++p) list[p] = kNoCandidate;
}

// Epilogue of W accumulator columns (queries c0 .. c0 + W - 1) of one key
// row: D = ||q||^2 + ||k||^2 - 2 q.k, clamped at 0, admitted at or below the
// query's threshold.  The admission test is branch-free over the W columns.
//
// On the pass that admits every key (no thresholds), word positions are the
// tensor-map rows, so no slots are taken.  Appending, when some lane admits a
// key on a thresholded pass:
//  * with reservations (a.resv > 0) and at most kStageK admitted keys per
//    lane, a branch-free pass stages each lane's admitted distances in
//    shared memory, then each lane takes a slot per key from this warp's
//    block for that column (a shared-memory atomic), or one fresh slot of
//    the list once the block is used up;
//  * otherwise the warp forms each column's ballot, lane i takes room in
//    column i's list (from the warp's block, or with one global atomic; all
//    columns' atomics in flight together), and every admitting lane writes
//    its word.
template <int W, int NM, bool WORD = false>
__device__ __forceinline__ void wide_columns(const uint32_t (&acc)[W], int c0, int nqv, float kn,
                                             bool valid, uint32_t key_idx, int64_t pos, int lane,
                                             const WideShared<NM>& sh, int2* resv,
                                             uint32_t* stage, const WideArgs& a, int q0)
{
    if constexpr (WORD) {
        // Recovery pass of overflowed lists: a key is admitted when its whole
        // word (distance bits, key index) is at or below the query's limit
        // (kNoCandidate: the query is not recovering), one list slot per key.
        if (!valid) return;
#pragma unroll 1
        for (int i = 0; i < W; ++i) {
            const int col = c0 + i;
            if (col >= nqv) break;
            const uint64_t lim = __ldg(a.word_lim + q0 + col);
            float dist = fmaf(-2.f, __uint_as_float(acc[i]), sh.qn[col] + kn);
            dist = (dist <= 0.f) ? 0.f : dist;
            const uint64_t w = ((uint64_t)__float_as_uint(dist) << 32) | key_idx;
            if (lim != kNoCandidate && w <= lim) {
                const uint32_t slot = (uint32_t)atomicAdd(&a.cnt[q0 + col], 1);
                if (slot < (uint64_t)a.cap) a.cand[(int64_t)(q0 + col) * a.cap + slot] = w;
            }
        }
        return;
    }
    if (a.s_sample == nullptr) {
        // every key is admitted: the word of tensor-map row `pos` goes to
        // position `pos` of each list (masked keys leave a padding word)
        if (pos < 0) return;
#pragma unroll
        for (int v = 0; v < W / 4; ++v) {
            const float4 qv = *reinterpret_cast<const float4*>(sh.qn + c0 + 4 * v);
            const float qa[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int col = c0 + 4 * v + k;
                float dist = fmaf(-2.f, __uint_as_float(acc[4 * v + k]), qa[k] + kn);
                dist = (dist <= 0.f) ? 0.f : dist;
                if (col < nqv)
                    a.cand[(int64_t)(q0 + col) * a.cap + pos] =
                        valid ? (((uint64_t)__float_as_uint(dist) << 32) | key_idx) : kNoCandidate;
            }
        }
        return;
    }
    // Admission: the fp32 bits of D compared as signed integers with the
    // query's threshold (thr[] >= 0; -1 for padding columns).  A negative D
    // (rounding) has the sign bit set and is admitted, as the clamp to 0
    // would; only stored words are clamped.  With reservations, each lane
    // also stages its admitted distances in the same pass (predicated
    // stores, no branch); slot kStageK and beyond are never written.
    const bool staging = a.resv > 0;
    uint32_t* st = stage + lane;
    uint32_t m = 0;
    int n = 0;
    const float2 kn2 = make_float2(kn, kn), m2 = make_float2(-2.f, -2.f);
#pragma unroll
    for (int v = 0; v < W / 4; ++v) {
        const float4 qv = *reinterpret_cast<const float4*>(sh.qn + c0 + 4 * v);
        const int4 tv = *reinterpret_cast<const int4*>(sh.thr + c0 + 4 * v);
        const int ta[4] = {tv.x, tv.y, tv.z, tv.w};
        // two columns per packed add / fma (each lane rounds as fmaf would)
        const float2 d01 = __ffma2_rn(m2,
                                      make_float2(__uint_as_float(acc[4 * v]),
                                                  __uint_as_float(acc[4 * v + 1])),
                                      __fadd2_rn(make_float2(qv.x, qv.y), kn2));
        const float2 d23 = __ffma2_rn(m2,
                                      make_float2(__uint_as_float(acc[4 * v + 2]),
                                                  __uint_as_float(acc[4 * v + 3])),
                                      __fadd2_rn(make_float2(qv.z, qv.w), kn2));
        const float da[4] = {d01.x, d01.y, d23.x, d23.y};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float dist = da[k];
            const bool b = valid && __float_as_int(dist) <= ta[k];
            m |= (b ? 1u : 0u) << (4 * v + k);
            if (staging) {
                st_shared_u32_if(b && n < kStageK, st + n * 32, __float_as_uint(dist));
                n += b ? 1 : 0;
            }
        }
    }
    const uint32_t any = __reduce_or_sync(~0u, m);
    if (any == 0) return;
    if (staging && __all_sync(~0u, n <= kStageK)) {
        // each lane takes one slot per staged key from this warp's block for
        // the column (a shared-memory atomic), or one fresh slot of the list
        // once the block is used up
        __syncwarp();
        uint32_t mm = m;
        for (int j = 0; j < n; ++j) {
            const int col = c0 + __ffs(mm) - 1;
            mm &= mm - 1;
            uint32_t dbits = st[j * 32];
            dbits = (int)dbits < 0 ? 0u : dbits;  // D <= 0 is stored as 0
            int slot = atomicAdd(&resv[col].x, 1);
            if (slot >= resv[col].y) slot = atomicAdd(&a.cnt[q0 + col], 1);
            // a full list drops the key; its count keeps growing past the
            // capacity, which the selection after the pass detects
            if ((uint32_t)slot < (uint64_t)a.cap)
                a.cand[(int64_t)(q0 + col) * a.cap + slot] = ((uint64_t)dbits << 32) | key_idx;
        }
        __syncwarp();
        return;
    }
    uint32_t my_bal = 0;  // lane i: ballot of column c0 + i
#pragma unroll
    for (int i = 0; i < W; ++i) {
        if ((any >> i) & 1u) {
            const uint32_t bal = __ballot_sync(~0u, (m >> i) & 1u);
            if (lane == i) my_bal = bal;
        }
    }
    int base = 0;
    if (my_bal != 0) {
        const int need = __popc(my_bal);
        if (a.resv > 0) {
            // from this warp's block for the column; a new block (padding the
            // rest of the old one) when it cannot hold them
            int2 rv = resv[c0 + lane];
            if (rv.x + need > rv.y) {
                wide_pad(a, q0 + c0 + lane, rv.x, rv.y);
                const int blk = need > a.resv ? need : a.resv;
                rv.x = atomicAdd(&a.cnt[q0 + c0 + lane], blk);
                rv.y = rv.x + blk;
            }
            base = rv.x;
            rv.x += need;
            resv[c0 + lane] = rv;
        } else {
            base = atomicAdd(&a.cnt[q0 + c0 + lane], need);
        }
    }
    const uint32_t lt = lanemask_lt();
#pragma unroll
    for (int i = 0; i < W; ++i) {
        if (!((any >> i) & 1u)) continue;
        const int at = __shfl_sync(~0u, base, i);
        const uint32_t bal = __shfl_sync(~0u, my_bal, i);
        if ((m >> i) & 1u) {
            float dist = fmaf(-2.f, __uint_as_float(acc[i]), sh.qn[c0 + i] + kn);
            dist = (dist <= 0.f) ? 0.f : dist;
            const uint64_t key = ((uint64_t)__float_as_uint(dist) << 32) | key_idx;
            const uint64_t pos = (uint64_t)(uint32_t)at + __popc(bal & lt);
            if (pos < (uint64_t)a.cap) a.cand[(int64_t)(q0 + c0 + i) * a.cap + pos] = key;
        }
    }
}

// First reservations: lane i reserves a.resv slots in each column
// c_begin + i + 32k < c_end for this warp (its atomics all in flight together).
__device__ __forceinline__ void wide_reserve(int2* resv, int c_begin, int c_end, int nqv, int lane,
                                             const WideArgs& a, int q0)
{
    for (int c = c_begin + lane; c < c_end; c += 32) {
        int2 rv = make_int2(0, 0);
        if (a.resv > 0 && c < nqv) {
            rv.x = atomicAdd(&a.cnt[q0 + c], a.resv);
            rv.y = rv.x + a.resv;
        }
        resv[c] = rv;
    }
    __syncwarp();
}

// Pads what is left of this warp's blocks once the pass is done.
__device__ __forceinline__ void wide_release(const int2* resv, int c_begin, int c_end, int nqv,
                                             int lane, const WideArgs& a, int q0)
{
    if (a.resv <= 0) return;
    __syncwarp();
    for (int c = c_begin + lane; c < nqv && c < c_end; c += 32) {
        const int2 rv = resv[c];
        if (rv.x < rv.y) wide_pad(a, q0 + c, rv.x, rv.y);
    }
}

// Drains NCOL columns (queries c_base ..) of one TMEM lane (this thread's
// key row) of an accumulator, starting at tbase, 32 columns per load, and
// hands the accumulator back once they have been read: an arrival on
// `release` in this CTA or, with CLUSTER_RELEASE (a CTA pair), on the even
// CTA's barrier at the shared::cluster address `release_cluster`.  With PIPE
// the next load is in flight while the current columns are tested (more
// registers); without it the other warps of the SM sub-partition hide the
// load latency.
template <int NM, int NCOL, bool PIPE, bool CLUSTER_RELEASE = false, bool WORD = false>
__device__ __forceinline__ void wide_drain_row(uint32_t tbase, int c_base, uint64_t* release,
                                               int nqv, float kn, bool valid, uint32_t key_idx,
                                               int64_t pos, int lane, const WideShared<NM>& sh,
                                               int2* resv,
                                               uint32_t* stage, const WideArgs& a, int q0,
                                               uint32_t release_cluster = 0)
{
    static_assert(NCOL % 64 == 0 || NCOL == 32, "columns are drained in pairs of 32");
    auto hand_back = [&] {
        tc_fence_before();
        if constexpr (CLUSTER_RELEASE) mbar_arrive_cluster(release_cluster);
        else mbar_arrive(release);
    };
    if constexpr (!PIPE) {
#pragma unroll 1
        for (int c0 = 0; c0 < NCOL; c0 += 32) {
            uint32_t acc[32];
            tmem_ld_32_async(tbase + (uint32_t)c0, acc);
            tmem_wait_ld(acc);
            if (c0 + 32 == NCOL) hand_back();
            wide_columns<32, NM, WORD>(acc, c_base + c0, nqv, kn, valid, key_idx, pos, lane, sh,
                                       resv, stage, a, q0);
        }
        return;
    }
    uint32_t a0[32], a1[32];
    tmem_ld_32_async(tbase, a0);
#pragma unroll 1
    for (int c0 = 0; c0 < NCOL; c0 += 64) {
        tmem_wait_ld(a0);
        if (c0 + 32 < NCOL) {
            tmem_ld_32_async(tbase + (uint32_t)(c0 + 32), a1);
        } else {
            hand_back();
        }
        wide_columns<32, NM, WORD>(a0, c_base + c0, nqv, kn, valid, key_idx, pos, lane, sh, resv,
                                   stage, a, q0);
        if (c0 + 32 < NCOL) {
            tmem_wait_ld(a1);
            if (c0 + 64 < NCOL) {
                tmem_ld_32_async(tbase + (uint32_t)(c0 + 64), a0);
            } else {
                hand_back();
            }
            wide_columns<32, NM, WORD>(a1, c_base + c0 + 32, nqv, kn, valid, key_idx, pos, lane, sh,
                                       resv, stage, a, q0);
        }
    }
}

template <int NM, bool WORD = false>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_wide_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ,
                   const WideArgs a)
{
    constexpr int kStage = stage_bytes<NM>();
    constexpr uint32_t kCols = tmem_cols<NM>();
    static_assert(NM % 16 == 0 && NM >= 16 && NM <= 256, "MMA N for M = 128");
    static_assert(kStage % 1024 == 0, "stage must keep 1024-byte alignment");

    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    unsigned char* stages = smem;
    WideShared<NM>& sh = *reinterpret_cast<WideShared<NM>*>(smem + (size_t)a.stages * kStage);

    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // CTAs of the same key range but different query groups are adjacent, so
    // they stream the same tiles at about the same time and share them in L2.
    const int part = blockIdx.x / a.groups, group = blockIdx.x - part * a.groups;
    const int q0 = group * NM;
    const int nqv = min(NM, a.B - q0);
    // a recovery pass runs only for groups with an overflowed list
    if constexpr (WORD) {
        if (a.group_flag[group] == 0) return;
    }

    const int64_t tiles = (a.N + kTileM - 1) / kTileM;
    const int64_t t0 = tiles * part / a.parts, t1 = tiles * (part + 1) / a.parts;
    const int64_t lo = t0 * kTileM;
    const int64_t hi = min(a.N, t1 * kTileM);
    const int ntiles = (int)(t1 - t0);
    const int kc = a.kchunks;
    const int nsteps = ntiles * kc;

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sh.acc_full[b], 1);
            mbar_init(&sh.acc_empty[b], kEpiThreads);
        }
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        sh.issued = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(&sh.tmem_base, kCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0 && nsteps > 0) {
            const uint64_t policy = l2_policy_evict_first();
            int slot = 0;
            uint32_t phase = 0;
            for (int s = 0; s < nsteps; ++s) {
                const int t = s / kc, c = s - t * kc;
                if (s >= a.stages) {
                    wait_or_abort_w(&sh.empty[slot], phase ^ 1u, &sh.abort, a.status);
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                }
                unsigned char* st = stages + (size_t)slot * kStage;
                mbar_arrive_expect_tx(&sh.full[slot], kStage);
                // the last query group reads the keys last: let them leave L2 then
                if (group == a.groups - 1)
                    tma_load_2d_hint(st, &tmK, c * kChunkK, (int32_t)(lo + (int64_t)t * kTileM),
                                     &sh.full[slot], policy);
                else
                    tma_load_2d(st, &tmK, c * kChunkK, (int32_t)(lo + (int64_t)t * kTileM),
                                &sh.full[slot]);
                tma_load_2d(st + kABytes, &tmQ, c * kChunkK, q0, &sh.full[slot]);
                *reinterpret_cast<volatile int*>(&sh.issued) = s + 1;
                if (++slot == a.stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && nsteps > 0) {
            constexpr uint32_t idesc = mma_idesc_bf16(kTileM, NM);
            int slot = 0;
            uint32_t phase = 0;
            for (int j = 0; j < ntiles; ++j) {
                const int buf = j & 1;
                if (j >= 2)
                    wait_or_abort_w(&sh.acc_empty[buf], (uint32_t)((j >> 1) - 1) & 1u, &sh.abort,
                                    a.status);
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * NM);
                for (int c = 0; c < kc; ++c) {
                    wait_or_abort_w(&sh.full[slot], phase, &sh.abort, a.status);
                    tc_fence_after();
                    const unsigned char* st = stages + (size_t)slot * kStage;
                    const uint64_t ad = smem_desc_sw128(st);
                    const uint64_t bd = smem_desc_sw128(st + kABytes);
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k)
                        mma_bf16(d_tmem, ad + 2u * k, bd + 2u * k, idesc, (c | k) != 0);
                    mma_commit(&sh.empty[slot]);
                    if (++slot == a.stages) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                mma_commit(&sh.acc_full[buf]);
            }
            mma_commit(&sh.drain);
            (void)mbar_wait_bounded(&sh.drain, 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int e = tid - 64;
        const int quarter = warp & 3;
        // Admission threshold of each query: every key at or below the r-th
        // distance of the sample (an upper bound of the true r-th distance),
        // or every key on the sampling pass itself (no s_sample).
        for (int j = e; j < NM; j += kEpiThreads) {
            // padding columns: -1 (never admitted); no sample threshold: every key
            uint32_t thr = 0xFFFFFFFFu;
            if (j < nqv) {
                thr = 0x7FFFFFFFu;
                if (a.s_sample != nullptr) {
                    const float s_r = a.s_sample[(int64_t)(q0 + j) * a.r + a.thr_rank - 1];
                    if (s_r > -INFINITY) thr = __float_as_uint(-s_r);
                }
            }
            sh.thr[j] = thr;
            // the pass that admits every key fills whole lists (positions = rows)
            if (a.s_sample == nullptr && part == 0 && j < nqv) a.cnt[q0 + j] = (int32_t)a.N;
        }
        // ||q||^2 of the group's queries, computed once per search
        for (int j = e; j < NM; j += kEpiThreads) sh.qn[j] = j < nqv ? a.qn[q0 + j] : 0.f;
        named_barrier(2, kEpiThreads);
        int2* resv = sh.resv + (warp - 2) * NM;
        uint32_t* stage = &sh.stage[warp - 2][0][0];
        wide_reserve(resv, 0, NM, nqv, lane, a, q0);

        const int row_in_tile = 32 * quarter + lane;
        const int64_t ks = a.key_stride;  // row i of the tensor map is key i * ks
        float kn_next =
            (ntiles > 0 && lo + row_in_tile < hi) ? __ldg(a.knorm + (lo + row_in_tile) * ks) : 0.f;
        for (int j = 0; j < ntiles; ++j) {
            const int buf = j & 1;
            const int64_t row = lo + (int64_t)j * kTileM + row_in_tile;
            const float kn = kn_next;
            kn_next = (row + kTileM < hi) ? __ldg(a.knorm + (row + kTileM) * ks) : 0.f;
            const bool valid = row < hi && !key_masked(a.key_mask, row * ks);
            const int64_t pos = row < hi ? row : -1;
            wait_or_abort_w(&sh.acc_full[buf], (uint32_t)(j >> 1) & 1u, &sh.abort, a.status);
            tc_fence_after();
            const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(buf * NM);
            const uint32_t key_idx = (uint32_t)(row * ks);
            if constexpr (NM == 16) {
                uint32_t acc[16];
                tmem_ld_16(tbase, acc);
                tc_fence_before();
                mbar_arrive(&sh.acc_empty[buf]);
                wide_columns<16, NM, WORD>(acc, 0, nqv, kn, valid, key_idx, pos, lane, sh, resv, stage,
                                           a, q0);
            } else {
                wide_drain_row<NM, NM, true, false, WORD>(tbase, 0, &sh.acc_empty[buf], nqv, kn, valid,
                                                          key_idx, pos, lane, sh, resv, stage, a, q0);
            }
        }
        wide_release(resv, 0, NM, nqv, lane, a, q0);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kCols);
    }
    if (tid == 0 && *reinterpret_cast<volatile int*>(&sh.abort)) {
        const int issued = *reinterpret_cast<volatile int*>(&sh.issued);
        for (int s = max(0, issued - a.stages); s < issued; ++s)
            (void)mbar_wait_bounded(&sh.full[s % a.stages], (uint32_t)(s / a.stages) & 1u);
    }
}

// Two 128-key tiles per pipeline stage for groups of 256 queries: both
// tiles' MMAs (M = 128, N = 256, K = 16 each) read the stage's query chunk,
// so one 64 KiB stage (32 KiB of keys, 32 KiB of queries) carries twice the
// MMA work of a one-tile stage and the stage ring covers twice the latency.
// The two 256-column fp32 accumulators fill TMEM, so a tile pair's epilogue
// runs between its last MMA and the next pair's first; sixteen epilogue
// warps (four per TMEM lane quarter: one per tile and half of the columns)
// keep that gap short.
constexpr int kWide2Epi = 4 * kEpiThreads;
constexpr int kWide2Threads = 64 + kWide2Epi;

__global__ void __launch_bounds__(kWide2Threads, 1)
    tc_wide2_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ,
                    const WideArgs a)
{
    constexpr int NM = 256;
    constexpr int kStage = 2 * kABytes + NM * kChunkK * 2;
    constexpr uint32_t kCols = 512;
    constexpr int kPairKeys = 2 * kTileM;

    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    unsigned char* stages = smem;
    WideShared<NM>& sh = *reinterpret_cast<WideShared<NM>*>(smem + (size_t)a.stages * kStage);

    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int part = blockIdx.x / a.groups, group = blockIdx.x - part * a.groups;
    const int q0 = group * NM;
    const int nqv = min(NM, a.B - q0);

    const int64_t pairs = (a.N + kPairKeys - 1) / kPairKeys;
    const int64_t t0 = pairs * part / a.parts, t1 = pairs * (part + 1) / a.parts;
    const int64_t lo = t0 * kPairKeys;
    const int64_t hi = min(a.N, t1 * kPairKeys);
    const int npairs = (int)(t1 - t0);
    const int kc = a.kchunks;
    const int nsteps = npairs * kc;

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        mbar_init(&sh.acc_full[0], 1);
        mbar_init(&sh.acc_empty[0], kWide2Epi);
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        sh.issued = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(&sh.tmem_base, kCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0 && nsteps > 0) {
            const uint64_t policy = l2_policy_evict_first();
            int slot = 0;
            uint32_t phase = 0;
            for (int s = 0; s < nsteps; ++s) {
                const int t = s / kc, c = s - t * kc;
                if (s >= a.stages) {
                    wait_or_abort_w(&sh.empty[slot], phase ^ 1u, &sh.abort, a.status);
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                }
                unsigned char* st = stages + (size_t)slot * kStage;
                mbar_arrive_expect_tx(&sh.full[slot], kStage);
                const int32_t y = (int32_t)(lo + (int64_t)t * kPairKeys);
                if (group == a.groups - 1) {
                    tma_load_2d_hint(st, &tmK, c * kChunkK, y, &sh.full[slot], policy);
                    tma_load_2d_hint(st + kABytes, &tmK, c * kChunkK, y + kTileM, &sh.full[slot],
                                     policy);
                } else {
                    tma_load_2d(st, &tmK, c * kChunkK, y, &sh.full[slot]);
                    tma_load_2d(st + kABytes, &tmK, c * kChunkK, y + kTileM, &sh.full[slot]);
                }
                tma_load_2d(st + 2 * kABytes, &tmQ, c * kChunkK, q0, &sh.full[slot]);
                *reinterpret_cast<volatile int*>(&sh.issued) = s + 1;
                if (++slot == a.stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && nsteps > 0) {
            constexpr uint32_t idesc = mma_idesc_bf16(kTileM, NM);
            int slot = 0;
            uint32_t phase = 0;
            for (int j = 0; j < npairs; ++j) {
                if (j >= 1)
                    wait_or_abort_w(&sh.acc_empty[0], (uint32_t)(j - 1) & 1u, &sh.abort, a.status);
                tc_fence_after();
                for (int c = 0; c < kc; ++c) {
                    wait_or_abort_w(&sh.full[slot], phase, &sh.abort, a.status);
                    tc_fence_after();
                    const unsigned char* st = stages + (size_t)slot * kStage;
                    const uint64_t ad0 = smem_desc_sw128(st);
                    const uint64_t ad1 = smem_desc_sw128(st + kABytes);
                    const uint64_t bd = smem_desc_sw128(st + 2 * kABytes);
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k) {
                        mma_bf16(tmem, ad0 + 2u * k, bd + 2u * k, idesc, (c | k) != 0);
                        mma_bf16(tmem + (uint32_t)NM, ad1 + 2u * k, bd + 2u * k, idesc, (c | k) != 0);
                    }
                    mma_commit(&sh.empty[slot]);
                    if (++slot == a.stages) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                mma_commit(&sh.acc_full[0]);
            }
            mma_commit(&sh.drain);
            (void)mbar_wait_bounded(&sh.drain, 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int e = tid - 64;  // 0 .. 511
        const int ew = warp - 2;  // 0 .. 15
        const int quarter = warp & 3;
        const int h = (ew >> 2) & 1;            // key tile of the pair this warp drains
        const int c_base = (ew >> 3) * (NM / 2);  // first of the NM / 2 columns it drains
        for (int j = e; j < NM; j += kWide2Epi) {
            // padding columns: -1 (never admitted); no sample threshold: every key
            uint32_t thr = 0xFFFFFFFFu;
            if (j < nqv) {
                thr = 0x7FFFFFFFu;
                if (a.s_sample != nullptr) {
                    const float s_r = a.s_sample[(int64_t)(q0 + j) * a.r + a.thr_rank - 1];
                    if (s_r > -INFINITY) thr = __float_as_uint(-s_r);
                }
            }
            sh.thr[j] = thr;
            // the pass that admits every key fills whole lists (positions = rows)
            if (a.s_sample == nullptr && part == 0 && j < nqv) a.cnt[q0 + j] = (int32_t)a.N;
        }
        for (int j = e; j < NM; j += kWide2Epi) sh.qn[j] = j < nqv ? a.qn[q0 + j] : 0.f;
        named_barrier(2, kWide2Epi);
        // this warp's reservation entries, indexed by the absolute column
        int2* resv = sh.resv + ew * (NM / 2) - c_base;
        uint32_t* stage = &sh.stage[ew][0][0];
        wide_reserve(resv, c_base, c_base + NM / 2, nqv, lane, a, q0);

        const int64_t ks = a.key_stride;
        const uint32_t tbase =
            tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(h * NM + c_base);
        for (int j = 0; j < npairs; ++j) {
            const int64_t row = lo + (int64_t)j * kPairKeys + h * kTileM + 32 * quarter + lane;
            const float kn = row < hi ? __ldg(a.knorm + row * ks) : 0.f;
            const bool valid = row < hi && !key_masked(a.key_mask, row * ks);
            const int64_t pos = row < hi ? row : -1;
            wait_or_abort_w(&sh.acc_full[0], (uint32_t)j & 1u, &sh.abort, a.status);
            tc_fence_after();
            wide_drain_row<NM, NM / 2, false>(tbase, c_base, &sh.acc_empty[0], nqv, kn, valid,
                                       (uint32_t)(row * ks), pos, lane, sh, resv, stage, a, q0);
        }
        wide_release(resv, c_base, c_base + NM / 2, nqv, lane, a, q0);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kCols);
    }
    if (tid == 0 && *reinterpret_cast<volatile int*>(&sh.abort)) {
        const int issued = *reinterpret_cast<volatile int*>(&sh.issued);
        for (int s = max(0, issued - a.stages); s < issued; ++s)
            (void)mbar_wait_bounded(&sh.full[s % a.stages], (uint32_t)(s / a.stages) & 1u);
    }
}

// Groups of 256 or 512 queries on CTA pairs (a cluster of two CTAs on one
// TPC): tcgen05.mma.cta_group::2 with M = 256 keys (128 in each CTA's shared
// memory and TMEM lanes), N = 256 queries (each CTA stages 128 of them; the
// MMA reads both halves) and K = 16.  Each CTA's TMEM holds two 256-column
// accumulators, filled in one of two ways:
//   MT = 2  groups of 256 queries, two 256-key tiles per stage;
//   MT = 1  groups of 512 queries, one 256-key tile per stage against both
//           256-query halves, so a batch of up to 512 queries reads every key
//           from DRAM once instead of once per group of 256.
// Either way a stage is 48 KiB per CTA (three 16 KiB blocks of 128 x 64 bf16:
// key rows, then query rows), where the single-CTA two-tile kernel above
// stages 64 KiB for the same MMA work per SM: the pair reads fewer query
// bytes from L2 per key byte, and four stages fit where three did, so the
// ring covers a third more latency.  The accumulators fill TMEM, so, as in
// the two-tile kernel, a step's epilogue runs between its last MMA and the
// next step's first.
//   * both CTAs' TMA loads complete on the even CTA's full barrier, which the
//     even CTA arms with the pair's bytes; the even CTA's MMA thread issues
//     for the pair and its commits arrive on both CTAs' empty and acc_full
//     barriers;
//   * both CTAs' sixteen epilogue warps hand the accumulators back on the
//     even CTA's acc_empty barrier;
//   * neither CTA leaves before the other (cluster barrier); a CTA whose wait
//     gave up pauses first, so that copies in flight land.
// Key tiles are loaded without an L2 eviction hint: the pairs of different
// query groups do not keep a fixed order over the same keys, so marking the
// last group's loads evict-first let lines leave L2 before the other group
// read them.
constexpr int kPairStageBytes = 3 * kABytes;  // key and query blocks of 128 x 64 per CTA

template <int MT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kWide2Threads, 1)
    tc_wide_pair_kernel(const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmQ, const WideArgs a)
{
    static_assert(MT == 1 || MT == 2, "one or two 256-key tiles per stage");
    constexpr int NG = 2 / MT;               // 256-query halves of the group
    constexpr int NM = 256 * NG;             // queries of the group
    constexpr int kUnitKeys = 2 * kTileM * MT;  // keys per pair and step
    constexpr uint32_t kCols = 512;

    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    unsigned char* stages = smem;
    WideShared<NM>& sh =
        *reinterpret_cast<WideShared<NM>*>(smem + (size_t)a.stages * kPairStageBytes);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_ctarank();
    const int cid = blockIdx.x >> 1;  // the pair
    const int part = cid / a.groups, group = cid - part * a.groups;
    const int q0 = group * NM;
    const int nqv = min(NM, a.B - q0);

    const int64_t units = (a.N + kUnitKeys - 1) / kUnitKeys;
    const int64_t t0 = units * part / a.parts, t1 = units * (part + 1) / a.parts;
    const int64_t lo = t0 * kUnitKeys;
    const int64_t hi = min(a.N, t1 * kUnitKeys);
    const int nunits = (int)(t1 - t0);
    const int kc = a.kchunks;
    const int nsteps = nunits * kc;

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        mbar_init(&sh.acc_full[0], 1);
        mbar_init(&sh.acc_empty[0], 2 * kWide2Epi);  // both CTAs' epilogue threads
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        sh.issued = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc_pair(&sh.tmem_base, kCols);
    tc_fence_before();
    __syncthreads();
    // both CTAs' barriers exist before either signals the other's
    cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ producer (both CTAs)
        if (lane == 0 && nsteps > 0) {
            const uint32_t full_base = mapa_shared(&sh.full[0], 0);
            int slot = 0;
            uint32_t phase = 0;
            for (int s = 0; s < nsteps; ++s) {
                const int t = s / kc, c = s - t * kc;
                if (s >= a.stages) {
                    wait_or_abort_w(&sh.empty[slot], phase ^ 1u, &sh.abort, a.status);
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                }
                unsigned char* st = stages + (size_t)slot * kPairStageBytes;
                const uint32_t full0 = full_base + (uint32_t)(slot * sizeof(uint64_t));
                if (rank == 0) mbar_arrive_expect_tx(&sh.full[slot], 2 * kPairStageBytes);
                // key tile tt of the step is keys [base + 256 tt, base + 256 tt + 256)
                // and query half g is queries [q0 + 256 g, q0 + 256 g + 256); this
                // CTA holds rows 128 rank .. 128 rank + 127 of each
                const int32_t y = (int32_t)(lo + (int64_t)t * kUnitKeys + kTileM * (int)rank);
#pragma unroll
                for (int tt = 0; tt < MT; ++tt)
                    tma_load_2d_pair(st + tt * kABytes, &tmK, c * kChunkK, y + 2 * kTileM * tt,
                                     full0);
#pragma unroll
                for (int g = 0; g < NG; ++g)
                    tma_load_2d_pair(st + (MT + g) * kABytes, &tmQ, c * kChunkK,
                                     q0 + 2 * kTileM * g + kTileM * (int)rank, full0);
                *reinterpret_cast<volatile int*>(&sh.issued) = s + 1;
                if (++slot == a.stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (even CTA)
        if (rank == 0 && lane == 0 && nsteps > 0) {
            constexpr uint32_t idesc = mma_idesc_bf16(2 * kTileM, 256);
            int slot = 0;
            uint32_t phase = 0;
            for (int j = 0; j < nunits; ++j) {
                if (j >= 1)
                    wait_or_abort_w(&sh.acc_empty[0], (uint32_t)(j - 1) & 1u, &sh.abort, a.status);
                tc_fence_after();
                for (int c = 0; c < kc; ++c) {
                    wait_or_abort_w(&sh.full[slot], phase, &sh.abort, a.status);
                    tc_fence_after();
                    const unsigned char* st = stages + (size_t)slot * kPairStageBytes;
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k) {
                        // accumulator tt * NG + g: key tile tt against query half g
#pragma unroll
                        for (int tt = 0; tt < MT; ++tt)
#pragma unroll
                            for (int g = 0; g < NG; ++g)
                                mma_bf16_pair(tmem + (uint32_t)(256 * (tt * NG + g)),
                                              smem_desc_sw128(st + tt * kABytes) + 2u * k,
                                              smem_desc_sw128(st + (MT + g) * kABytes) + 2u * k,
                                              idesc, (c | k) != 0);
                    }
                    mma_commit_pair_both(&sh.empty[slot]);
                    if (++slot == a.stages) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                mma_commit_pair_both(&sh.acc_full[0]);
            }
            // every MMA above has completed once this arrives
            mma_commit_pair_local(&sh.drain);
            (void)mbar_wait_bounded(&sh.drain, 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (both CTAs)
        const int e = tid - 64;  // 0 .. 511
        const int ew = warp - 2;  // 0 .. 15
        const int quarter = warp & 3;
        const int acc = (ew >> 2) & 1;            // accumulator this warp drains
        const int tt = MT == 2 ? acc : 0;         // its key tile
        const int g = MT == 2 ? 0 : acc;          // its query half
        const int c_base = (ew >> 3) * 128;       // first of its 128 columns in the accumulator
        const int col0 = 256 * g + c_base;        // ... as a query of the group
        for (int j = e; j < NM; j += kWide2Epi) {
            // padding columns: -1 (never admitted); no sample threshold: every key
            uint32_t thr = 0xFFFFFFFFu;
            if (j < nqv) {
                thr = 0x7FFFFFFFu;
                if (a.s_sample != nullptr) {
                    const float s_r = a.s_sample[(int64_t)(q0 + j) * a.r + a.thr_rank - 1];
                    if (s_r > -INFINITY) thr = __float_as_uint(-s_r);
                }
            }
            sh.thr[j] = thr;
            // the pass that admits every key fills whole lists (positions = rows)
            if (a.s_sample == nullptr && part == 0 && rank == 0 && j < nqv)
                a.cnt[q0 + j] = (int32_t)a.N;
            sh.qn[j] = j < nqv ? a.qn[q0 + j] : 0.f;
        }
        named_barrier(2, kWide2Epi);
        // this warp's reservation entries, indexed by the query of the group
        int2* resv = sh.resv + ew * 128 - col0;
        uint32_t* stage = &sh.stage[ew][0][0];
        wide_reserve(resv, col0, col0 + 128, nqv, lane, a, q0);

        const int64_t ks = a.key_stride;
        const uint32_t tbase =
            tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(256 * acc + c_base);
        const uint32_t release = mapa_shared(&sh.acc_empty[0], 0);
        const int row_off = 2 * kTileM * tt + kTileM * (int)rank + 32 * quarter + lane;
        for (int j = 0; j < nunits; ++j) {
            const int64_t row = lo + (int64_t)j * kUnitKeys + row_off;
            const float kn = row < hi ? __ldg(a.knorm + row * ks) : 0.f;
            const bool valid = row < hi && !key_masked(a.key_mask, row * ks);
            const int64_t pos = row < hi ? row : -1;
            wait_or_abort_w(&sh.acc_full[0], (uint32_t)j & 1u, &sh.abort, a.status);
            tc_fence_after();
            wide_drain_row<NM, 128, false, true>(tbase, col0, nullptr, nqv, kn, valid,
                                                 (uint32_t)(row * ks), pos, lane, sh, resv, stage,
                                                 a, q0, release);
        }
        wide_release(resv, col0, col0 + 128, nqv, lane, a, q0);
    }

    tc_fence_before();
    __syncthreads();
    if (*reinterpret_cast<volatile int*>(&sh.abort)) {
        // a wait gave up: let this CTA's copies in flight land before leaving
        if (tid == 0) {
            const uint64_t t_0 = global_timer_ns();
            while (global_timer_ns() - t_0 < 10000000ull) {
            }
        }
        __syncthreads();
    }
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, kCols);
    }
}

// ---------------------------------------------------------------- query norms
// ||q||^2 of each bf16 query row, one warp per row: lane l sums the squares
// of 16-byte chunks l, l + 32, ... in order, then the warp adds the lanes'
// sums by a butterfly.  Both passes of a search read the same values.
__global__ void __launch_bounds__(256) wide_qnorm_kernel(const unsigned char* q, int32_t B,
                                                         int32_t d, float* qn)
{
    grid_dependency_wait();
    grid_dependents_launch();
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (j >= B) return;
    const unsigned char* row = q + (size_t)j * d * 2;
    const int chunks = d / 8;  // 16-byte chunks of a row (d * 2 is a multiple of 16)
    float s = 0.f;
    for (int c = lane; c < chunks; c += 32) {
        const uint4 v = ld_global_nc_v4(row + (size_t)c * 16);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float lo = __uint_as_float(w[i] << 16);
            const float hi = __uint_as_float(w[i] & 0xffff0000u);
            s = fmaf(lo, lo, s);
            s = fmaf(hi, hi, s);
        }
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) s += __shfl_xor_sync(~0u, s, o);
    if (lane == 0) qn[j] = s;
}

// ---------------------------------------------------------------- exact top-r of each global list
// One CTA per query.  Three streaming passes over the query's list (eight
// loads in flight per thread) replace a radix select in global memory:
//   1. the number of real words (reserved slots never written hold
//      kNoCandidate) and the least and greatest distance halves;
//   2. a 2048-bin histogram of the 11 bits below the leading bits all real
//      words share, which locates the bin b* holding the r-th smallest;
//   3. every real word of a bin <= b* is copied to shared memory.
// The bins order the words (same leading bits), so the copied words hold the
// r smallest; the exact select and the sort then run in shared memory.  A
// list with few real words is copied whole; if the bins up to b* hold more
// words than shared memory takes, the radix select runs on the list in place.
constexpr int kGselBins = 2048;
constexpr int kGselUnroll = 8;

struct GselShared {
    int cnt;
    uint64_t thr;
    uint32_t hmin, hmax;
    int nreal, take, bstar, upto;
    int wsum[kSelThreads / 32];
    uint32_t hist[kGselBins];
    SelectSmem<kSelThreads, 1> sel;
};

// Copies the real words of list[0, n) that `keep` accepts into stage[]
// (order not kept; the caller sorts).  Returns after a barrier.  The loop
// runs while the warp's first element is in range, so all 32 lanes make the
// same number of trips and meet at every ballot and shuffle inside it (a
// lane leaving early for the closing barrier would leave the others waiting
// at the ballot forever).
template <class Keep>
__device__ __forceinline__ void gsel_copy(const uint64_t* list, int n, uint64_t* stage,
                                          GselShared& sh, int tid, Keep keep)
{
    const int lane = tid & 31;
    for (int wbase = tid - lane; wbase < n; wbase += kGselUnroll * kSelThreads) {
        uint64_t v[kGselUnroll];
#pragma unroll
        for (int u = 0; u < kGselUnroll; ++u) {
            const int j = wbase + lane + u * kSelThreads;
            v[u] = j < n ? list[j] : kNoCandidate;
        }
#pragma unroll
        for (int u = 0; u < kGselUnroll; ++u) {
            const bool k = v[u] != kNoCandidate && keep(v[u]);
            const uint32_t bal = __ballot_sync(~0u, k);
            if (bal == 0) continue;
            int at = 0;
            if (lane == __ffs(bal) - 1) at = atomicAdd(&sh.take, __popc(bal));
            at = __shfl_sync(~0u, at, __ffs(bal) - 1);
            if (k) stage[at + __popc(bal & lanemask_lt())] = v[u];
        }
    }
    __syncthreads();
}

__global__ void __launch_bounds__(kSelThreads, 1) gselect_kernel(const GselectArgs a)
{
    extern __shared__ __align__(16) uint64_t stage[];  // a.stage_words words
    __shared__ GselShared sh;
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int q = blockIdx.x;
    uint64_t* list = a.cand + (int64_t)q * a.cap;
    // slots taken, which keep counting past the capacity when a list overflows
    const uint32_t c = (uint32_t)a.cnt[q];
    const bool overflowed = c > (uint64_t)a.cap;
    const int n = overflowed ? (int)a.cap : (int)c;
    if (a.lim_out != nullptr && !overflowed) {
        // Recovery preparation of a list within its capacity: complete,
        // unless it holds fewer than r real words after the optimistic
        // threshold (then every key up to the sample's r-th distance, a safe
        // bound, is scanned again).
        bool under = false;
        if (a.check_underflow) {
            if (threadIdx.x == 0) sh.nreal = 0;
            __syncthreads();
            int real = 0;
            for (int j = threadIdx.x; j < n; j += kSelThreads) real += list[j] != kNoCandidate;
            real = __reduce_add_sync(~0u, real);
            if ((threadIdx.x & 31) == 0) atomicAdd(&sh.nreal, real);
            __syncthreads();
            under = sh.nreal < a.r;
        }
        if (threadIdx.x == 0) {
            uint64_t lim = kNoCandidate;
            if (under) {
                const float s_r = a.s_sample[(int64_t)q * a.r + a.r - 1];
                lim = s_r > -INFINITY ? (((uint64_t)__float_as_uint(-s_r) << 32) | 0xFFFFFFFFull)
                                      : kNoCandidate - 1;  // fewer than r sampled keys: all
                a.cnt[q] = 0;
                a.group_flag[q / a.group_size] = 1;
            }
            a.lim_out[q] = lim;
        }
        return;
    }
    if (a.words_out != nullptr && overflowed && threadIdx.x == 0)
        record_status(a.status, NEST_ERR_OVERFLOW);  // recovery did not bring it under the capacity
    if (tid == 0) {
        sh.hmin = ~0u;
        sh.hmax = 0;
        sh.nreal = 0;
        sh.take = 0;
        sh.thr = kNoCandidate;
    }
    for (int i = tid; i < kGselBins; i += kSelThreads) sh.hist[i] = 0;
    __syncthreads();

    // 1. real words and the range of their distance halves
    {
        uint32_t lo = ~0u, hi = 0, cnt = 0;
        for (int base = tid; base < n; base += kGselUnroll * kSelThreads) {
            uint64_t v[kGselUnroll];
#pragma unroll
            for (int u = 0; u < kGselUnroll; ++u) {
                const int j = base + u * kSelThreads;
                v[u] = j < n ? list[j] : kNoCandidate;
            }
#pragma unroll
            for (int u = 0; u < kGselUnroll; ++u) {
                if (v[u] == kNoCandidate) continue;
                const uint32_t h = (uint32_t)(v[u] >> 32);
                lo = h < lo ? h : lo;
                hi = h > hi ? h : hi;
                ++cnt;
            }
        }
        lo = __reduce_min_sync(~0u, lo);
        hi = __reduce_max_sync(~0u, hi);
        cnt = __reduce_add_sync(~0u, cnt);
        if (lane == 0) {
            atomicMin(&sh.hmin, lo);
            atomicMax(&sh.hmax, hi);
            atomicAdd(&sh.nreal, (int)cnt);
        }
    }
    __syncthreads();
    const int nreal = sh.nreal;
    int m = -1;  // words staged in shared memory; -1: select in place
    if (nreal <= a.stage_words && nreal <= 4 * a.r) {
        gsel_copy(list, n, stage, sh, tid, [](uint64_t) { return true; });
        m = sh.take;
    } else {
        const uint32_t x = sh.hmin ^ sh.hmax;
        const int L = x ? __clz(x) : 32;  // leading bits all real words share
        const int shift = 53 - L;          // the 11 bits below them
        // 2. histogram
        for (int base = tid; base < n; base += kGselUnroll * kSelThreads) {
            uint64_t v[kGselUnroll];
#pragma unroll
            for (int u = 0; u < kGselUnroll; ++u) {
                const int j = base + u * kSelThreads;
                v[u] = j < n ? list[j] : kNoCandidate;
            }
#pragma unroll
            for (int u = 0; u < kGselUnroll; ++u)
                if (v[u] != kNoCandidate)
                    atomicAdd(&sh.hist[(uint32_t)(v[u] >> shift) & (kGselBins - 1)], 1u);
        }
        __syncthreads();
        // the bin holding the r-th smallest (thread t: bins 2t, 2t + 1)
        const uint32_t h0 = sh.hist[2 * tid], h1 = sh.hist[2 * tid + 1];
        uint32_t incl = h0 + h1;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(~0u, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) sh.wsum[warp] = (int)incl;
        __syncthreads();
        uint32_t carry = 0;
        for (int w = 0; w < warp; ++w) carry += (uint32_t)sh.wsum[w];
        const uint32_t excl = carry + incl - (h0 + h1);
        const uint32_t r = (uint32_t)a.r;
        if (excl < r && r <= excl + h0 + h1) {
            const bool first = excl + h0 >= r;
            sh.bstar = first ? 2 * tid : 2 * tid + 1;
            sh.upto = (int)(first ? excl + h0 : excl + h0 + h1);
        }
        __syncthreads();
        if (sh.upto <= a.stage_words) {
            // 3. the real words of bins <= b*
            const uint32_t bstar = (uint32_t)sh.bstar;
            gsel_copy(list, n, stage, sh, tid, [shift, bstar](uint64_t e) {
                return ((uint32_t)(e >> shift) & (kGselBins - 1)) <= bstar;
            });
            m = sh.take;
        }
    }

    int nsel;
    if (m >= 0) {
        if (tid == 0) sh.cnt = m;
        __syncthreads();
        select_smallest<kSelThreads, 1>(stage, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid,
                                        [] { __syncthreads(); });
        nsel = sh.cnt;
    } else {
        // keeps the r smallest at the front of the list, in place
        if (tid == 0) sh.cnt = n;
        __syncthreads();
        select_smallest<kSelThreads, 1>(list, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid,
                                        [] { __syncthreads(); });
        nsel = sh.cnt;
    }
    // The select leaves at most r words because the words of a list are
    // distinct (each carries its key index).  More would mean a list held
    // repeated words: recorded, and no more than r are used, so that nothing
    // is written past the r words the stage and the outputs hold.
    if (nsel > a.r) {
        if (tid == 0 && a.status != nullptr) record_status(a.status, NEST_ERR_OVERFLOW);
        nsel = a.r;
    }
    if (m < 0)
        for (int j = tid; j < nsel; j += kSelThreads) stage[j] = list[j];
    if (a.lim_out != nullptr) {
        // Recovery preparation of an overflowed list: the r-th smallest of
        // the words it holds bounds the r-th smallest of all keys from
        // above, so a pass admitting every word up to it misses none of the
        // r nearest.  The list starts over; its group is flagged.
        __shared__ unsigned long long lim;
        if (tid == 0) lim = 0;
        __syncthreads();
        for (int j = tid; j < nsel; j += kSelThreads)
            if (stage[j] != kNoCandidate) atomicMax(&lim, (unsigned long long)stage[j]);
        __syncthreads();
        if (tid == 0) {
            a.lim_out[q] = lim;
            a.cnt[q] = 0;
            a.group_flag[q / a.group_size] = 1;
        }
        return;
    }
    if (a.words_out != nullptr) {
        // the r smallest words, unsorted, for the exact re-ranking
        uint64_t* wo = a.words_out + (int64_t)q * a.r;
        for (int j = tid; j < a.r; j += kSelThreads) wo[j] = j < nsel ? stage[j] : kNoCandidate;
        if (tid == 0) {
            a.words_cnt[q] = nsel;
            refine_state_reset(a.refine_state, a.refine_apair, a.B, q);
        }
        return;
    }
    int P2 = 1;
    while (P2 < (nsel > 0 ? nsel : 1)) P2 <<= 1;
    for (int j = nsel + tid; j < P2; j += kSelThreads) stage[j] = kNoCandidate;
    __syncthreads();
    bitonic_sort<kSelThreads>(stage, P2, tid, [] { __syncthreads(); });
    float* so = a.s_out + (int64_t)q * a.r;
    int64_t* io = a.idx_out + (int64_t)q * a.r;
    for (int j = tid; j < a.r; j += kSelThreads) {
        const uint64_t e = j < nsel ? stage[j] : kNoCandidate;
        if (e != kNoCandidate) {  // reserved slots never written hold kNoCandidate
            so[j] = -__uint_as_float((uint32_t)(e >> 32));
            io[j] = (int64_t)(uint32_t)e;
        } else {
            so[j] = -INFINITY;
            io[j] = -1;
        }
    }
}

template <int NM>
size_t wide_fixed()
{
    return 1024 + sizeof(WideShared<NM>);
}

template <int NM>
bool wide_plan_nm(size_t smem_limit, bool pairs, WidePlan* p)
{
    const size_t fixed = wide_fixed<NM>();
    p->pair = false;
    if (NM >= 256 && pairs && fixed + 4 * (size_t)kPairStageBytes <= smem_limit) {
        // CTA pairs: 48 KiB stages per CTA; groups of 256 take two 256-key
        // tiles per step, groups of 512 one
        int stages = (int)((smem_limit - fixed) / kPairStageBytes);
        stages = stages > kMaxStagesW ? kMaxStagesW : stages;
        p->nm = NM;
        p->mb = NM == 256 ? 4 : 2;
        p->pair = true;
        p->stages = stages;
        p->smem = fixed + (size_t)stages * kPairStageBytes;
        return true;
    }
    if (NM > 256) return false;  // groups of 512 run on pairs only
    if (NM == 256) {
        // two key tiles per stage when three 64 KiB stages fit
        const size_t st2 = (size_t)(2 * kABytes + NM * kChunkK * 2);
        if (fixed + 3 * st2 <= smem_limit) {
            int stages = (int)((smem_limit - fixed) / st2);
            stages = stages > kMaxStagesW ? kMaxStagesW : stages;
            p->nm = NM;
            p->mb = 2;
            p->stages = stages;
            p->smem = fixed + (size_t)stages * st2;
            return true;
        }
    }
    const size_t st = (size_t)stage_bytes<NM>();
    if (fixed + 3 * st > smem_limit) return false;
    int stages = (int)((smem_limit - fixed) / st);
    stages = stages > kMaxStagesW ? kMaxStagesW : stages;
    p->nm = NM;
    p->mb = 1;
    p->stages = stages;
    p->smem = fixed + (size_t)stages * st;
    return true;
}

template <int NM>
cudaError_t wide_launch_nm(const WidePlan& p, const CUtensorMap& tmK, const CUtensorMap& tmQ,
                           const WideArgs& a, cudaStream_t stream)
{
    if constexpr (NM >= 256) {
        if (p.pair) {
            auto kern = tc_wide_pair_kernel<NM == 256 ? 2 : 1>;
            cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
            if (e != cudaSuccess) return e;
            kern<<<2 * p.groups * p.parts, kWide2Threads, p.smem, stream>>>(tmK, tmQ, a);
            return cudaGetLastError();
        }
    }
    if constexpr (NM > 256) {
        return cudaErrorInvalidValue;  // groups of 512 run on pairs only
    } else {
        if (NM == 256 && p.mb == 2) {
            cudaError_t e =
                raise_smem_limit(reinterpret_cast<const void*>(tc_wide2_kernel), (int)p.smem);
            if (e != cudaSuccess) return e;
            return launch_pdl(tc_wide2_kernel, dim3(p.groups * p.parts), dim3(kWide2Threads),
                              p.smem, stream, tmK, tmQ, a);
        }
        auto kern = tc_wide_kernel<NM>;
        cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
        if (e != cudaSuccess) return e;
        return launch_pdl(kern, dim3(p.groups * p.parts), dim3(kTcThreads), p.smem, stream, tmK,
                          tmQ, a);
    }
}

}  // namespace

bool wide_plan_smem(int nm, size_t smem_limit, bool pairs, WidePlan* p)
{
    switch (nm) {
    case 16: return wide_plan_nm<16>(smem_limit, pairs, p);
    case 32: return wide_plan_nm<32>(smem_limit, pairs, p);
    case 64: return wide_plan_nm<64>(smem_limit, pairs, p);
    case 128: return wide_plan_nm<128>(smem_limit, pairs, p);
    case 256: return wide_plan_nm<256>(smem_limit, pairs, p);
    case 512: return wide_plan_nm<512>(smem_limit, pairs, p);
    default: return false;
    }
}

namespace {

// Clusters of the pair kernel for groups of NM queries that the device can
// hold at once (0: none, or the plan does not fit).
template <int NM>
int pair_clusters_nm(size_t smem_limit)
{
    WidePlan p{};
    if (!wide_plan_nm<NM>(smem_limit, true, &p) || !p.pair) return 0;
    auto kern = tc_wide_pair_kernel<NM == 256 ? 2 : 1>;
    if (raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem) != cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2, 1, 1);
    cfg.blockDim = dim3(kWide2Threads, 1, 1);
    cfg.dynamicSmemBytes = p.smem;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kern), &cfg) !=
        cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    return n;
}

}  // namespace

int wide_pair_clusters(size_t smem_limit)
{
    const int a = pair_clusters_nm<256>(smem_limit);
    const int b = pair_clusters_nm<512>(smem_limit);
    return a < b ? a : b;
}

namespace {

template <int NM>
bool wide_recover_plan_nm(size_t smem_limit, WidePlan* p)
{
    const size_t fixed = wide_fixed<NM>();
    const size_t st = (size_t)stage_bytes<NM>();
    if (fixed + 3 * st > smem_limit) return false;
    int stages = (int)((smem_limit - fixed) / st);
    stages = stages > kMaxStagesW ? kMaxStagesW : stages;
    p->nm = NM;
    p->mb = 1;
    p->pair = false;
    p->stages = stages;
    p->smem = fixed + (size_t)stages * st;
    return true;
}

template <int NM>
cudaError_t recover_launch_nm(const WidePlan& p, const CUtensorMap& tmK, const CUtensorMap& tmQ,
                              const WideArgs& a, cudaStream_t stream)
{
    auto kern = tc_wide_kernel<NM, true>;
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(p.groups * p.parts), dim3(kTcThreads), p.smem, stream, tmK, tmQ,
                      a);
}

}  // namespace

bool wide_recover_plan(int nm, size_t smem_limit, WidePlan* p)
{
    switch (nm) {
    case 16: return wide_recover_plan_nm<16>(smem_limit, p);
    case 32: return wide_recover_plan_nm<32>(smem_limit, p);
    case 64: return wide_recover_plan_nm<64>(smem_limit, p);
    case 128: return wide_recover_plan_nm<128>(smem_limit, p);
    case 256: return wide_recover_plan_nm<256>(smem_limit, p);
    default: return false;
    }
}

cudaError_t launch_tc_wide_recover(const WidePlan& p, const CUtensorMap& tmK,
                                   const CUtensorMap& tmQ, const WideArgs& a, cudaStream_t stream)
{
    switch (p.nm) {
    case 16: return recover_launch_nm<16>(p, tmK, tmQ, a, stream);
    case 32: return recover_launch_nm<32>(p, tmK, tmQ, a, stream);
    case 64: return recover_launch_nm<64>(p, tmK, tmQ, a, stream);
    case 128: return recover_launch_nm<128>(p, tmK, tmQ, a, stream);
    case 256: return recover_launch_nm<256>(p, tmK, tmQ, a, stream);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_tc_wide(const WidePlan& p, const CUtensorMap& tmK, const CUtensorMap& tmQ,
                           const WideArgs& a, cudaStream_t stream)
{
    switch (p.nm) {
    case 16: return wide_launch_nm<16>(p, tmK, tmQ, a, stream);
    case 32: return wide_launch_nm<32>(p, tmK, tmQ, a, stream);
    case 64: return wide_launch_nm<64>(p, tmK, tmQ, a, stream);
    case 128: return wide_launch_nm<128>(p, tmK, tmQ, a, stream);
    case 256: return wide_launch_nm<256>(p, tmK, tmQ, a, stream);
    case 512: return wide_launch_nm<512>(p, tmK, tmQ, a, stream);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_wide_qnorm(const void* q, int32_t B, int32_t d, float* qn, cudaStream_t stream)
{
    return launch_pdl(wide_qnorm_kernel, dim3((B + 7) / 8), dim3(256), 0, stream,
                      static_cast<const unsigned char*>(q), B, d, qn);
}

cudaError_t launch_gselect(const GselectArgs& in, cudaStream_t stream)
{
    GselectArgs a = in;
    int P2 = 1;
    while (P2 < a.r) P2 <<= 1;
    a.stage_words = P2 > 16384 ? P2 : 16384;  // at least next_pow2(r): the sort runs there
    const size_t smem = (size_t)a.stage_words * sizeof(uint64_t);
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(gselect_kernel), (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(gselect_kernel, dim3(a.B), dim3(kSelThreads), smem, stream, a);
}

}  // namespace nest
