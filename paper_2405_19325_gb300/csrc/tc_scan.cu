// tc_scan.cu -- tensor-core distance scan with fused per-CTA top-r for bf16
// datastores (the search of Sec. 2.2 / Sec. 3.1: s(q, k) = -||q - k||^2,
// r nearest), on tcgen05 with TMEM accumulators and TMA tensor copies.
//
// The dot products q.k of a group of up to 16 queries against 128-key tiles
// are a small dense contraction (keys as M = 128, queries as N = 16, d as K):
//
//   producer warp   TMA-loads, per stage, a 128 x 64 key tile and the
//                   16 x 64 query tile of the same columns (128-byte
//                   swizzle, L2 evict-first for keys) into a ring of stages;
//   MMA warp        one thread issues 4 x tcgen05.mma (K = 16 each) per stage
//                   into one of two TMEM accumulators (128 lanes x 16 fp32
//                   columns), frees the stage with tcgen05.commit, and hands
//                   a finished tile to the epilogue with another commit;
//   4 epilogue warps read their 32 TMEM lanes (one key per thread), form
//                   ||q||^2 + ||k||^2 - 2 q.k, append candidates that can
//                   still enter each query's r nearest to shared-memory
//                   lists, and trim the lists with the radix select when
//                   they fill.
//
// The output is the same per-CTA candidate lists as scan.cu, merged by
// merge.cu.  The arithmetic of the scan costs a handful of instructions per
// 16 KiB of keys, so the kernel runs at the speed of the key stream.
#include <cuda.h>

#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kTileM = 128;                     // keys per tile (TMEM lanes)
constexpr int kMmaN = 16;                       // query columns per MMA
constexpr int kChunkK = 64;                     // bf16 columns per stage (128 bytes)
constexpr int kABytes = kTileM * kChunkK * 2;   // 16 KiB of keys
constexpr int kBBytes = kMmaN * kChunkK * 2;    // 2 KiB of queries
constexpr int kStageBytes = kABytes + kBBytes;  // multiple of 1024: stages stay swizzle-aligned
constexpr int kMaxStagesTc = 12;
constexpr int kEpiThreads = 128;
constexpr int kBarEpi = 2;  // hardware barrier of the epilogue warps
constexpr uint32_t kTmemCols = 32;  // two accumulators of 16 columns

static_assert(kTcThreads == 64 + kEpiThreads, "producer, MMA and four epilogue warps");
static_assert(kStageBytes % 1024 == 0, "stage must keep 1024-byte alignment");

template <int NQ>
struct TcShared {
    uint64_t full[kMaxStagesTc];
    uint64_t empty[kMaxStagesTc];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint64_t thr[NQ];
    int cnt[NQ];
    float qn_part[4][NQ];
    uint32_t tmem_base;
    int abort;
    int issued;
    SelectSmem<kEpiThreads, NQ> sel;
};

__device__ __forceinline__ void wait_or_abort_tc(uint64_t* bar, uint32_t parity, int* abort_flag,
                                                 int* status)
{
    if (*reinterpret_cast<volatile int*>(abort_flag)) return;
    if (!mbar_wait_bounded(bar, parity)) {
        record_status(status, NEST_ERR_TIMEOUT);
        *reinterpret_cast<volatile int*>(abort_flag) = 1;
    }
}

template <int NQ>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_scan_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ,
                   const TcScanArgs a)
{
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    unsigned char* stages = smem;
    uint64_t* cand = reinterpret_cast<uint64_t*>(smem + (size_t)a.stages * kStageBytes);
    TcShared<NQ>& sh = *reinterpret_cast<TcShared<NQ>*>(cand + (size_t)NQ * a.cap);

    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int item = blockIdx.x;
    const int group = item / a.parts, part = item - group * a.parts;

    // ---- queries and key rows [lo, hi) of this CTA, in whole 128-key tiles
    int64_t base = 0, len = 0;
    int q0, nqv;
    if (a.seg_off != nullptr) {
        q0 = group;
        nqv = 1;
        const int64_t so = a.seg_off[group], eo = a.seg_off[group + 1];
        if (so < 0 || eo < so || eo > a.N) {
            if (tid == 0 && part == 0) record_status(a.status, NEST_ERR_INVALID_ARG);
        } else {
            base = so;
            len = eo - so;
        }
    } else {
        q0 = group * NQ;
        nqv = min(NQ, a.B - q0);
        len = a.N;
    }
    const int64_t tiles = (len + kTileM - 1) / kTileM;
    const int64_t t0 = tiles * part / a.parts, t1 = tiles * (part + 1) / a.parts;
    const int64_t lo = base + t0 * kTileM;
    const int64_t hi = min(base + len, base + t1 * kTileM);
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
    if (warp == 1) tmem_alloc(&sh.tmem_base, kTmemCols);
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
                    wait_or_abort_tc(&sh.empty[slot], phase ^ 1u, &sh.abort, a.status);
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                }
                unsigned char* st = stages + (size_t)slot * kStageBytes;
                mbar_arrive_expect_tx(&sh.full[slot], kStageBytes);
                tma_load_2d_hint(st, &tmK, c * kChunkK, (int32_t)(lo + (int64_t)t * kTileM),
                                 &sh.full[slot], policy);
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
            constexpr uint32_t idesc = mma_idesc_bf16(kTileM, kMmaN);
            int slot = 0;
            uint32_t phase = 0;
            for (int j = 0; j < ntiles; ++j) {
                const int buf = j & 1;
                if (j >= 2)
                    wait_or_abort_tc(&sh.acc_empty[buf], (uint32_t)((j >> 1) - 1) & 1u, &sh.abort,
                                     a.status);
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * kMmaN);
                for (int c = 0; c < kc; ++c) {
                    wait_or_abort_tc(&sh.full[slot], phase, &sh.abort, a.status);
                    tc_fence_after();
                    const unsigned char* st = stages + (size_t)slot * kStageBytes;
                    const uint64_t ad = smem_desc_sw128(st);
                    const uint64_t bd = smem_desc_sw128(st + kABytes);
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k)  // 32 bytes of K per MMA
                        mma_bf16(d_tmem, ad + 2u * k, bd + 2u * k, idesc, (c | k) != 0);
                    mma_commit(&sh.empty[slot]);
                    if (++slot == a.stages) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
                mma_commit(&sh.acc_full[buf]);
            }
            // every MMA above has completed once this arrives
            mma_commit(&sh.drain);
            (void)mbar_wait_bounded(&sh.drain, 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int e = tid - 64;
        const int quarter = warp & 3;  // this warp may read TMEM lanes [32 quarter, 32 quarter + 32)
        auto bar = [] { named_barrier(kBarEpi, kEpiThreads); };
        if (e < NQ) {
            sh.cnt[e] = 0;
            sh.thr[e] = kNoCandidate;
        }
        // ||q||^2 of the group's queries, from the stored bf16 values
        float qn[NQ];
        const uint16_t* qh = static_cast<const uint16_t*>(a.q);
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            float s = 0.f;
            if (b < nqv) {
                const uint16_t* row = qh + (size_t)(q0 + b) * a.d;
                for (int j = e; j < a.d; j += kEpiThreads) {
                    const float x = __uint_as_float((uint32_t)__ldg(row + j) << 16);
                    s = fmaf(x, x, s);
                }
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) s += __shfl_xor_sync(~0u, s, o);
            if (lane == 0) sh.qn_part[warp - 2][b] = s;
        }
        bar();
#pragma unroll
        for (int b = 0; b < NQ; ++b)
            qn[b] = (sh.qn_part[0][b] + sh.qn_part[1][b]) + (sh.qn_part[2][b] + sh.qn_part[3][b]);

        const int row_in_tile = 32 * quarter + lane;
        const int64_t ks = a.key_stride;  // row i of the tensor map is key i * ks
        float kn_next =
            (ntiles > 0 && lo + row_in_tile < hi) ? __ldg(a.knorm + (lo + row_in_tile) * ks) : 0.f;
        for (int j = 0; j < ntiles; ++j) {
            const int buf = j & 1;
            const int64_t row = lo + (int64_t)j * kTileM + row_in_tile;
            const float kn = kn_next;
            kn_next = (row + kTileM < hi) ? __ldg(a.knorm + (row + kTileM) * ks) : 0.f;
            wait_or_abort_tc(&sh.acc_full[buf], (uint32_t)(j >> 1) & 1u, &sh.abort, a.status);
            tc_fence_after();
            uint32_t acc[16];
            tmem_ld_16(tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(buf * kMmaN), acc);
            tc_fence_before();
            mbar_arrive(&sh.acc_empty[buf]);
            const bool valid = row < hi && !key_masked(a.key_mask, row * ks);
#pragma unroll
            for (int b = 0; b < NQ; ++b) {
                float dist = fmaf(-2.f, __uint_as_float(acc[b]), qn[b] + kn);
                dist = (dist <= 0.f) ? 0.f : dist;  // NaN stays NaN and sorts last
                const uint64_t key = ((uint64_t)__float_as_uint(dist) << 32) | (uint32_t)(row * ks);
                const bool accept = valid && (b < nqv) && (key <= sh.thr[b]);
                const uint32_t bal = __ballot_sync(~0u, accept);
                if (bal) {
                    const int leader = __ffs(bal) - 1;
                    int at = 0;
                    if (lane == leader) at = atomicAdd(&sh.cnt[b], __popc(bal));
                    at = __shfl_sync(~0u, at, leader);
                    if (accept) cand[(size_t)b * a.cap + at + __popc(bal & lanemask_lt())] = key;
                }
            }
            bar();
            bool need = false;
#pragma unroll
            for (int b = 0; b < NQ; ++b) need |= sh.cnt[b] > a.cap - kTileM;
            bar();  // every thread has decided before any appends of the next tile
            if (need) select_smallest<kEpiThreads, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, e, bar);
        }
        bar();
        select_smallest<kEpiThreads, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, e, bar);
        uint64_t* out = a.cand + (size_t)item * NQ * a.r;
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            const int n = sh.cnt[b];
            for (int jj = e; jj < a.r; jj += kEpiThreads)
                out[(size_t)b * a.r + jj] = jj < n ? cand[(size_t)b * a.cap + jj] : kNoCandidate;
            if (e == 0) a.cand_cnt[(size_t)item * NQ + b] = n;
        }
    }

    // ---- teardown: TMEM back, copies landed
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (tid == 0 && *reinterpret_cast<volatile int*>(&sh.abort)) {
        const int issued = *reinterpret_cast<volatile int*>(&sh.issued);
        for (int s = max(0, issued - a.stages); s < issued; ++s)
            (void)mbar_wait_bounded(&sh.full[s % a.stages], (uint32_t)(s / a.stages) & 1u);
    }
}

template <int NQ>
size_t tc_fixed_smem(int cap)
{
    return 1024 /* alignment slack */ + (size_t)NQ * cap * sizeof(uint64_t) + sizeof(TcShared<NQ>);
}

template <int NQ>
cudaError_t tc_launch_nq(const TcPlan& p, const CUtensorMap& tmK, const CUtensorMap& tmQ,
                         const TcScanArgs& a, cudaStream_t stream)
{
    auto kern = tc_scan_kernel<NQ>;
    cudaError_t e =
        raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(p.groups * p.parts), dim3(kTcThreads), p.smem, stream, tmK, tmQ,
                      a);
}

}  // namespace

int tc_cap(int r) { return r + (r < 512 ? 256 : 512); }

bool tc_plan_smem(int nq, int r, size_t smem_limit, TcPlan* plan)
{
    const int cap = tc_cap(r);
    size_t fixed;
    switch (nq) {
    case 1: fixed = tc_fixed_smem<1>(cap); break;
    case 2: fixed = tc_fixed_smem<2>(cap); break;
    case 4: fixed = tc_fixed_smem<4>(cap); break;
    case 8: fixed = tc_fixed_smem<8>(cap); break;
    case 16: fixed = tc_fixed_smem<16>(cap); break;
    default: return false;
    }
    if (fixed + 4 * (size_t)kStageBytes > smem_limit) return false;
    int stages = (int)((smem_limit - fixed) / kStageBytes);
    stages = stages > kMaxStagesTc ? kMaxStagesTc : stages;
    plan->nq = nq;
    plan->cap = cap;
    plan->stages = stages;
    plan->smem = fixed + (size_t)stages * kStageBytes;
    return true;
}

cudaError_t launch_tc_scan(const TcPlan& p, const CUtensorMap& tmK, const CUtensorMap& tmQ,
                           const TcScanArgs& a, cudaStream_t stream)
{
    switch (p.nq) {
    case 1: return tc_launch_nq<1>(p, tmK, tmQ, a, stream);
    case 2: return tc_launch_nq<2>(p, tmK, tmQ, a, stream);
    case 4: return tc_launch_nq<4>(p, tmK, tmQ, a, stream);
    case 8: return tc_launch_nq<8>(p, tmK, tmQ, a, stream);
    case 16: return tc_launch_nq<16>(p, tmK, tmQ, a, stream);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace nest
