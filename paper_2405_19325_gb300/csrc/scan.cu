// scan.cu -- HBM-streaming distance scan with fused per-CTA top-r
// (the search of Sec. 2.2 / Sec. 3.1: s(q, k) = -||q - k||^2, r nearest).
//
// One CTA owns a group of up to NQ queries and a contiguous range of key
// rows (a slice of the datastore, or a slice of one query's candidate
// segment).  Three warp roles, decoupled by mbarrier rings:
//
//   producer warp   streams the rows into a ring of shared-memory stages of
//                   kScanRows rows with 1-D TMA bulk copies (L2 evict-first);
//   8 consumer warps hold the queries in registers (each thread owns fixed
//                   16-byte column chunks of every row) and compute q.k with
//                   packed fp32 FMA (two lanes of the sum per instruction);
//                   per stage a warp reduce-scatter leaves one partial dot
//                   product per (row, query) and warp in a ring of partials;
//   selector warp   adds the 8 partials, forms ||q||^2 + ||k||^2 - 2 q.k,
//                   appends every candidate that can still enter its
//                   query's r nearest to a shared-memory list, and, when a
//                   list fills up, trims it back to r with a radix select
//                   (which also tightens the admission threshold).
//
// No block-wide barrier is taken per stage: the consumers only wait for
// data and for free slots of the partial ring.  At the end the selector
// writes the CTA's r best candidates per query; merge.cu combines the CTAs.
// No distance ever goes to global memory.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kProducerWarp = kConsumerWarps;
constexpr int kSelectorWarp = kConsumerWarps + 1;
static_assert((kSelectorWarp + 1) * 32 == kScanThreads, "warp roles must fill the block");
constexpr int kBarSetup = 1;      // consumers + selector, once (query norms)
constexpr int kMaxStages = 8;
constexpr int kPartialRing = 16;  // stages of partial sums in flight (a power of two)

template <int DT>
struct Elem;
template <>
struct Elem<NEST_F32> {
    static constexpr int kPerChunk = 4;
};
template <>
struct Elem<NEST_BF16> {
    static constexpr int kPerChunk = 8;
};

// 16 bytes of a row -> fp32 pairs (element 2p, element 2p + 1); bf16 -> fp32 is exact.
template <int DT>
__device__ __forceinline__ void unpack_pairs(const uint4& v, float2* x)
{
    if constexpr (DT == NEST_BF16) {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
            x[i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xffff0000u));
    } else {
        x[0] = make_float2(__uint_as_float(v.x), __uint_as_float(v.y));
        x[1] = make_float2(__uint_as_float(v.z), __uint_as_float(v.w));
    }
}

template <int NQ>
struct ScanShared {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t pfull[kPartialRing];
    uint64_t pempty[kPartialRing];
    uint64_t thr[NQ];
    int cnt[NQ];
    float qnorm_part[kConsumerWarps][NQ];
    int abort;
    int issued;
    SelectSmem<32, NQ> sel;
};

// Warp reduce-scatter of NV values: afterwards lane l holds the warp-wide
// sum of value (l >> (5 - log2 NV)).  NV - 1 + log2(32 / NV) shuffles.
template <int NV>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[NV], int lane)
{
#pragma unroll
    for (int c = NV, o = 16; c > 1; c >>= 1, o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < c / 2; ++i) {
            const float send = upper ? v[i] : v[i + c / 2];
            const float keep = upper ? v[i + c / 2] : v[i];
            v[i] = keep + __shfl_xor_sync(~0u, send, o);
        }
    }
    float x = v[0];
#pragma unroll
    for (int o = 16 / NV; o >= 1; o >>= 1) x += __shfl_xor_sync(~0u, x, o);
    return x;
}

// Lanes l < NV with l % NQ == qb.
template <int NQ, int NV>
__device__ __forceinline__ uint32_t query_lanes(int qb)
{
    uint32_t m = 0;
#pragma unroll
    for (int l = 0; l < NV; ++l)
        if (l % NQ == qb) m |= 1u << l;
    return m;
}

// Bounded wait that records a timeout and raises the CTA's abort flag; once
// the flag is up every later wait returns at once so the CTA drains.
__device__ __forceinline__ void wait_or_abort(uint64_t* bar, uint32_t parity, int* abort_flag,
                                              int* status)
{
    if (*reinterpret_cast<volatile int*>(abort_flag)) return;
    if (!mbar_wait_bounded(bar, parity)) {
        record_status(status, NEST_ERR_TIMEOUT);
        *reinterpret_cast<volatile int*>(abort_flag) = 1;
    }
}

template <int DT, int NQ, int CPT>
__global__ void __launch_bounds__(kScanThreads, 1) scan_topr_kernel(const ScanArgs a)
{
    constexpr int EPC = Elem<DT>::kPerChunk;
    constexpr int PPC = EPC / 2;        // fp32 pairs per 16-byte chunk
    constexpr int NV = kScanRows * NQ;  // (row, query) dot products per stage
    constexpr int kLanesPerValue = 32 / NV;
    static_assert(NV <= 32 && (NV & (NV - 1)) == 0, "NV must be a power of two <= 32");

    extern __shared__ __align__(128) unsigned char smem[];
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int item = blockIdx.x;
    const int group = item / a.parts, part = item - group * a.parts;

    unsigned char* stages = smem;
    uint64_t* cand = reinterpret_cast<uint64_t*>(smem + (size_t)a.stages * a.stage_bytes);
    float* partial = reinterpret_cast<float*>(cand + (size_t)NQ * a.cap);  // [ring][warps][NV]
    ScanShared<NQ>& sh =
        *reinterpret_cast<ScanShared<NQ>*>(partial + kPartialRing * kConsumerWarps * NV);

    // ---- this CTA's queries and key rows [lo, hi)
    int64_t lo = 0, hi = 0;
    int q0, nqv;
    if (a.seg_off != nullptr) {
        q0 = group;
        nqv = 1;
        const int64_t so = a.seg_off[group], eo = a.seg_off[group + 1];
        if (so < 0 || eo < so || eo > a.N) {
            if (tid == 0 && part == 0) record_status(a.status, NEST_ERR_INVALID_ARG);
        } else {
            const int64_t len = eo - so;
            lo = so + len * part / a.parts;
            hi = so + len * (part + 1) / a.parts;
        }
    } else {
        q0 = group * NQ;
        nqv = min(NQ, a.B - q0);
        lo = a.N * part / a.parts;
        hi = a.N * (part + 1) / a.parts;
    }
    const int64_t nrows = hi - lo;
    const int nst = (int)((nrows + kScanRows - 1) / kScanRows);
    auto rows_of = [&](int i) -> int {
        const int64_t left = nrows - (int64_t)i * kScanRows;
        return (int)(left < kScanRows ? left : kScanRows);
    };

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], kConsumerWarps);
        }
        for (int s = 0; s < kPartialRing; ++s) {
            mbar_init(&sh.pfull[s], kConsumers);
            mbar_init(&sh.pempty[s], 32);
        }
        sh.abort = 0;
        sh.issued = 0;
        mbar_init_fence();
    }
    __syncthreads();

    // ---------------------------------------------------------------- producer
    if (warp == kProducerWarp) {
        if (lane == 0 && nst > 0) {
            const uint64_t policy = l2_policy_evict_first();
            const unsigned char* src = static_cast<const unsigned char*>(a.K) + lo * a.row_bytes;
            int slot = 0;
            uint32_t phase = 0;  // phase of the slot's current round
            for (int i = 0; i < nst; ++i) {
                if (i >= a.stages) {
                    wait_or_abort(&sh.empty[slot], phase ^ 1u, &sh.abort, a.status);
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                }
                const uint32_t bytes = (uint32_t)rows_of(i) * (uint32_t)a.row_bytes;
                mbar_arrive_expect_tx(&sh.full[slot], bytes);
                bulk_copy_g2s_evict_first(stages + (size_t)slot * a.stage_bytes,
                                          src + (size_t)i * kScanRows * a.row_bytes, bytes,
                                          &sh.full[slot], policy);
                *reinterpret_cast<volatile int*>(&sh.issued) = i + 1;
                if (++slot == a.stages) {
                    slot = 0;
                    phase ^= 1u;
                }
            }
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    if (warp < kConsumerWarps) {
        // Queries of the group, fixed column chunks of this thread, as fp32 pairs.
        float2 qf[CPT][NQ][PPC];
        float qn[NQ];
#pragma unroll
        for (int b = 0; b < NQ; ++b) qn[b] = 0.f;
#pragma unroll
        for (int k = 0; k < CPT; ++k) {
            const int c = tid + k * kConsumers;
#pragma unroll
            for (int b = 0; b < NQ; ++b) {
                float2 x[PPC];
                if (c < a.chunks && b < nqv) {
                    const uint4 v = ld_global_nc_v4(static_cast<const unsigned char*>(a.q) +
                                                    (size_t)(q0 + b) * a.row_bytes + (size_t)c * 16);
                    unpack_pairs<DT>(v, x);
                } else {
#pragma unroll
                    for (int p = 0; p < PPC; ++p) x[p] = make_float2(0.f, 0.f);
                }
#pragma unroll
                for (int p = 0; p < PPC; ++p) {
                    qf[k][b][p] = x[p];
                    qn[b] = fmaf(x[p].x, x[p].x, qn[b]);
                    qn[b] = fmaf(x[p].y, x[p].y, qn[b]);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) qn[b] += __shfl_xor_sync(~0u, qn[b], o);
            if (lane == 0) sh.qnorm_part[warp][b] = qn[b];
        }
        named_barrier(kBarSetup, kConsumers + 32);

        int slot = 0;
        uint32_t phase = 0;
        for (int i = 0; i < nst; ++i) {
            const int rows = rows_of(i);
            wait_or_abort(&sh.full[slot], phase, &sh.abort, a.status);
            float2 acc[kScanRows][NQ];
#pragma unroll
            for (int rr = 0; rr < kScanRows; ++rr)
#pragma unroll
                for (int b = 0; b < NQ; ++b) acc[rr][b] = make_float2(0.f, 0.f);
            const unsigned char* st = stages + (size_t)slot * a.stage_bytes;
#pragma unroll
            for (int rr = 0; rr < kScanRows; ++rr) {
                if (rr < rows) {
#pragma unroll
                    for (int k = 0; k < CPT; ++k) {
                        const int c = tid + k * kConsumers;
                        if (c < a.chunks) {
                            const uint4 v = *reinterpret_cast<const uint4*>(
                                st + (size_t)rr * a.row_bytes + (size_t)c * 16);
                            float2 x[PPC];
                            unpack_pairs<DT>(v, x);
#pragma unroll
                            for (int b = 0; b < NQ; ++b)
#pragma unroll
                                for (int p = 0; p < PPC; ++p)
                                    acc[rr][b] = __ffma2_rn(qf[k][b][p], x[p], acc[rr][b]);
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.empty[slot]);
            if (++slot == a.stages) {
                slot = 0;
                phase ^= 1u;
            }

            float v[NV];
#pragma unroll
            for (int rr = 0; rr < kScanRows; ++rr)
#pragma unroll
                for (int b = 0; b < NQ; ++b) v[rr * NQ + b] = acc[rr][b].x + acc[rr][b].y;
            const float red = warp_reduce_scatter<NV>(v, lane);
            const int ps = i & (kPartialRing - 1);
            if (i >= kPartialRing)
                wait_or_abort(&sh.pempty[ps], (uint32_t)((i / kPartialRing) - 1) & 1u, &sh.abort,
                              a.status);
            if ((lane & (kLanesPerValue - 1)) == 0)
                partial[(ps * kConsumerWarps + warp) * NV + lane / kLanesPerValue] = red;
            mbar_arrive(&sh.pfull[ps]);
        }
        return;
    }

    // ---------------------------------------------------------------- selector
    named_barrier(kBarSetup, kConsumers + 32);
    float qnorm[NQ];
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
        float t = 0.f;
        for (int w = 0; w < kConsumerWarps; ++w) t += sh.qnorm_part[w][b];
        qnorm[b] = t;
    }
    if (lane < NQ) {
        sh.cnt[lane] = 0;
        sh.thr[lane] = kNoCandidate;
    }
    __syncwarp();
    int cnt[NQ];
#pragma unroll
    for (int b = 0; b < NQ; ++b) cnt[b] = 0;

    // Key norms of a stage's rows, prefetched two stages ahead (lanes < kScanRows).
    auto load_kn = [&](int i) -> float {
        const int64_t row = lo + (int64_t)i * kScanRows + lane;
        return (lane < kScanRows && i < nst && row < hi) ? __ldg(a.knorm + row) : 0.f;
    };
    float kn_cur = load_kn(0), kn_next = load_kn(1);
    const int rr = lane / NQ, b = lane % NQ;
    float qnorm_b = 0.f;  // ||q_b||^2 of this lane's query (no dynamic register indexing)
#pragma unroll
    for (int qb = 0; qb < NQ; ++qb)
        if (b == qb) qnorm_b = qnorm[qb];

    for (int i = 0; i < nst; ++i) {
        const int ps = i & (kPartialRing - 1);
        const int rows = rows_of(i);
        wait_or_abort(&sh.pfull[ps], (uint32_t)(i / kPartialRing) & 1u, &sh.abort, a.status);
        const float kn = __shfl_sync(~0u, kn_cur, rr & (kScanRows - 1));
        bool accept = false;
        uint64_t key = 0;
        if (lane < NV) {
            float dot = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) dot += partial[(ps * kConsumerWarps + w) * NV + lane];
            float dist = fmaf(-2.f, dot, qnorm_b + kn);
            dist = (dist <= 0.f) ? 0.f : dist;  // NaN stays NaN and sorts last
            const int64_t row = lo + (int64_t)i * kScanRows + rr;
            key = ((uint64_t)__float_as_uint(dist) << 32) | (uint32_t)row;
            accept = (rr < rows) && (b < nqv) && (key <= sh.thr[b]) && !key_masked(a.key_mask, row);
        }
        __syncwarp();
        mbar_arrive(&sh.pempty[ps]);
        const uint32_t bal = __ballot_sync(~0u, accept);
        bool full = false;
#pragma unroll
        for (int qb = 0; qb < NQ; ++qb) {
            const uint32_t qm = bal & query_lanes<NQ, NV>(qb);
            if (accept && b == qb) cand[(size_t)qb * a.cap + cnt[qb] + __popc(qm & lanemask_lt())] = key;
            cnt[qb] += __popc(qm);
            full |= cnt[qb] > a.cap - kScanRows;
        }
        kn_cur = kn_next;
        kn_next = load_kn(i + 2);
        if (full) {
            __syncwarp();
            if (lane == 0) {
#pragma unroll
                for (int qb = 0; qb < NQ; ++qb) sh.cnt[qb] = cnt[qb];
            }
            __syncwarp();
            select_smallest<32, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, lane,
                                    [] { __syncwarp(); });
#pragma unroll
            for (int qb = 0; qb < NQ; ++qb) cnt[qb] = sh.cnt[qb];
        }
    }
    __syncwarp();
    if (lane == 0) {
#pragma unroll
        for (int qb = 0; qb < NQ; ++qb) sh.cnt[qb] = cnt[qb];
    }
    __syncwarp();
    select_smallest<32, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, lane, [] { __syncwarp(); });

    // Copies still in flight after an abort must land before the CTA exits.
    if (lane == 0 && *reinterpret_cast<volatile int*>(&sh.abort)) {
        const int issued = *reinterpret_cast<volatile int*>(&sh.issued);
        for (int i = max(0, issued - a.stages); i < issued; ++i)
            (void)mbar_wait_bounded(&sh.full[i % a.stages], (uint32_t)(i / a.stages) & 1u);
    }

    uint64_t* out = a.cand + (size_t)item * NQ * a.r;
#pragma unroll
    for (int qb = 0; qb < NQ; ++qb) {
        const int n = sh.cnt[qb];
        for (int j = lane; j < a.r; j += 32)
            out[(size_t)qb * a.r + j] = j < n ? cand[(size_t)qb * a.cap + j] : kNoCandidate;
        if (lane == 0) a.cand_cnt[(size_t)item * NQ + qb] = n;
    }
}

template <int DT, int NQ, int CPT>
cudaError_t launch_impl(const ScanPlan& p, const ScanArgs& a, cudaStream_t stream)
{
    auto kern = scan_topr_kernel<DT, NQ, CPT>;
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(p.groups * p.parts), dim3(kScanThreads), p.smem, stream, a);
}

template <int DT, int NQ>
cudaError_t launch_cpt(const ScanPlan& p, const ScanArgs& a, cudaStream_t stream)
{
    switch (p.cpt) {
    case 1: return launch_impl<DT, NQ, 1>(p, a, stream);
    case 2: return launch_impl<DT, NQ, 2>(p, a, stream);
    case 4: return launch_impl<DT, NQ, 4>(p, a, stream);
    default: return cudaErrorInvalidValue;
    }
}

template <int DT>
cudaError_t launch_nq(const ScanPlan& p, const ScanArgs& a, cudaStream_t stream)
{
    switch (p.nq) {
    case 1: return launch_cpt<DT, 1>(p, a, stream);
    case 2: return launch_cpt<DT, 2>(p, a, stream);
    case 4: return launch_cpt<DT, 4>(p, a, stream);
    default: return cudaErrorInvalidValue;
    }
}

template <int NQ>
size_t fixed_smem(int cap)
{
    return (size_t)NQ * cap * sizeof(uint64_t) +
           (size_t)kPartialRing * kConsumerWarps * kScanRows * NQ * sizeof(float) +
           sizeof(ScanShared<NQ>) + 128;
}

}  // namespace

bool scan_plan_smem(int dtype, int nq, int cpt, int r, int row_bytes, size_t smem_limit,
                    ScanPlan* plan)
{
    if (dtype != NEST_F32 && dtype != NEST_BF16) return false;
    if (cpt != 1 && cpt != 2 && cpt != 4) return false;
    // r kept candidates plus room to append before a trim; trims are cheap
    // enough that 512 slots of room suffice once r is large.
    const int cap = r < 64 ? r + 64 : (r < 512 ? 2 * r : r + 512);
    size_t fixed;
    switch (nq) {
    case 1: fixed = fixed_smem<1>(cap); break;
    case 2: fixed = fixed_smem<2>(cap); break;
    case 4: fixed = fixed_smem<4>(cap); break;
    default: return false;
    }
    const size_t stage_bytes = (size_t)kScanRows * row_bytes;
    if (fixed + 2 * stage_bytes > smem_limit) return false;
    int stages = (int)((smem_limit - fixed) / stage_bytes);
    stages = stages > kMaxStages ? kMaxStages : stages;
    plan->nq = nq;
    plan->cpt = cpt;
    plan->cap = cap;
    plan->stages = stages;
    plan->stage_bytes = (int)stage_bytes;
    plan->smem = (size_t)stages * stage_bytes + fixed;
    return true;
}

cudaError_t launch_scan(int dtype, const ScanPlan& plan, const ScanArgs& args, cudaStream_t stream)
{
    if (dtype == NEST_BF16) return launch_nq<NEST_BF16>(plan, args, stream);
    if (dtype == NEST_F32) return launch_nq<NEST_F32>(plan, args, stream);
    return cudaErrorInvalidValue;
}

}  // namespace nest
