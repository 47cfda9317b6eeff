// scan.cu -- HBM-streaming distance scan with fused per-CTA top-r
// (the search of Sec. 2.2 / Sec. 3.1: s(q, k) = -||q - k||^2, r nearest).
//
// One CTA owns a group of up to NQ queries and a contiguous range of key
// rows (a slice of the datastore, or a slice of one query's candidate
// segment).  A producer warp streams the rows through a ring of shared-memory
// stages with 1-D TMA bulk copies (mbarrier-tracked, L2 evict-first); eight
// consumer warps hold the queries in registers and compute q.k in fp32 FMA,
// each thread owning fixed 16-byte column chunks of every row.  Per stage of
// kScanRows rows the partial dot products are reduced across the CTA, turned
// into squared distances ||q||^2 + ||k||^2 - 2 q.k, and every candidate that
// can still enter its query's r nearest is appended to a shared-memory list.
// When a list fills up, a radix select trims every list back to r and
// tightens the admission threshold.  At the end the CTA writes its r best
// candidates per query; merge.cu combines the CTAs.  No distance ever goes
// to global memory.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kBarConsumers = 1;  // hardware barrier id used by the consumer warps
constexpr int kMaxStages = 8;

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

// 16 bytes of a row -> fp32 values (bf16 -> fp32 is exact).
template <int DT>
__device__ __forceinline__ void unpack_chunk(const uint4& v, float* x)
{
    if constexpr (DT == NEST_BF16) {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(w[i] << 16);
            x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    } else {
        x[0] = __uint_as_float(v.x);
        x[1] = __uint_as_float(v.y);
        x[2] = __uint_as_float(v.z);
        x[3] = __uint_as_float(v.w);
    }
}

template <int NQ>
struct ScanShared {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t thr[NQ];
    int cnt[NQ];
    float qnorm[NQ];
    int need_select[2];
    int abort;
    int issued;
    SelectSmem<kConsumers, NQ> sel;
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

template <int DT, int NQ, int CPT>
__global__ void __launch_bounds__(kScanThreads, 1) scan_topr_kernel(const ScanArgs a)
{
    constexpr int EPC = Elem<DT>::kPerChunk;
    constexpr int NV = kScanRows * NQ;  // (row, query) dot products per stage
    constexpr int kLanesPerValue = 32 / NV;
    static_assert(NV <= 32 && (NV & (NV - 1)) == 0, "NV must be a power of two <= 32");

    extern __shared__ __align__(128) unsigned char smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int item = blockIdx.x;
    const int group = item / a.parts, part = item - group * a.parts;

    unsigned char* stages = smem;
    uint64_t* cand = reinterpret_cast<uint64_t*>(smem + (size_t)a.stages * a.stage_bytes);
    float* partial = reinterpret_cast<float*>(cand + (size_t)NQ * a.cap);  // [2][warps][NV]
    ScanShared<NQ>& sh =
        *reinterpret_cast<ScanShared<NQ>*>(partial + 2 * kConsumerWarps * NV);

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

    if (tid == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], kConsumerWarps);
        }
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            sh.cnt[b] = 0;
            sh.thr[b] = kNoCandidate;
        }
        sh.need_select[0] = sh.need_select[1] = 0;
        sh.abort = 0;
        sh.issued = 0;
        mbar_init_fence();
    }
    __syncthreads();

    // ---------------------------------------------------------------- producer
    if (warp == kConsumerWarps) {
        if (lane == 0 && nst > 0) {
            const uint64_t policy = l2_policy_evict_first();
            const unsigned char* src = static_cast<const unsigned char*>(a.K) + lo * a.row_bytes;
            for (int i = 0; i < nst; ++i) {
                const int slot = i % a.stages;
                if (i >= a.stages) {
                    if (*reinterpret_cast<volatile int*>(&sh.abort)) break;
                    if (!mbar_wait_bounded(&sh.empty[slot], ((i / a.stages) - 1) & 1)) {
                        record_status(a.status, NEST_ERR_TIMEOUT);
                        *reinterpret_cast<volatile int*>(&sh.abort) = 1;
                        break;
                    }
                }
                const int rows = (int)((nrows - (int64_t)i * kScanRows) < kScanRows ? (nrows - (int64_t)i * kScanRows) : kScanRows);
                const uint32_t bytes = (uint32_t)rows * (uint32_t)a.row_bytes;
                mbar_arrive_expect_tx(&sh.full[slot], bytes);
                bulk_copy_g2s_evict_first(stages + (size_t)slot * a.stage_bytes,
                                          src + (size_t)i * kScanRows * a.row_bytes, bytes,
                                          &sh.full[slot], policy);
                *reinterpret_cast<volatile int*>(&sh.issued) = i + 1;
            }
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    auto bar = [] { named_barrier(kBarConsumers, kConsumers); };

    // Queries of the group, fixed column chunks of this thread, in registers.
    float qf[CPT][NQ][EPC];
    float qn[NQ];
#pragma unroll
    for (int b = 0; b < NQ; ++b) qn[b] = 0.f;
#pragma unroll
    for (int k = 0; k < CPT; ++k) {
        const int c = tid + k * kConsumers;
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            float x[EPC];
            if (c < a.chunks && b < nqv) {
                const uint4 v = ld_global_nc_v4(static_cast<const unsigned char*>(a.q) +
                                                (size_t)(q0 + b) * a.row_bytes + (size_t)c * 16);
                unpack_chunk<DT>(v, x);
            } else {
#pragma unroll
                for (int e = 0; e < EPC; ++e) x[e] = 0.f;
            }
#pragma unroll
            for (int e = 0; e < EPC; ++e) {
                qf[k][b][e] = x[e];
                qn[b] = fmaf(x[e], x[e], qn[b]);
            }
        }
    }
    // ||q||^2 of each query, reduced over the CTA.
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) qn[b] += __shfl_xor_sync(~0u, qn[b], o);
        if (lane == 0) partial[warp * NQ + b] = qn[b];
    }
    bar();
    if (tid < NQ) {
        float t = 0.f;
        for (int w = 0; w < kConsumerWarps; ++w) t += partial[w * NQ + tid];
        sh.qnorm[tid] = t;
    }
    bar();

    // Key norms of a stage's rows, prefetched two stages ahead by warp 0.
    const bool kn_lane = (warp == 0) && (lane < kScanRows);
    auto load_kn = [&](int i) -> float {
        const int64_t row = lo + (int64_t)i * kScanRows + lane;
        return (kn_lane && i < nst && row < hi) ? __ldg(a.knorm + row) : 0.f;
    };
    float kn_cur = load_kn(0), kn_next = load_kn(1);

    for (int i = 0; i < nst; ++i) {
        const int slot = i % a.stages;
        const int rows = (int)((nrows - (int64_t)i * kScanRows) < kScanRows ? (nrows - (int64_t)i * kScanRows) : kScanRows);
        if (!*reinterpret_cast<volatile int*>(&sh.abort)) {
            if (!mbar_wait_bounded(&sh.full[slot], (uint32_t)(i / a.stages) & 1u)) {
                record_status(a.status, NEST_ERR_TIMEOUT);
                *reinterpret_cast<volatile int*>(&sh.abort) = 1;
            }
        }
        float acc[kScanRows][NQ];
#pragma unroll
        for (int rr = 0; rr < kScanRows; ++rr)
#pragma unroll
            for (int b = 0; b < NQ; ++b) acc[rr][b] = 0.f;
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
                        float x[EPC];
                        unpack_chunk<DT>(v, x);
#pragma unroll
                        for (int b = 0; b < NQ; ++b)
#pragma unroll
                            for (int e = 0; e < EPC; ++e)
                                acc[rr][b] = fmaf(qf[k][b][e], x[e], acc[rr][b]);
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.empty[slot]);

        float v[NV];
#pragma unroll
        for (int rr = 0; rr < kScanRows; ++rr)
#pragma unroll
            for (int b = 0; b < NQ; ++b) v[rr * NQ + b] = acc[rr][b];
        const float red = warp_reduce_scatter<NV>(v, lane);
        if ((lane & (kLanesPerValue - 1)) == 0)
            partial[((i & 1) * kConsumerWarps + warp) * NV + lane / kLanesPerValue] = red;
        bar();

        if (sh.need_select[i & 1]) select_smallest<kConsumers, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, tid, bar);

        if (warp == 0) {
            const int rr = lane / NQ, b = lane % NQ;
            const float kn = __shfl_sync(~0u, kn_cur, rr & (kScanRows - 1));
            bool accept = false;
            uint64_t key = 0;
            if (lane < NV) {
                float dot = 0.f;
#pragma unroll
                for (int w = 0; w < kConsumerWarps; ++w)
                    dot += partial[((i & 1) * kConsumerWarps + w) * NV + lane];
                float dist = fmaf(-2.f, dot, sh.qnorm[b] + kn);
                dist = (dist <= 0.f) ? 0.f : dist;  // NaN stays NaN and sorts last
                const int64_t row = lo + (int64_t)i * kScanRows + rr;
                key = ((uint64_t)__float_as_uint(dist) << 32) | (uint32_t)row;
                accept = (rr < rows) && (b < nqv) && (key <= sh.thr[b]);
            }
            const uint32_t bal = __ballot_sync(~0u, accept);
            bool full = false;
#pragma unroll
            for (int qb = 0; qb < NQ; ++qb) {
                const uint32_t qm = bal & query_lanes<NQ, NV>(qb);
                const int base = sh.cnt[qb];
                if (accept && b == qb) cand[(size_t)qb * a.cap + base + __popc(qm & lanemask_lt())] = key;
                const int nc = base + __popc(qm);
                full |= nc > a.cap - kScanRows;
                __syncwarp();
                if (lane == 0) sh.cnt[qb] = nc;
            }
            if (lane == 0) sh.need_select[(i + 1) & 1] = full ? 1 : 0;
            kn_cur = kn_next;
            kn_next = load_kn(i + 2);
        }
    }
    bar();
    select_smallest<kConsumers, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, tid, bar);

    // Copies still in flight after an abort must land before the CTA exits.
    if (tid == 0 && *reinterpret_cast<volatile int*>(&sh.abort)) {
        const int issued = *reinterpret_cast<volatile int*>(&sh.issued);
        for (int i = max(0, issued - a.stages); i < issued; ++i)
            (void)mbar_wait_bounded(&sh.full[i % a.stages], (uint32_t)(i / a.stages) & 1u);
    }

    uint64_t* out = a.cand + (size_t)item * NQ * a.r;
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
        const int n = sh.cnt[b];
        for (int j = tid; j < a.r; j += kConsumers)
            out[(size_t)b * a.r + j] = j < n ? cand[(size_t)b * a.cap + j] : kNoCandidate;
    }
}

template <int DT, int NQ, int CPT>
cudaError_t launch_impl(const ScanPlan& p, const ScanArgs& a, cudaStream_t stream)
{
    auto kern = scan_topr_kernel<DT, NQ, CPT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e != cudaSuccess) return e;
    kern<<<p.groups * p.parts, kScanThreads, p.smem, stream>>>(a);
    return cudaGetLastError();
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
    return (size_t)NQ * cap * sizeof(uint64_t) + 2 * kConsumerWarps * kScanRows * NQ * sizeof(float) +
           sizeof(ScanShared<NQ>) + 128;
}

}  // namespace

bool scan_plan_smem(int dtype, int nq, int cpt, int r, int row_bytes, size_t smem_limit,
                    ScanPlan* plan)
{
    if (dtype != NEST_F32 && dtype != NEST_BF16) return false;
    if (cpt != 1 && cpt != 2 && cpt != 4) return false;
    const int cap = r < 64 ? r + 64 : 2 * r;
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
