// scan_rows.cu -- distance scan with fused per-CTA top-r for fp32 datastores
// with narrow rows (the search of Sec. 2.2 / Sec. 3.1: s(q, k) = -||q - k||^2,
// r nearest), as search path 5.
//
// scan.cu gives each consumer thread fixed 16-byte column chunks of every
// row, which suits rows of kilobytes; a 256-byte row (d = 64) would keep 16
// of its 256 consumer threads busy and move 1 KiB per pipeline stage.  Here
// each thread takes whole key rows instead:
//
//   * a 128-thread CTA owns a group of up to NQ queries (in shared memory,
//     read as broadcasts) and a contiguous range of key rows, 128 rows per
//     tile, one row per thread;
//   * a warp stages its 32 rows through shared memory 128 bytes of each row
//     at a time, with per-thread asynchronous copies into two buffers (the
//     next slab is in flight while the current one is used): eight 16-byte
//     copies per lane, each warp-wide copy reading four runs of 128
//     contiguous bytes, stored with the chunk index XOR-ed by the row so
//     that the per-row reads after them are free of bank conflicts;
//   * each thread then accumulates its row's NQ dot products in fp32 with
//     packed FMAs (two partial sums per query);
//   * it forms ||q||^2 + ||k||^2 - 2 q.k and appends the candidates that can
//     still enter each query's r nearest to shared-memory lists (warp ballot,
//     one atomic per warp and query); a list that fills up is trimmed back
//     to r by the radix select, which also tightens the admission threshold.
//
// Three CTAs share an SM (shared memory) and each warp keeps its next slab in
// flight.  At d = 64 with 8 queries the kernel streams about 0.45 of the HBM
// copy rate and is bound by instruction issue (some 1,600 instructions per
// warp and 32 keys), not by memory.  The output is the same per-CTA
// candidate lists as the other narrow scans, merged by merge.cu and
// re-ranked exactly by refine.cu.
#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kRowsSlab = 8;  // 16-byte chunks of each row staged per pass (128 bytes)
constexpr int kRowsPerCopy = 32 / kRowsSlab;  // rows one warp-wide copy brings
constexpr int kRowsStageBytes = (kRowsThreads / 32) * 2 * 32 * kRowsSlab * 16;  // 32 KiB per CTA

// Candidate words of the lists in shared memory, rounded up to an even count
// so that the query rows after them start on a 16-byte boundary.
__host__ __device__ constexpr size_t rows_cand_words(int nq, int cap)
{
    return ((size_t)nq * cap + 1) & ~(size_t)1;
}

template <int NQ>
struct RowsShared {
    uint64_t thr[NQ];
    int cnt[NQ];
    float qn[NQ];
    SelectSmem<kRowsThreads, NQ> sel;
};

template <int NQ>
__global__ void __launch_bounds__(kRowsThreads, kRowsCtasPerSm) scan_rows_kernel(const ScanArgs a)
{
    // [NQ][cap] candidate words (an even count, so that what follows is
    // 16-byte aligned), then [NQ][chunks] 16-byte chunks of the query rows,
    // then each warp's two staging buffers of 32 rows x kRowsSlab chunks
    extern __shared__ __align__(16) unsigned char smem[];
    uint64_t* cand = reinterpret_cast<uint64_t*>(smem);
    uint4* qs = reinterpret_cast<uint4*>(cand + rows_cand_words(NQ, a.cap));
    __shared__ RowsShared<NQ> sh;

    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int item = blockIdx.x;
    const int group = item / a.parts, part = item - group * a.parts;
    auto bar = [] { __syncthreads(); };

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
    const int nch = a.chunks;  // 16-byte chunks of a row (4 fp32 values)

    // ---- the group's query rows (zero for padding queries) and their norms
    for (int i = tid; i < NQ * nch; i += kRowsThreads) {
        const int b = i / nch, c = i - b * nch;
        qs[i] = b < nqv ? ld_global_nc_v4(static_cast<const unsigned char*>(a.q) +
                                          (size_t)(q0 + b) * a.row_bytes + (size_t)c * 16)
                        : make_uint4(0u, 0u, 0u, 0u);
    }
    if (tid < NQ) {
        sh.cnt[tid] = 0;
        sh.thr[tid] = kNoCandidate;
    }
    bar();
    for (int b = warp; b < NQ; b += kRowsThreads / 32) {
        float s = 0.f;
        for (int c = lane; c < nch; c += 32) {
            const uint4 v = qs[b * nch + c];
            s = fmaf(__uint_as_float(v.x), __uint_as_float(v.x), s);
            s = fmaf(__uint_as_float(v.y), __uint_as_float(v.y), s);
            s = fmaf(__uint_as_float(v.z), __uint_as_float(v.z), s);
            s = fmaf(__uint_as_float(v.w), __uint_as_float(v.w), s);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) s += __shfl_xor_sync(~0u, s, o);
        if (lane == 0) sh.qn[b] = s;
    }
    bar();
    float qn[NQ];
#pragma unroll
    for (int b = 0; b < NQ; ++b) qn[b] = sh.qn[b];

    const int64_t nrows = hi - lo;
    const int ntiles = (int)((nrows + kRowsThreads - 1) / kRowsThreads);
    const int nslab = (nch + kRowsSlab - 1) / kRowsSlab;  // 128-byte slabs of a row
    const int total = ntiles * nslab;
    // this warp's two staging buffers of 32 rows x kRowsSlab chunks
    uint4* stg = qs + (size_t)NQ * nch + (size_t)warp * 2 * 32 * kRowsSlab;
    const unsigned char* kbase = static_cast<const unsigned char*>(a.K);
    // Slab k (tile k / nslab, chunks from (k % nslab) * kRowsSlab) of the
    // warp's 32 rows into buffer k & 1: copy i brings rows 4i .. 4i + 3
    // (eight lanes each), four runs of up to 128 contiguous bytes; chunk c of
    // row rr goes to slot rr * kRowsSlab + (c ^ (rr % kRowsSlab)).  Chunks
    // past the row or rows past the range are zero-filled.
    auto issue = [&](int k) {
        const int tt = k / nslab, c0 = (k - tt * nslab) * kRowsSlab;
        const int64_t wrow0 = lo + (int64_t)tt * kRowsThreads + 32 * warp;
        uint4* buf = stg + (size_t)(k & 1) * 32 * kRowsSlab;
#pragma unroll
        for (int i = 0; i < kRowsSlab; ++i) {
            const int rr = kRowsPerCopy * i + lane / kRowsSlab, c = lane % kRowsSlab;
            const int64_t lr = wrow0 + rr;
            const bool ok = lr < hi && c0 + c < nch;
            const unsigned char* src =
                ok ? kbase + (size_t)lr * a.row_bytes + (size_t)(c0 + c) * 16 : kbase;
            cp_async_16(buf + rr * kRowsSlab + (c ^ (rr % kRowsSlab)), src, ok ? 16u : 0u);
        }
        cp_async_commit();
    };
    if (total > 0) issue(0);
    float2 acc[NQ];  // two partial sums per query (even and odd elements)
    float kn = 0.f;
    bool in = false;
    int64_t row = 0;
    for (int k = 0; k < total; ++k) {
        const int t = k / nslab, s = k - t * nslab;
        // the next slab's copies go out before this one is used
        if (k + 1 < total) issue(k + 1);
        else cp_async_commit();  // an empty group keeps the count of groups in flight
        cp_async_wait<1>();
        __syncwarp();  // every lane's copies of slab k have landed
        if (s == 0) {
            row = lo + (int64_t)t * kRowsThreads + 32 * warp + lane;
            in = row < hi;
            kn = in ? __ldg(a.knorm + row) : 0.f;
#pragma unroll
            for (int b = 0; b < NQ; ++b) acc[b] = make_float2(0.f, 0.f);
        }
        const uint4* buf = stg + (size_t)(k & 1) * 32 * kRowsSlab;
        const int c0 = s * kRowsSlab;
#pragma unroll
        for (int c = 0; c < kRowsSlab; ++c) {
            if (c0 + c >= nch) break;  // the same for every thread
            const uint4 kv = buf[lane * kRowsSlab + (c ^ (lane % kRowsSlab))];
            const float2 k01 = make_float2(__uint_as_float(kv.x), __uint_as_float(kv.y));
            const float2 k23 = make_float2(__uint_as_float(kv.z), __uint_as_float(kv.w));
#pragma unroll
            for (int b = 0; b < NQ; ++b) {
                const uint4 qv = qs[b * nch + c0 + c];
                // packed: lane 0 sums the even elements, lane 1 the odd ones
                acc[b] = __ffma2_rn(make_float2(__uint_as_float(qv.x), __uint_as_float(qv.y)), k01,
                                    acc[b]);
                acc[b] = __ffma2_rn(make_float2(__uint_as_float(qv.z), __uint_as_float(qv.w)), k23,
                                    acc[b]);
            }
        }
        __syncwarp();  // buffer k & 1 is read before slab k + 2 is copied into it
        if (s != nslab - 1) continue;
        const bool valid = in && !key_masked(a.key_mask, row);
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            float dist = fmaf(-2.f, acc[b].x + acc[b].y, qn[b] + kn);
            dist = (dist <= 0.f) ? 0.f : dist;  // NaN stays NaN and sorts last
            const uint64_t key = ((uint64_t)__float_as_uint(dist) << 32) | (uint32_t)row;
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
        for (int b = 0; b < NQ; ++b) need |= sh.cnt[b] > a.cap - kRowsThreads;
        bar();  // every thread has decided before any appends of the next tile
        if (need) select_smallest<kRowsThreads, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, tid, bar);
    }
    bar();
    select_smallest<kRowsThreads, NQ>(cand, a.cap, sh.cnt, sh.thr, a.r, sh.sel, tid, bar);
    uint64_t* out = a.cand + (size_t)item * NQ * a.r;
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
        const int n = sh.cnt[b];
        for (int j = tid; j < a.r; j += kRowsThreads)
            out[(size_t)b * a.r + j] = j < n ? cand[(size_t)b * a.cap + j] : kNoCandidate;
        if (tid == 0) a.cand_cnt[(size_t)item * NQ + b] = n;
    }
}

template <int NQ>
size_t rows_static_smem()
{
    return sizeof(RowsShared<NQ>);
}

template <int NQ>
cudaError_t rows_launch(const ScanPlan& p, const ScanArgs& a, cudaStream_t stream)
{
    auto kern = scan_rows_kernel<NQ>;
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), (int)p.smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(p.groups * p.parts), dim3(kRowsThreads), p.smem, stream, a);
}

}  // namespace

bool rows_plan_smem(int nq, int r, int row_bytes, size_t smem_limit, ScanPlan* plan)
{
    if (row_bytes <= 0 || row_bytes > kRowsMaxBytes || row_bytes % 16 != 0) return false;
    size_t stat;
    switch (nq) {
    case 1: stat = rows_static_smem<1>(); break;
    case 2: stat = rows_static_smem<2>(); break;
    case 4: stat = rows_static_smem<4>(); break;
    case 8: stat = rows_static_smem<8>(); break;
    default: return false;
    }
    const int cap = tc_cap(r);  // r kept plus room for at least one tile of appends
    const size_t dyn = rows_cand_words(nq, cap) * sizeof(uint64_t) + (size_t)nq * row_bytes +
                       kRowsStageBytes;
    if (dyn + stat > smem_limit) return false;
    plan->nq = nq;
    plan->cpt = 0;
    plan->cap = cap;
    plan->stages = 1;
    plan->stage_bytes = 0;
    plan->smem = dyn;
    // CTAs of this size one SM holds at once (its shared memory taken as the
    // per-block limit plus the 1 KiB the runtime reserves per block)
    const size_t per_cta = dyn + stat + 1024;
    const size_t fit = (smem_limit + 1024) / per_cta;
    plan->ctas_per_sm = (int)(fit < 1 ? 1 : (fit > 16 ? 16 : fit));
    return true;
}

cudaError_t launch_scan_rows(const ScanPlan& plan, const ScanArgs& args, cudaStream_t stream)
{
    switch (plan.nq) {
    case 1: return rows_launch<1>(plan, args, stream);
    case 2: return rows_launch<2>(plan, args, stream);
    case 4: return rows_launch<4>(plan, args, stream);
    case 8: return rows_launch<8>(plan, args, stream);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace nest
