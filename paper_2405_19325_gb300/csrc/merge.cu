// merge.cu -- combine per-CTA candidate lists into each query's r' nearest
// screened candidates (the selection of pi, Sec. 2.2 / Algorithm 1's search
// step; refine.cu then re-ranks them by exact distance).
//
// A CTA copies the real entries of up to per_cta lists of one query into
// shared memory (one warp per list, at offsets from the lists' lengths),
// keeps the r' smallest words with the same radix select the scan uses, and
// writes them as one list: for the next level, or, on the final level (one
// CTA per query), for the exact re-ranking.
#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kMergeThreads = 1024;
constexpr size_t kMergeBufBytes = 192 * 1024;
constexpr int kMaxListsPerCta = 1024;

struct MergeShared {
    uint64_t thr;
    int cnt;
    int off[kMaxListsPerCta + 1];  // exclusive prefix of the list lengths
    int wsum[kMergeThreads / 32];
    SelectSmem<kMergeThreads, 1> sel;
};

__host__ __device__ inline int next_pow2(int x)
{
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

__host__ __device__ inline size_t buf_words(int per_cta, int r)
{
    const size_t a = (size_t)per_cta * r, b = (size_t)next_pow2(r);
    return a > b ? a : b;
}

__global__ void __launch_bounds__(kMergeThreads, 1) merge_kernel(const MergeArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    uint64_t* buf = reinterpret_cast<uint64_t*>(smem);
    MergeShared& sh = *reinterpret_cast<MergeShared*>(smem + buf_words(a.per_cta, a.r) * 8);
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.y, grp = blockIdx.x;
    const int l0 = grp * a.per_cta;
    const int nl = min(a.lists, l0 + a.per_cta) - l0;
    const int64_t base = (int64_t)(b / a.nq_in) * a.lists * a.nq_in + b % a.nq_in;
    const uint64_t* src = a.in + base * (int64_t)a.r;

    // exclusive prefix of this CTA's list lengths (nl <= 1024: one value per thread)
    int len = 0;
    if (tid < nl) {
        len = a.in_cnt[base + (int64_t)(l0 + tid) * a.nq_in];
        len = len < 0 ? 0 : (len > a.r ? a.r : len);
    }
    int incl = len;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(~0u, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) sh.wsum[warp] = incl;
    __syncthreads();
    int carry = 0;
    for (int w = 0; w < warp; ++w) carry += sh.wsum[w];
    if (tid < nl) sh.off[tid] = carry + incl - len;
    if (tid == kMergeThreads - 1) sh.off[nl] = carry + incl;  // nl <= 1024: total
    __syncthreads();
    const int total = sh.off[nl];

    // copy the real entries: warp w copies lists w, w + 32, ... to their
    // offsets, eight loads in flight per lane
    for (int l = warp; l < nl; l += kMergeThreads / 32) {
        const int o = sh.off[l], len = sh.off[l + 1] - o;
        const uint64_t* ls = src + (int64_t)(l0 + l) * a.list_stride;
        for (int j0 = lane; j0 < len; j0 += 8 * 32) {
            uint64_t v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int j = j0 + 32 * u;
                if (j < len) v[u] = ls[j];
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int j = j0 + 32 * u;
                if (j < len) buf[o + j] = v[u];
            }
        }
    }
    __syncthreads();
    if (tid == 0) {
        sh.cnt = total;
        sh.thr = kNoCandidate;
    }
    __syncthreads();
    select_smallest<kMergeThreads, 1>(buf, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid,
                                      [] { __syncthreads(); });
    const int n = sh.cnt;

    uint64_t* dst = a.out + ((int64_t)b * gridDim.x + grp) * a.r;
    for (int j = tid; j < a.r; j += kMergeThreads) dst[j] = j < n ? buf[j] : kNoCandidate;
    if (tid == 0) {
        a.out_cnt[(int64_t)b * gridDim.x + grp] = n;
        // the final level hands the query's list to the exact re-ranking
        if (a.refine_state != nullptr)
            refine_state_reset(a.refine_state, a.refine_apair, a.B, b);
    }
}

}  // namespace

int merge_lists_per_cta(int r)
{
    int per = (int)(kMergeBufBytes / ((size_t)r * 8));
    per = per > kMaxListsPerCta ? kMaxListsPerCta : per;
    return per < 2 ? 2 : per;
}

int merge_fanin(int lists, int r)
{
    const int maxper = merge_lists_per_cta(r);
    if (lists <= maxper) return lists;
    // about sqrt(lists) per CTA balances two levels, but no fewer than the
    // next level needs to fit one CTA
    int per = 1;
    while (per * per < lists) ++per;
    const int need = (lists + maxper - 1) / maxper;
    per = per > need ? per : need;
    return per < maxper ? per : maxper;
}

// ---------------------------------------------------------------- two-phase merge
// With many lists per query (one per scan CTA), of which each holds up to r
// words but typically only a few of the query's r nearest, a merge tree
// spends most of its time in radix selects over all the words.  Instead:
//   A. summary_kernel (one 128-thread CTA per list) keeps each list's kTop
//      smallest words (the radix select) and t, the largest of them.
//   B. merge_final_kernel (one 1024-thread CTA per query) takes the r
//      smallest words of all summaries; the largest of those, G, bounds the
//      query's r-th smallest word from above, since at least r words lie at
//      or below it (with fewer than r summary words in all, G is unbounded).
//      Every word <= G is in some summary, except in the lists whose t < G
//      ("saturated"): they may hold more, so they are read in full for their
//      words in (t, G].  A list whose words all fit its
//      summary has no t (kNoCandidate) and is never saturated.  The r
//      smallest of the words <= G are the query's r smallest.  When the
//      saturated lists' words do not fit shared memory they are taken one
//      list at a time, keeping the r smallest seen so far.
// Lists are rarely saturated: with the keys spread over the scan's key
// ranges, each list holds about r / lists of the r nearest (7 of 1,088 at the
// decode workload's 152 lists), far below kTop = 32.
constexpr int kTop = 32;
constexpr int kSumThreads = 128;
constexpr int kFinalThreads = 1024;
constexpr int kFinalWords = 16384;  // shared-memory candidate buffer (128 KiB)

struct SumShared {
    uint64_t thr;
    int cnt;
    unsigned long long tmax;
    SelectSmem<kSumThreads, 1> sel;
};

__global__ void __launch_bounds__(kSumThreads) summary_kernel(const MergeArgs a)
{
    extern __shared__ __align__(16) uint64_t words[];  // the list, up to r words
    __shared__ SumShared sh;
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x;
    const int c = blockIdx.x, b = blockIdx.y;
    const int64_t base = (int64_t)(b / a.nq_in) * a.lists * a.nq_in + b % a.nq_in;
    const int64_t li = base + (int64_t)c * a.nq_in;
    int n = a.in_cnt[li];
    n = n < 0 ? 0 : (n > a.r ? a.r : n);
    const uint64_t* list = a.in + li * a.r;
    for (int j = tid; j < n; j += kSumThreads) words[j] = list[j];
    if (tid == 0) {
        sh.cnt = n;
        sh.thr = kNoCandidate;
        sh.tmax = 0;
    }
    __syncthreads();
    uint64_t* sum = a.sum + ((int64_t)b * a.lists + c) * kTop;
    if (n <= kTop) {
        // the whole list is its summary; it can hold nothing more
        for (int j = tid; j < kTop; j += kSumThreads) sum[j] = j < n ? words[j] : kNoCandidate;
        if (tid == 0) a.tsum[(int64_t)b * a.lists + c] = kNoCandidate;
        return;
    }
    select_smallest<kSumThreads, 1>(words, 0, &sh.cnt, &sh.thr, kTop, sh.sel, tid,
                                    [] { __syncthreads(); });
    for (int j = tid; j < kTop; j += kSumThreads) {
        sum[j] = words[j];
        atomicMax(&sh.tmax, (unsigned long long)words[j]);
    }
    __syncthreads();
    if (tid == 0) a.tsum[(int64_t)b * a.lists + c] = sh.tmax;
}

struct FinalShared {
    uint64_t thr;
    int cnt;
    int extra;
    unsigned long long G;
    SelectSmem<kFinalThreads, 1> sel;
};

// Appends the words w of list[0, n) with lo < w <= hi to buf (warp-aggregated
// slots from sh.cnt).  All threads of the block call it.
__device__ __forceinline__ void append_range(const uint64_t* list, int n, uint64_t lo, uint64_t hi,
                                             uint64_t* buf, int* cnt, int tid, int nthreads)
{
    const int lane = tid & 31;
    for (int base = tid - lane; base < n; base += nthreads) {
        const int j = base + lane;
        const uint64_t w = j < n ? list[j] : kNoCandidate;
        const bool take = w > lo && w <= hi && w != kNoCandidate;
        const uint32_t bal = __ballot_sync(~0u, take);
        if (bal == 0) continue;
        int at = 0;
        if (lane == __ffs(bal) - 1) at = atomicAdd(cnt, __popc(bal));
        at = __shfl_sync(~0u, at, __ffs(bal) - 1);
        if (take) buf[at + __popc(bal & lanemask_lt())] = w;
    }
}

__global__ void __launch_bounds__(kFinalThreads, 1) merge_final_kernel(const MergeArgs a)
{
    extern __shared__ __align__(16) uint64_t buf[];  // kFinalWords words, then the lists' t
    uint64_t* tv = buf + kFinalWords;
    __shared__ FinalShared sh;
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.x;
    const int64_t base = (int64_t)(b / a.nq_in) * a.lists * a.nq_in + b % a.nq_in;
    auto bar = [] { __syncthreads(); };
    for (int c = tid; c < a.lists; c += kFinalThreads) tv[c] = a.tsum[(int64_t)b * a.lists + c];
    if (tid == 0) {
        sh.cnt = 0;
        sh.extra = 0;
        sh.thr = kNoCandidate;
        sh.G = 0;
    }
    __syncthreads();
    // all summary words (at most lists * kTop <= kFinalWords)
    append_range(a.sum + (int64_t)b * a.lists * kTop, a.lists * kTop, 0, kNoCandidate - 1, buf,
                 &sh.cnt, tid, kFinalThreads);
    // word 0 (distance 0, key 0) is real but not above lo = 0: add it if present
    for (int j = tid; j < a.lists * kTop; j += kFinalThreads)
        if (a.sum[(int64_t)b * a.lists * kTop + j] == 0ull) buf[atomicAdd(&sh.cnt, 1)] = 0ull;
    __syncthreads();
    const bool enough = sh.cnt >= a.r;
    select_smallest<kFinalThreads, 1>(buf, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid, bar);
    const int m = sh.cnt;
    for (int j = tid; j < m; j += kFinalThreads) atomicMax(&sh.G, (unsigned long long)buf[j]);
    __syncthreads();
    // With fewer than r summary words in all, nothing bounds the r-th
    // smallest: every word of every list that has more is taken.
    const uint64_t G = enough ? sh.G : kNoCandidate - 1;
    // the saturated lists' further words: counted first
    if (m > 0) {
        for (int c = warp; c < a.lists; c += kFinalThreads / 32) {
            const uint64_t t = tv[c];
            if (t == kNoCandidate || t >= G) continue;  // t == G: nothing in (t, G]
            const int64_t li = base + (int64_t)c * a.nq_in;
            int n = a.in_cnt[li];
            n = n < 0 ? 0 : (n > a.r ? a.r : n);
            const uint64_t* list = a.in + li * a.r;
            int k = 0;
            for (int j = lane; j < n; j += 32) k += list[j] > t && list[j] <= G;
            k = __reduce_add_sync(~0u, k);
            if (lane == 0 && k) atomicAdd(&sh.extra, k);
        }
    }
    __syncthreads();
    if (sh.extra > 0) {
        if (m + sh.extra <= kFinalWords) {
            for (int c = warp; c < a.lists; c += kFinalThreads / 32) {
                const uint64_t t = tv[c];
                if (t == kNoCandidate || t >= G) continue;
                const int64_t li = base + (int64_t)c * a.nq_in;
                int n = a.in_cnt[li];
                n = n < 0 ? 0 : (n > a.r ? a.r : n);
                append_range(a.in + li * a.r, n, t, G, buf, &sh.cnt, lane, 32);
            }
            __syncthreads();
        } else {
            // one saturated list at a time, keeping the r smallest so far
            for (int c = 0; c < a.lists; ++c) {
                const uint64_t t = tv[c];
                if (t == kNoCandidate || t >= G) continue;
                const int64_t li = base + (int64_t)c * a.nq_in;
                int n = a.in_cnt[li];
                n = n < 0 ? 0 : (n > a.r ? a.r : n);
                if (sh.cnt + n > kFinalWords) {
                    select_smallest<kFinalThreads, 1>(buf, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid,
                                                      bar);
                }
                append_range(a.in + li * a.r, n, t, G, buf, &sh.cnt, tid, kFinalThreads);
                __syncthreads();
            }
        }
        select_smallest<kFinalThreads, 1>(buf, 0, &sh.cnt, &sh.thr, a.r, sh.sel, tid, bar);
    }
    const int n = sh.cnt;
    uint64_t* dst = a.out + (int64_t)b * a.r;
    for (int j = tid; j < a.r; j += kFinalThreads) dst[j] = j < n ? buf[j] : kNoCandidate;
    if (tid == 0) {
        a.out_cnt[b] = n;
        refine_state_reset(a.refine_state, a.refine_apair, a.B, b);
    }
}

size_t merge_smem_bytes(int per_cta, int r)
{
    return buf_words(per_cta, r) * 8 + sizeof(MergeShared);
}

cudaError_t launch_merge(const MergeArgs& a, cudaStream_t stream)
{
    const int groups = (a.lists + a.per_cta - 1) / a.per_cta;
    const size_t smem = merge_smem_bytes(a.per_cta, a.r);
    const dim3 grid(groups, a.B);
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(merge_kernel), (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(merge_kernel, grid, dim3(kMergeThreads), smem, stream, a);
}

bool merge_two_phase(int lists, int r)
{
    // more lists than one merge CTA takes, few enough summaries for one CTA,
    // and room for the r kept words plus a list beside them
    return lists > merge_lists_per_cta(r) && lists <= 1024 && (size_t)lists * kTop <= kFinalWords &&
           2 * (size_t)r <= kFinalWords;
}

size_t merge_two_phase_words(int B, int lists)
{
    return (size_t)B * lists * (kTop + 1);
}

cudaError_t launch_merge_two_phase(const MergeArgs& a, cudaStream_t stream)
{
    const size_t wsmem = (size_t)a.r * sizeof(uint64_t);
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(summary_kernel), (int)wsmem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(summary_kernel, dim3(a.lists, a.B), dim3(kSumThreads), wsmem, stream, a);
    if (e != cudaSuccess) return e;
    const size_t fsmem = (size_t)(kFinalWords + a.lists) * sizeof(uint64_t);
    e = raise_smem_limit(reinterpret_cast<const void*>(merge_final_kernel), (int)fsmem);
    if (e != cudaSuccess) return e;
    return launch_pdl(merge_final_kernel, dim3(a.B), dim3(kFinalThreads), fsmem, stream, a);
}

}  // namespace nest
