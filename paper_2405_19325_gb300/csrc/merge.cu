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

}  // namespace nest
