// refine.cu -- exact re-ranking of each query's screened candidates (the
// r nearest keys by s(q, k) = -||q - k||^2, Sec. 2.2 / App. A).
//
// The scans rank keys by ||q||^2 + ||k||^2 - 2 q.k evaluated in fp32.  Its
// rounding error is absolute in the norms (the dot product is accumulated
// over d terms of the size of ||q|| ||k||), so two keys whose distances
// differ by less than that error can come out in either order, and a key
// very close to the query gets a distance with a large relative error.  The
// searches therefore keep r' = r + margin candidates per query, and this
// kernel recomputes each candidate's distance directly as the sum of the
// squared differences of the stored elements (fp32, exact products of the
// widened bf16 values; eight interleaved partial sums per lane and a warp
// tree, so at most ~40 additions separate any term from the result).  It
// then puts the r nearest by those distances in order (ties: smaller key
// index) and writes s = -distance and the key index.
//
// Two kernels (the second a programmatic dependent of the first):
//   refine_dist_kernel  grid (chunks of 16 candidates, B queries), 512
//                       threads: warp w of chunk c recomputes candidate
//                       16 c + w, all of its row's 16-byte loads in flight
//                       at once (8 or 16 KiB rows), and rewrites the word in
//                       place; each CTA folds its screening errors into the
//                       query's state with atomics.
//   then, for a few queries (B < kSortMinB):
//   refine_rank_kernel  grid (chunks of 16 candidates, B queries), 512
//                       threads: warp w of chunk c takes candidate 16 c + w,
//                       counts the query's words below its own (the words
//                       are distinct, so the counts are the sorted
//                       positions), and writes s and idx at that position
//                       when it is below r.  No sort and no CTA that waits
//                       for the others: r' x r' comparisons per query spread
//                       over r' / 16 CTAs, which suits a handful of queries;
//   or, for more queries:
//   refine_sort_kernel  one 1024-thread CTA per query sorts its r' words in
//                       shared memory (bitonic network, O(r' log^2 r')
//                       compare-exchanges) and writes the first r.
//
// It also checks the margin.  A key left out of the r' candidates had a
// screened distance of at least A, the largest screened distance kept.  The
// screening errors e = screened - exact of the candidates span [e_min, e_max]
// (mostly a common offset: the accumulation error grows with ||q|| ||k||,
// which is about the same for keys at about the same distance).  Taking an
// excluded key's error to exceed that of the candidate at A by at most
// W = 2 (e_max - e_min), its exact distance is at least A_exact - W, where
// A_exact is the exact distance of that candidate.  So the r nearest are
// certain when A_exact - W > D_r, the r-th exact distance.  When instead the
// candidate at A ties the r-th exactly, the boundary lies inside a run of
// exact ties (duplicated keys: equal screened and exact distances, broken
// by index the same way in both), which also passes.  Otherwise a key
// outside the candidates might belong to the r nearest and NEST_ERR_MARGIN
// is recorded.
#include <cmath>

#include "internal.h"
#include "ptx.cuh"
#include "select.cuh"

namespace nest {
namespace {

constexpr int kRefineThreads = 512;
constexpr int kRefineRows = kRefineThreads / 32;  // candidates per CTA
constexpr int kRefineLoads = 16;                  // 16-byte loads in flight per lane
constexpr int kRankThreads = 512;  // one warp per position, 16 per CTA
constexpr int kSortThreads = 1024;
// From this many queries on, each query's words are sorted by one CTA
// instead of ranked by r' / 16 CTAs.  One CTA sorts r' = 1,088 words in
// about 20 us; the rank kernel spends about 0.38 us per query at that r'
// once its grid fills the GPU (97 against 29 us at B = 256 on a GB300, about
// even at B = 64, and the rank kernel ahead below).
constexpr int kSortMinB = 96;
// Distance bits no real distance has (a NaN pattern above +inf's bits).
constexpr uint64_t kPadHigh = 0xFFFFFFFFull << 32;

// fp32 values as unsigned integers that order like the values.
__device__ __forceinline__ uint32_t ordered_bits(float x)
{
    const uint32_t u = __float_as_uint(x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float from_ordered_bits(uint32_t o)
{
    return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

struct RefineShared {
    uint32_t emax, emin;      // largest / smallest screened - exact distance (ordered bits)
    unsigned long long apair; // largest (screened bits << 32 | exact bits) of this CTA
};

// Sum of squared differences of one 16-byte chunk (8 bf16 or 4 fp32 values)
// into the lane's partial sums.
template <int DT>
__device__ __forceinline__ void chunk_sqdiff(const uint4& k, const uint4& q, float (&acc)[8])
{
    const uint32_t kw[4] = {k.x, k.y, k.z, k.w};
    const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
    if constexpr (DT == NEST_BF16) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float d0 = __uint_as_float(qw[i] << 16) - __uint_as_float(kw[i] << 16);
            const float d1 = __uint_as_float(qw[i] & 0xffff0000u) - __uint_as_float(kw[i] & 0xffff0000u);
            acc[2 * i] = fmaf(d0, d0, acc[2 * i]);
            acc[2 * i + 1] = fmaf(d1, d1, acc[2 * i + 1]);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float d0 = __uint_as_float(qw[i]) - __uint_as_float(kw[i]);
            acc[i] = fmaf(d0, d0, acc[i]);
        }
    }
}

template <int DT>
__global__ void __launch_bounds__(kRefineThreads) refine_dist_kernel(const RefineArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    uint4* qs = reinterpret_cast<uint4*>(smem);  // the query row
    __shared__ RefineShared sh;
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.y;
    const int chunks = a.row_bytes / 16;
    uint64_t* list = a.cand + (int64_t)b * a.rp;
    const int n = min(max(a.cand_cnt[b], 0), a.rp);
    const int j = blockIdx.x * kRefineRows + warp;
    const uint64_t w = j < n ? list[j] : kNoCandidate;

    const uint4* qrow = reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(a.q) +
                                                       (size_t)b * a.row_bytes);
    for (int c = tid; c < chunks; c += kRefineThreads) qs[c] = ld_global_nc_v4(qrow + c);
    if (tid == 0) {
        sh.emax = 0;
        sh.emin = ~0u;
        sh.apair = 0;
    }
    __syncthreads();

    // ---- one warp per candidate: exact distance, word rewritten in place
    if (w != kNoCandidate) {
        const uint32_t key = (uint32_t)w;
        const uint4* krow = reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(a.K) +
                                                           (size_t)key * a.row_bytes);
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        int c = lane;
        for (; c + (kRefineLoads - 1) * 32 < chunks; c += kRefineLoads * 32) {
            uint4 kv[kRefineLoads];
#pragma unroll
            for (int u = 0; u < kRefineLoads; ++u) kv[u] = ld_global_nc_v4(krow + c + 32 * u);
            // every load is issued before the first use of any: the empty
            // volatile statements keep the arithmetic after all sixteen
#pragma unroll
            for (int u = 0; u < kRefineLoads; ++u)
                asm volatile("" : "+r"(kv[u].x), "+r"(kv[u].y), "+r"(kv[u].z), "+r"(kv[u].w));
#pragma unroll
            for (int u = 0; u < kRefineLoads; ++u) chunk_sqdiff<DT>(kv[u], qs[c + 32 * u], acc);
        }
        for (; c < chunks; c += 32) chunk_sqdiff<DT>(ld_global_nc_v4(krow + c), qs[c], acc);
        float s = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) s += __shfl_xor_sync(~0u, s, o);
        if (lane == 0) {
            const float screened = __uint_as_float((uint32_t)(w >> 32));
            list[j] = ((uint64_t)__float_as_uint(s) << 32) | key;
            const uint32_t e = ordered_bits(screened - s);
            atomicMax(&sh.emax, e);
            atomicMin(&sh.emin, e);
            // distances are >= 0, so their bits order like the values
            atomicMax(&sh.apair, ((unsigned long long)(w >> 32) << 32) | __float_as_uint(s));
        }
    }
    __syncthreads();
    if (tid == 0 && sh.emin != ~0u) {
        atomicMax(&a.state[b], sh.emax);
        atomicMin(&a.state[a.B + b], sh.emin);
        atomicMax(&a.apair[b], sh.apair);
    }
}

// The margin of query b, given its r-th smallest exact word.  Keys outside
// the candidates exist only when the list is full (the callers check n ==
// rp); the kernel that writes the lists resets the state.
__device__ __forceinline__ void check_margin(const RefineArgs& a, int b, uint64_t rth)
{
    const float A_exact = __uint_as_float((uint32_t)a.apair[b]);
    const float emax = from_ordered_bits(a.state[b]);
    const float emin = from_ordered_bits(a.state[a.B + b]);
    const float Dr = __uint_as_float((uint32_t)(rth >> 32));
    const float W = 2.f * (emax - emin);
    const bool ok = (A_exact - W > Dr) || (A_exact == Dr);
    if (!ok) record_status(a.status, NEST_ERR_MARGIN);
}

__global__ void __launch_bounds__(kRankThreads) refine_rank_kernel(const RefineArgs a)
{
    extern __shared__ __align__(16) uint64_t words[];  // the query's n words
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.y;
    const uint64_t* list = a.cand + (int64_t)b * a.rp;
    const int n = min(max(a.cand_cnt[b], 0), a.rp);
    // A padding word (none is expected among the n) becomes a distinct
    // word above every real one, so the positions stay a permutation.
    for (int i = tid; i < n; i += kRankThreads) {
        const uint64_t w = list[i];
        words[i] = w != kNoCandidate ? w : (kPadHigh | (uint32_t)i);
    }
    __syncthreads();
    // one warp per position i: candidate i's rank, or the padding of a short row
    const int i = blockIdx.x * (kRankThreads / 32) + warp;
    float* so = a.s_out + (int64_t)b * a.r;
    int64_t* io = a.idx_out + (int64_t)b * a.r;
    if (i < n) {
        const uint64_t mine = words[i];
        int below = 0;
        for (int k = lane; k < n; k += 32) below += words[k] < mine;
        const int rank = __reduce_add_sync(~0u, below);
        if (lane == 0 && rank < a.r) {
            if ((mine >> 32) < 0xFFFFFFFFu) {
                so[rank] = -__uint_as_float((uint32_t)(mine >> 32));
                io[rank] = (int64_t)(uint32_t)mine;
            } else {
                so[rank] = -INFINITY;
                io[rank] = -1;
            }
        }
        if (lane == 0 && rank == a.r - 1 && n == a.rp) check_margin(a, b, mine);
    } else if (i < a.r && lane == 0) {
        so[i] = -INFINITY;  // positions n .. r - 1 of a short row
        io[i] = -1;
    }
}

// One CTA per query: its n words (exact distances : key), padded to P2 (a
// power of two >= max(r', r)) with distinct words above every real one,
// sorted ascending; position j < r gives s and idx, as refine_rank_kernel
// writes them.
__global__ void __launch_bounds__(kSortThreads) refine_sort_kernel(const RefineArgs a, int P2)
{
    extern __shared__ __align__(16) uint64_t sorted[];  // P2 words
    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x;
    const int b = blockIdx.x;
    const uint64_t* list = a.cand + (int64_t)b * a.rp;
    const int n = min(max(a.cand_cnt[b], 0), a.rp);
    for (int i = tid; i < P2; i += kSortThreads) {
        const uint64_t w = i < n ? list[i] : kNoCandidate;
        sorted[i] = w != kNoCandidate ? w : (kPadHigh | (uint32_t)i);
    }
    __syncthreads();
    bitonic_sort<kSortThreads>(sorted, P2, tid, [] { __syncthreads(); });
    float* so = a.s_out + (int64_t)b * a.r;
    int64_t* io = a.idx_out + (int64_t)b * a.r;
    for (int j = tid; j < a.r; j += kSortThreads) {
        const uint64_t w = sorted[j];
        if ((w >> 32) < 0xFFFFFFFFu) {
            so[j] = -__uint_as_float((uint32_t)(w >> 32));
            io[j] = (int64_t)(uint32_t)w;
        } else {
            so[j] = -INFINITY;
            io[j] = -1;
        }
        if (j == a.r - 1 && n == a.rp) check_margin(a, b, w);
    }
}

}  // namespace

int refine_margin(int r)
{
    const int m = r / 16;
    return m < 16 ? 16 : (m > 128 ? 128 : m);
}

cudaError_t launch_refine(int dtype, const RefineArgs& a, cudaStream_t stream)
{
    const dim3 grid((a.rp + kRefineRows - 1) / kRefineRows, a.B);
    const size_t qbytes = (size_t)a.row_bytes;
    cudaError_t e;
    if (dtype == NEST_BF16) {
        e = raise_smem_limit(reinterpret_cast<const void*>(refine_dist_kernel<NEST_BF16>), qbytes);
        if (e == cudaSuccess)
            e = launch_pdl(refine_dist_kernel<NEST_BF16>, grid, dim3(kRefineThreads), qbytes, stream, a);
    } else {
        e = raise_smem_limit(reinterpret_cast<const void*>(refine_dist_kernel<NEST_F32>), qbytes);
        if (e == cudaSuccess)
            e = launch_pdl(refine_dist_kernel<NEST_F32>, grid, dim3(kRefineThreads), qbytes, stream, a);
    }
    if (e != cudaSuccess) return e;
    const int cover = a.rp > a.r ? a.rp : a.r;
    if (a.B >= kSortMinB) {
        int P2 = 1;
        while (P2 < cover) P2 <<= 1;
        const size_t sbytes = (size_t)P2 * sizeof(uint64_t);
        e = raise_smem_limit(reinterpret_cast<const void*>(refine_sort_kernel), sbytes);
        if (e != cudaSuccess) return e;
        return launch_pdl(refine_sort_kernel, dim3(a.B), dim3(kSortThreads), sbytes, stream, a, P2);
    }
    // rank threads cover max(r', r) positions: candidates, then the padding of short rows
    const dim3 rgrid((cover + kRankThreads / 32 - 1) / (kRankThreads / 32), a.B);
    const size_t wbytes = (size_t)a.rp * sizeof(uint64_t);
    e = raise_smem_limit(reinterpret_cast<const void*>(refine_rank_kernel), wbytes);
    if (e != cudaSuccess) return e;
    return launch_pdl(refine_rank_kernel, rgrid, dim3(kRankThreads), wbytes, stream, a);
}

}  // namespace nest
