// internal.h -- declarations shared by the library's translation units
// (host launchers of the kernels; constants of the candidate encoding).
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/nest.h"

namespace nest {

// Launches `kernel` with programmatic stream serialization: its CTAs may be
// scheduled while the previous kernel in the stream finishes (hiding the
// launch latency between the steps of a search); the kernel itself waits
// for that kernel's results with grid_dependency_wait().
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, const Args&... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Raises a kernel's dynamic shared-memory limit on the current device when a
// launch needs more than the largest size set for it so far (one driver
// call per kernel and increase, not per launch).
cudaError_t raise_smem_limit(const void* kernel, size_t smem);

// A candidate neighbour is one 64-bit word: the fp32 bits of its squared
// distance (non-negative, so the bits order like the values) above its
// 32-bit key index.  Ordering the words orders neighbours nearest first
// with ties broken by the smaller key index.  kNoCandidate pads lists.
constexpr uint64_t kNoCandidate = ~0ull;

// Bit k of a key mask set: key k has been used and is never a candidate.
__device__ __forceinline__ bool key_masked(const uint32_t* mask, int64_t k)
{
    return mask != nullptr && ((__ldg(mask + (k >> 5)) >> (k & 31)) & 1u);
}

// Device status word: the first recorded nest_status_t value wins.
__device__ __forceinline__ void record_status(int* status, int code)
{
    atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------- norms.cu
cudaError_t launch_key_norms(const void* K, int64_t N, int32_t d, int dtype, float* knorm,
                             cudaStream_t stream);
cudaError_t launch_check_values(const int32_t* V, int64_t N, int32_t vocab, int* status,
                                cudaStream_t stream);

// ---------------------------------------------------------------- scan.cu
// Distance scan with fused per-CTA top-r (decode / ragged regime).
struct ScanPlan {
    int nq;           // queries per CTA (1, 2 or 4)
    int cpt;          // 16-byte chunks of a row per consumer thread (1, 2 or 4)
    int groups;       // query groups
    int parts;        // key-range parts per group
    int cap;          // candidate buffer entries per query
    int stages;       // pipeline depth
    int stage_bytes;  // bytes of one stage (kScanRows rows)
    size_t smem;      // dynamic shared memory of one CTA
    int ctas_per_sm;  // scan_rows.cu: CTAs one SM holds at once
};

constexpr int kScanRows = 4;           // key rows per pipeline stage
constexpr int kScanThreads = 320;      // 8 consumer warps, 1 producer warp, 1 selector warp

struct ScanArgs {
    const void* K;
    const float* knorm;
    const void* q;
    const int64_t* seg_off;  // nullptr: full scan
    const uint32_t* key_mask;  // nullptr, or bit k set: key k is never a candidate
    uint64_t* cand;          // [groups * parts][nq][r] candidate lists
    int32_t* cand_cnt;       // [groups * parts][nq] real entries of each list
    int* status;
    int64_t N;
    int32_t row_bytes;
    int32_t chunks;  // 16-byte chunks per row
    int32_t B;
    int32_t r;
    int32_t cap;
    int32_t parts;
    int32_t stages;
    int32_t stage_bytes;
};

// Returns false if no kernel exists for (dtype, nq, cpt).
bool scan_plan_smem(int dtype, int nq, int cpt, int r, int row_bytes, size_t smem_limit,
                    ScanPlan* plan);

// ---------------------------------------------------------------- scan_rows.cu
// fp32 keys with rows of at most kRowsMaxBytes: one key row per thread of a
// 128-thread CTA, NQ = 1, 2, 4 or 8 queries per CTA (ScanPlan: nq, cap,
// smem, ctas_per_sm; groups and parts set by the caller).  Same arguments
// and outputs as the scan above.
constexpr int kRowsThreads = 128;
constexpr int kRowsCtasPerSm = 4;  // the kernels' register budget: 128 per thread
constexpr int kRowsMaxBytes = 2048;
bool rows_plan_smem(int nq, int r, int row_bytes, size_t smem_limit, ScanPlan* plan);
cudaError_t launch_scan_rows(const ScanPlan& plan, const ScanArgs& args, cudaStream_t stream);
cudaError_t launch_scan(int dtype, const ScanPlan& plan, const ScanArgs& args,
                        cudaStream_t stream);

// ---------------------------------------------------------------- tc_scan.cu
// Tensor-core (tcgen05) distance scan with fused per-CTA top-r, bf16 keys.
constexpr int kTcThreads = 192;  // producer warp, MMA warp, 4 epilogue warps
constexpr int kTcTileKeys = 128;  // keys per tensor-core tile

struct TcPlan {
    int nq;       // queries per CTA (1, 2, 4, 8 or 16; the MMA always has 16 columns)
    int cap;      // candidate buffer entries per query
    int stages;   // pipeline depth (18 KiB per stage)
    int groups;   // query groups
    int parts;    // key-range parts per group (whole 128-key tiles)
    size_t smem;  // dynamic shared memory of one CTA
};

struct TcScanArgs {
    const float* knorm;
    const void* q;
    const int64_t* seg_off;  // nullptr: full scan
    const uint32_t* key_mask;  // nullptr, or bit k set: key k is never a candidate
    uint64_t* cand;          // [groups * parts][nq][r]
    int32_t* cand_cnt;       // [groups * parts][nq] real entries of each list
    int* status;
    int64_t N;
    int32_t d;
    int32_t B;
    int32_t r;
    int32_t cap;
    int32_t parts;
    int32_t stages;
    int32_t kchunks;     // ceil(d / 64)
    int64_t key_stride;  // the tensor map's row i is key i * key_stride (1, or a sample stride)
};

int tc_cap(int r);
bool tc_plan_smem(int nq, int r, size_t smem_limit, TcPlan* plan);
cudaError_t launch_tc_scan(const TcPlan& plan, const CUtensorMap& keys, const CUtensorMap& queries,
                           const TcScanArgs& args, cudaStream_t stream);

// ---------------------------------------------------------------- tc_wide.cu
// Large query batches: threshold-admission scan into global lists + exact selection.
struct WidePlan {
    int nm;       // MMA N = queries per CTA (16, 32, 64, 128 or 256)
    int mb;       // 128-key tiles per pipeline step: 1, 2 (nm = 256 on one CTA) or 4
                  // (nm = 256 on a CTA pair: two 256-key tiles)
    bool pair;    // nm = 256 on CTA pairs (tcgen05 cta_group::2): M = 256 keys per MMA,
                  // each part is a pair of CTAs
    int stages;
    int groups;   // query groups of nm
    int parts;    // key-range parts (whole 128-key tiles)
    size_t smem;
};

struct WideArgs {
    const float* knorm;
    const void* q;
    const float* qn;  // B: ||q||^2 (launch_wide_qnorm)
    const uint32_t* key_mask;  // nullptr, or bit k set: key k is never a candidate
    int* status;
    const float* s_sample;  // B x r sample neighbours (threshold = s[thr_rank-1]); null: admit all
    int32_t r;
    int32_t thr_rank;       // 1 <= thr_rank <= r
    uint64_t* cand;  // [B][cap] candidate words
    int32_t* cnt;    // [B] candidates appended (must start at 0)
    int64_t cap;
    int64_t N;       // rows of the key tensor map
    int32_t d;
    int32_t B;
    int32_t groups;
    int32_t parts;
    int32_t stages;
    int32_t kchunks;
    int64_t key_stride;  // row i of the key tensor map is key i * key_stride
    // > 0: each epilogue warp reserves list slots per query in blocks of
    // resv (one atomic per block) and pads unused slots with kNoCandidate,
    // so cnt counts reserved slots.  0: one atomic per admitting column.
    int32_t resv;
    // Recovery pass only (launch_tc_wide_recover): per-query word limits
    // (kNoCandidate: not recovering) and per-group flags; groups whose flag
    // is 0 return at once.
    const uint64_t* word_lim;
    const int32_t* group_flag;
};

struct GselectArgs {
    uint64_t* cand;  // [B][cap]; reordered in place
    int32_t* cnt;    // slots taken per list (past cap when a list overflowed)
    int64_t cap;
    int32_t r;
    int32_t B;
    float* s_out;      // B x r (sorted s and idx), unless words_out is set
    int64_t* idx_out;  // B x r
    uint64_t* words_out;    // non-null: the r smallest words of each list, unsorted, [B][r]
    int32_t* words_cnt;     // with words_out: [B] real words
    uint32_t* refine_state;  // with words_out: the exact re-ranking's state, reset per query
    unsigned long long* refine_apair;
    int* status;          // with words_out: NEST_ERR_OVERFLOW if a list is still over capacity
                          // (or held repeated words, which the scans never write)
    // Recovery preparation (instead of any output): for an overflowed list,
    // lim_out[q] = the r-th smallest word it holds; for a list with fewer
    // than r real words (when check_underflow), lim_out[q] = every word up to
    // the sample's r-th distance s_sample[q * r + r - 1]; for either,
    // cnt[q] = 0 and group_flag[q / group_size] = 1.  Otherwise
    // lim_out[q] = kNoCandidate.
    uint64_t* lim_out;
    int32_t* group_flag;
    int32_t group_size;
    const float* s_sample;
    int32_t check_underflow;
    int32_t stage_words;  // shared-memory words per CTA (set by launch_gselect)
};

// ---------------------------------------------------------------- selftest.cu
// One kernel whose bounded mbarrier wait runs out: records NEST_ERR_TIMEOUT
// in *status and the nanoseconds it waited in *waited_ns (device memory).
cudaError_t launch_wait_selftest(int* status, int64_t* waited_ns, cudaStream_t stream);

// Plan of the wide kernel for groups of nm queries; CTA pairs only when `pairs`.
bool wide_plan_smem(int nm, size_t smem_limit, bool pairs, WidePlan* plan);
// 2-CTA clusters of the pair kernel the device can hold at once (0: none or
// the query failed), for the given shared-memory limit per block.
int wide_pair_clusters(size_t smem_limit);
// ||q||^2 of B bf16 rows of d elements into qn (fp32, one warp per row).
cudaError_t launch_wide_qnorm(const void* q, int32_t B, int32_t d, float* qn, cudaStream_t stream);
cudaError_t launch_tc_wide(const WidePlan& plan, const CUtensorMap& keys,
                           const CUtensorMap& queries, const WideArgs& args, cudaStream_t stream);
// Plan of the recovery pass for groups of nm queries: one 128-key tile per
// stage (tc_wide_kernel), whatever kernel the main pass used.
bool wide_recover_plan(int nm, size_t smem_limit, WidePlan* plan);
// The recovery pass (word limits and group flags of args must be set).
cudaError_t launch_tc_wide_recover(const WidePlan& plan, const CUtensorMap& keys,
                                   const CUtensorMap& queries, const WideArgs& args,
                                   cudaStream_t stream);
cudaError_t launch_gselect(const GselectArgs& args, cudaStream_t stream);

// ---------------------------------------------------------------- merge.cu
// Merge candidate lists of each query into its r smallest words.
struct MergeArgs {
    const uint64_t* in;    // candidate lists; list (b, l) starts at (base(b) + l * nq_in) * r with
                           // base(b) = (b / nq_in) * lists * nq_in + b % nq_in
    const int32_t* in_cnt; // real entries of list (b, l), at base(b) + l * nq_in
    int64_t list_stride;   // entries between consecutive lists of one query (nq_in * r)
    int32_t nq_in;
    int32_t lists;         // lists per query
    int32_t per_cta;       // lists merged by one CTA
    int32_t B;
    int32_t r;
    uint64_t* out;         // [B][ceil(lists / per_cta)][r]
    int32_t* out_cnt;      // [B][ceil(lists / per_cta)] real entries of each output list
    uint32_t* refine_state;  // non-null on the final level (one list per query): the exact
    unsigned long long* refine_apair;  // re-ranking's state is reset for each query
    // two-phase merge only: [B][lists][32] summary words and [B][lists] their largest
    uint64_t* sum;
    uint64_t* tsum;
};

int merge_lists_per_cta(int r);
// Lists one merge CTA takes at a level with `lists` input lists per query.
int merge_fanin(int lists, int r);
size_t merge_smem_bytes(int per_cta, int r);
cudaError_t launch_merge(const MergeArgs& args, cudaStream_t stream);
// Whether the two-phase merge (per-list summaries, then one CTA per query)
// applies to `lists` lists of up to r words per query, the scratch words its
// summaries take, and its two launches (out / out_cnt: one list per query).
bool merge_two_phase(int lists, int r);
size_t merge_two_phase_words(int B, int lists);
cudaError_t launch_merge_two_phase(const MergeArgs& args, cudaStream_t stream);

// ---------------------------------------------------------------- refine.cu
// Exact re-ranking: each query's r' = r + refine_margin(r) screened
// candidates get their distances recomputed as sums of squared differences;
// the r nearest by those are sorted into s and idx.
//
// Per-query state: two rows of B 32-bit words (largest and smallest
// screening error as fp32 ordered bits) and B 64-bit words (the largest
// screened distance's bits above its candidate's exact distance bits).  The
// kernel that writes a query's candidate list resets the query's entries.
__device__ __forceinline__ void refine_state_reset(uint32_t* state, unsigned long long* apair,
                                                   int B, int b)
{
    state[b] = 0;
    state[B + b] = ~0u;
    apair[b] = 0;
}

struct RefineArgs {
    const void* K;
    const void* q;       // B x d, same element type as K
    int32_t row_bytes;   // d * element size
    uint64_t* cand;      // [B][rp] screened words (distance bits : key), rewritten in place
    const int32_t* cand_cnt;  // [B] real words of each list
    uint32_t* state;     // [2][B], reset by the kernel that wrote the lists
    unsigned long long* apair;  // [B], likewise
    int* status;
    int32_t B;
    int32_t r;
    int32_t rp;
    float* s_out;        // B x r
    int64_t* idx_out;    // B x r
};

int refine_margin(int r);
cudaError_t launch_refine(int dtype, const RefineArgs& args, cudaStream_t stream);

// ---------------------------------------------------------------- mix.cu
struct MixArgs {
    const float* s;
    const int64_t* idx;
    const int32_t* V;
    const float* p_lm;
    float* p_knn;    // may be null
    float* p_m;
    float* lam_out;  // may be null
    int* status;
    int64_t N;
    int32_t vocab;
    int32_t B;
    int32_t r;
    float mu;
    float lambda;
    int32_t rrc;  // 1: Eq. 4 lambda_t from (alpha, tau)
    float alpha;
    float tau;
    int32_t slices;  // vocabulary slices per query (grid.x)
};

cudaError_t launch_mix(const MixArgs& args, cudaStream_t stream);
int mix_min_slices(int vocab);  // slices needed so each fits the shared-memory sums

// ---------------------------------------------------------------- decide.cu
struct DecideArgs {
    const float* p_m;    // B x vocab
    const float* s;      // B x r
    const int64_t* idx;  // B x r
    const int32_t* V;
    const float* lambda;  // B
    int* status;
    int64_t N;
    int32_t vocab;
    int32_t B;
    int32_t r;
    float delta;
    int32_t* token;
    float* p_max;
    int64_t* span_key;
    int32_t* use_span;
};

struct VerifyArgs {
    const float* p_m;      // rows x vocab
    const int32_t* draft;  // rows
    const int32_t* span_off;  // spans + 1
    int* status;
    int32_t vocab;
    int32_t rows;
    int32_t spans;
    float gamma;
    float* ratio;
    int32_t* accept;
    int32_t* n_accept;
};

cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream);
cudaError_t launch_verify(const VerifyArgs& args, cudaStream_t stream);
cudaError_t launch_mask(uint32_t* mask, int64_t first, int64_t count, cudaStream_t stream);

// ---------------------------------------------------------------- api.cu, for noalloc.cu
// The host checks nest_knn_search makes (arguments, then the datastore's
// device being the current one), with the same status codes.
nest_status_t check_search_call(const nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                                const int64_t* seg_off, const float* s_out,
                                const int64_t* idx_out);
// Scratch words (64-bit) a search of this shape needs; no allocation, no launch.
nest_status_t search_scratch_words(const nest_datastore_t* ds, int32_t B, int32_t r, bool ragged,
                                   size_t* words);
// nest_knn_search with the candidate lists in caller-provided device memory
// of scratch_words words; NEST_ERR_OVERFLOW if the search needs more.
nest_status_t search_with_scratch(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                                  const int64_t* seg_off, float* s_out, int64_t* idx_out,
                                  uint64_t* scratch, size_t scratch_words, cudaStream_t stream);

}  // namespace nest
