// api.cu -- the C ABI of include/nest.h: argument validation, the datastore
// handle, scratch memory, and the choice and launch of the kernels.
#include <algorithm>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <new>
#include <map>
#include <mutex>
#include <vector>

#include <cudaTypedefs.h>

#include "internal.h"

using namespace nest;

struct nest_datastore {
    const void* K = nullptr;
    const int32_t* V = nullptr;
    int64_t N = 0;
    int32_t d = 0;
    int dtype = 0;
    int32_t vocab = 0;
    int32_t row_bytes = 0;
    int device = 0;
    int num_sms = 1;
    size_t smem_optin = 0;
    bool tc = false;         // bf16 keys with a TMA tensor map: tensor-core scan
    bool pairs_ok = false;   // the device can place the wide kernel's CTA pairs
    int pairs_mode = 0;      // 1: groups of 256 on pairs, 0: never, -1: when one group
    CUtensorMap keys_map;  // TMA map of K (type is 64-byte aligned)
    float* knorm = nullptr;  // owned: ||k_i||^2, N floats
    int* status = nullptr;   // owned: device status word
    uint64_t* scratch = nullptr;  // owned: candidate lists of the search
    size_t scratch_words = 0;
    unsigned char* host_stage = nullptr;  // owned: device copies for nest_knn_step_host
    size_t host_stage_bytes = 0;
    cudaStream_t aux = nullptr;           // owned: side stream of nest_knn_step_host
    cudaEvent_t aux_ev[3] = {nullptr, nullptr, nullptr};
    int* host_status = nullptr;           // owned, page-locked: status copy of nest_knn_step_host
    bool timing = false;
    std::vector<cudaEvent_t> events;  // pairs (start, end)
    size_t events_used = 0;
    int64_t launches = 0;
};

namespace {

constexpr int64_t kMaxKeys = 4294967294LL;  // key indices travel as 32 bits
// Recovery passes after an overflowed large-batch list (each at most one
// more scan of the keys, only for the query groups concerned).
constexpr int kRecoverRounds = 3;
constexpr int32_t kMaxB = 65535;

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

nest_status_t from_cuda(cudaError_t e)
{
    if (e == cudaSuccess) return NEST_OK;
    if (e == cudaErrorMemoryAllocation) return NEST_ERR_OOM;
    return NEST_ERR_CUDA;
}

cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

int element_size(int dtype) { return dtype == NEST_BF16 ? 2 : 4; }

// Search layout chosen for a call: which scan kernel, its plan, and the
// candidate words of the scan output and of the merge levels.
struct SearchPlan {
    int r;         // neighbours returned
    int rp;        // screened candidates kept per query for the exact re-ranking
    bool tc;       // tensor-core scan (bf16) or CUDA-core scan
    bool rows;     // CUDA-core scan of narrow fp32 rows, one row per thread (scan_rows.cu)
    ScanPlan scan;
    TcPlan tcp;
    int nq, groups, parts;
    bool two_phase;      // merge by per-list summaries (merge.cu) instead of a tree
    size_t cand_words;   // scan output: groups * parts * nq * rp
    size_t level_words;  // merge level outputs (ping-pong partner of the scan output)
    size_t cnt_words;    // list lengths of the scan output and of the merge levels
    size_t off_fin;      // each query's rp candidates for the re-ranking: B * rp words,
                         // B int32 lengths and 2 * B uint32 of re-ranking state (rounded
                         // up to whole words), then B 64-bit words of state
    size_t total_words;  // all scratch of the search
    // Large query batches (tc_wide.cu): sample pass + thresholded pass.
    bool wide;
    WidePlan wps, wpm, wpr;   // sample pass, main pass, recovery pass
    int64_t stride;           // sample = every stride-th key
    int32_t thr_rank;         // main pass admits keys up to the sample's thr_rank-th distance
    int64_t sample_rows;
    bool single_pass;         // the sample is the whole datastore
    int64_t cap_s, cap_m;     // list capacities per query
    int32_t resv;             // main pass: list slots an epilogue warp reserves at a time
    size_t off_cnt, off_qn, off_lim, off_cand_s, off_s_s, off_i_s, off_cand_m, wide_words;
    size_t cnt_ints;          // int32 counters and flags zeroed per search
};

// Parts per query group.  Time ~ waves * (work per part + fixed cost per part),
// the fixed cost (prologue, final selection, one more list to merge) being
// worth about 64 keys of streaming; parts hold at least 256 keys.
int choose_parts(int groups, int64_t keys_per_group, int num_sms, bool ragged)
{
    const int64_t by_keys = std::max<int64_t>(1, keys_per_group / 256);
    const int max_parts = (int)std::min<int64_t>(ragged ? 256 : 4096, by_keys);
    const double fixed = 64.0 / (double)std::max<int64_t>(1, keys_per_group);
    int best = 1;
    double best_cost = 1e30;
    for (int p = 1; p <= max_parts; ++p) {
        const int64_t items = (int64_t)groups * p;
        const int64_t waves = (items + num_sms - 1) / num_sms;
        const double cost = (double)waves * (1.0 / p + fixed);
        if (cost < best_cost * (1 - 1e-9)) {
            best_cost = cost;
            best = p;
        }
    }
    return best;
}

int ceil_pow2(int x)
{
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

nest_status_t plan_search(const nest_datastore* ds, int B, int r_out, bool ragged,
                          SearchPlan* sp)
{
    // Every step below keeps r = r_out + margin screened candidates; the
    // exact re-ranking (refine.cu) returns r_out of them.
    const int r = r_out + refine_margin(r_out);
    sp->r = r_out;
    sp->rp = r;
    const size_t fin_words = (size_t)B * r + ((size_t)3 * B + 1) / 2 + (size_t)B;
    sp->tc = false;
    const int64_t keys_per_group_full = ds->N;
    if (ds->tc) {
        int nq = ragged ? 1 : ceil_pow2(std::min(B, 16));
        TcPlan tp{};
        bool ok = false;
        for (;;) {
            if (tc_plan_smem(nq, r, ds->smem_optin, &tp)) {
                ok = true;
                break;
            }
            if (nq == 1) break;
            nq /= 2;
        }
        if (ok) {
            tp.groups = ragged ? B : (B + nq - 1) / nq;
            const int64_t keys_per_group = ragged ? (ds->N + B - 1) / B : keys_per_group_full;
            tp.parts = choose_parts(tp.groups, keys_per_group, ds->num_sms, ragged);
            sp->tc = true;
            sp->tcp = tp;
            sp->nq = nq;
            sp->groups = tp.groups;
            sp->parts = tp.parts;
        }
    }
    sp->rows = false;
    if (!sp->tc && ds->dtype == NEST_F32 && ds->row_bytes <= kRowsMaxBytes) {
        // narrow fp32 rows: one row per thread (scan_rows.cu), several CTAs per SM
        int nq = ragged ? 1 : ceil_pow2(std::min(B, 8));
        ScanPlan p{};
        while (!rows_plan_smem(nq, r, ds->row_bytes, ds->smem_optin, &p)) {
            if (nq == 1) return NEST_ERR_UNSUPPORTED;
            nq /= 2;
        }
        p.groups = ragged ? B : (B + nq - 1) / nq;
        const int64_t keys_per_group = ragged ? (ds->N + B - 1) / B : keys_per_group_full;
        // up to four CTAs per SM (the kernel's register budget) count as
        // slots: more parts would only add lists to merge
        const int slots = ds->num_sms * std::min(p.ctas_per_sm, kRowsCtasPerSm);
        p.parts = choose_parts(p.groups, keys_per_group, slots, ragged);
        sp->rows = true;
        sp->scan = p;
        sp->nq = p.nq;
        sp->groups = p.groups;
        sp->parts = p.parts;
    }
    if (!sp->tc && !sp->rows) {
        const int chunks = ds->row_bytes / 16;
        const int cpt = chunks <= 256 ? 1 : (chunks <= 512 ? 2 : 4);
        int nq = ragged ? 1 : (B >= 3 ? 4 : B);
        ScanPlan p{};
        while (!scan_plan_smem(ds->dtype, nq, cpt, r, ds->row_bytes, ds->smem_optin, &p)) {
            if (nq == 1) return NEST_ERR_UNSUPPORTED;
            nq /= 2;
        }
        p.groups = ragged ? B : (B + nq - 1) / nq;
        const int64_t keys_per_group = ragged ? (ds->N + B - 1) / B : keys_per_group_full;
        p.parts = choose_parts(p.groups, keys_per_group, ds->num_sms, ragged);
        sp->scan = p;
        sp->nq = p.nq;
        sp->groups = p.groups;
        sp->parts = p.parts;
    }
    sp->cand_words = (size_t)sp->groups * sp->parts * sp->nq * r;
    const int per = merge_fanin(sp->parts, r);
    const int lvl1 = (sp->parts + per - 1) / per;
    sp->level_words = lvl1 > 1 ? (size_t)B * lvl1 * r : 0;
    sp->two_phase = merge_two_phase(sp->parts, r);
    if (sp->two_phase) sp->level_words = merge_two_phase_words(B, sp->parts);
    // int32 counts: [groups * parts * nq] then [B * lvl1], as 64-bit words
    sp->cnt_words = ((size_t)sp->groups * sp->parts * sp->nq + 1) / 2 + ((size_t)B * lvl1 + 1) / 2;
    sp->off_fin = sp->cand_words + sp->level_words + sp->cnt_words;
    sp->total_words = sp->off_fin + fin_words;
    sp->wide = false;
    // More queries than one CTA can keep lists for: stream the keys once per
    // group of up to 256 queries (512 on CTA pairs) against sampled
    // admission thresholds.
    if (sp->tc && !ragged && sp->groups > 1) {
        // CTA pairs: when asked for, or (automatic) when the batch is one
        // group of up to 512, whose key ranges no other group's CTAs stream
        // beside them
        const bool pairs =
            ds->pairs_ok && (ds->pairs_mode == 1 || (ds->pairs_mode < 0 && B <= 512));
        int nm = B >= 256 ? 256 : std::max(16, ceil_pow2(B));
        if (pairs && B > 256 && B <= 512) nm = 512;  // one pair group of 512
        WidePlan wp{};
        bool planned = wide_plan_smem(nm, ds->smem_optin, pairs, &wp);
        if (!planned && nm == 512) {
            nm = 256;
            planned = wide_plan_smem(nm, ds->smem_optin, false, &wp);
        }
        if (planned) {
            wp.groups = (B + nm - 1) / nm;
            // A sample of every stride-th key, about max(65,536, 64 r) keys.
            const int64_t target = std::max<int64_t>(65536, 64 * (int64_t)r);
            sp->stride = std::max<int64_t>(1, ds->N / target);
            sp->sample_rows = ds->N / sp->stride;
            sp->single_pass = sp->stride == 1;
            // Admission threshold of the main pass: the sample's j-th
            // smallest distance.  The sample holds on average r / stride of
            // a query's r nearest keys; j = max(32, 4 r / stride) lets about
            // max(32 stride, 4 r) keys of the datastore through, and the
            // chance that the sample holds j of the r nearest (so that fewer
            // than r keys pass) is negligible for any layout that systematic
            // sampling does not alias.  It is checked all the same: a query
            // left with fewer than r survivors is scanned again with the
            // sample's r-th distance, which bounds the true r-th from above.
            sp->thr_rank = (int32_t)std::min<int64_t>(
                r, std::max<int64_t>(32, (4 * (int64_t)r + sp->stride - 1) / sp->stride));
            sp->wps = wp;
            // a CTA pair takes two SMs
            const int slots = wp.pair ? ds->num_sms / 2 : ds->num_sms;
            sp->wps.parts = choose_parts(wp.groups, sp->sample_rows, slots, false);
            sp->wpm = wp;
            sp->wpm.parts = choose_parts(wp.groups, ds->N, slots, false);
            sp->cap_s = sp->sample_rows;
            const int64_t expect =
                (ds->N * (int64_t)sp->thr_rank + sp->sample_rows - 1) / sp->sample_rows;
            // Main-pass lists hold 8x the expected survivors plus what the
            // epilogue warps' reservations can leave unwritten.  About a
            // fraction j / sample_rows of the keys pass the sample's j-th
            // distance, so a warp that drains `rows` key rows admits about
            // rows * j / sample_rows keys per query; it reserves twice that
            // plus 16 slots at a time (one atomic per block).  Each column
            // has 4 reserving warps per 128-key tile of a step (8 with two
            // key tiles per stage, 16 over a CTA pair's four).
            const int epi_warps = 4 * wp.mb;
            const int64_t unit = (int64_t)kTcTileKeys * wp.mb;
            const int64_t units = (ds->N + unit - 1) / unit;
            const int64_t rows = (units + sp->wpm.parts - 1) / sp->wpm.parts * 32;
            const int64_t per_warp =
                (rows * sp->thr_rank + sp->sample_rows - 1) / sp->sample_rows;
            sp->resv = (int32_t)std::min<int64_t>(2 * per_warp + 16, 1024);
            const int64_t unwritten = (int64_t)sp->wpm.parts * epi_warps * sp->resv;
            sp->cap_m = std::min<int64_t>(ds->N, std::max<int64_t>(8LL * r, 8 * expect)) + unwritten;
            // recovery of overflowed main-pass lists: groups of up to 256
            // queries (a group of 512 as two), one 128-key tile per stage
            const int nr = std::min(nm, 256);
            if (!wide_recover_plan(nr, ds->smem_optin, &sp->wpr)) return NEST_ERR_UNSUPPORTED;
            sp->wpr.groups = (B + nr - 1) / nr;
            sp->wpr.parts = choose_parts(sp->wpr.groups, ds->N, ds->num_sms, false);
            // 2 * B int32 counters, then kRecoverRounds * recovery groups
            // int32 flags (zeroed by one memset per search)
            sp->off_cnt = 0;
            sp->cnt_ints = 2 * (size_t)B + (size_t)kRecoverRounds * sp->wpr.groups;
            sp->off_qn = (sp->cnt_ints + 1) / 2;
            sp->off_lim = sp->off_qn + ((size_t)B + 1) / 2;  // after B floats ||q||^2
            sp->off_cand_s = sp->off_lim + (size_t)B;       // after B word limits
            sp->off_s_s = sp->off_cand_s + (size_t)B * sp->cap_s;
            sp->off_i_s = sp->off_s_s + ((size_t)B * r + 1) / 2;
            sp->off_cand_m = sp->off_i_s + (size_t)B * r;
            sp->wide_words = sp->single_pass ? sp->off_s_s : sp->off_cand_m + (size_t)B * sp->cap_m;
            // list positions and counters are 32-bit in the kernels: lists
            // that could pass 2^31 words stay on the narrow scan
            if (sp->cap_s < INT32_MAX && (sp->single_pass || sp->cap_m < INT32_MAX)) {
                sp->wide = true;
                sp->cand_words = sp->wide_words;
                sp->level_words = 0;
                sp->cnt_words = 0;
                sp->off_fin = sp->wide_words;
                sp->total_words = sp->wide_words + fin_words;
            }
        }
    }
    return NEST_OK;
}

// cuTensorMapEncodeTiled from the driver, looked up once.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            (void)cudaGetLastError();
            p = nullptr;
        }
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }();
    return fn;
}

// 2-D bf16 tensor map over rows x d (row stride d * 2 bytes), box of
// box_rows rows x 64 columns, 128-byte swizzle; rows and columns outside
// the tensor read as zero.
bool encode_bf16_rows(CUtensorMap* map, const void* base, int64_t rows, int32_t d, int box_rows,
                      bool keys, int64_t row_step = 1)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)d * 2 * (cuuint64_t)row_step};
    const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    const cuuint32_t elem[2] = {1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                           strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B,
                           keys ? CU_TENSOR_MAP_L2_PROMOTION_L2_256B : CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

nest_status_t ensure_scratch(nest_datastore* ds, size_t words)
{
    if (words <= ds->scratch_words) return NEST_OK;
    if (ds->scratch) {
        cudaError_t e = cudaFree(ds->scratch);
        ds->scratch = nullptr;
        ds->scratch_words = 0;
        if (e != cudaSuccess) return from_cuda(e);
    }
    void* p = nullptr;
    cudaError_t e = cudaMalloc(&p, words * sizeof(uint64_t));
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return NEST_ERR_OOM;
    }
    ds->scratch = static_cast<uint64_t*>(p);
    ds->scratch_words = words;
    return NEST_OK;
}

nest_status_t record_event(nest_datastore* ds, cudaStream_t stream)
{
    if (ds->events_used == ds->events.size()) {
        cudaEvent_t ev;
        cudaError_t e = cudaEventCreate(&ev);
        if (e != cudaSuccess) return from_cuda(e);
        ds->events.push_back(ev);
    }
    return from_cuda(cudaEventRecord(ds->events[ds->events_used++], stream));
}

}  // namespace

cudaError_t nest::raise_smem_limit(const void* kernel, size_t smem)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    static std::mutex mu;
    static std::map<std::pair<const void*, int>, size_t> limit;
    {
        std::lock_guard<std::mutex> lock(mu);
        const auto it = limit.find({kernel, dev});
        if (it != limit.end() && it->second >= smem) return cudaSuccess;
    }
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) {
        std::lock_guard<std::mutex> lock(mu);
        size_t& v = limit[{kernel, dev}];
        v = v > smem ? v : smem;
    }
    return e;
}

namespace {

// Device buffers of nest_knn_step_host, grown on demand (never shrunk).
nest_status_t ensure_host_stage(nest_datastore* ds, size_t bytes)
{
    if (bytes <= ds->host_stage_bytes) return NEST_OK;
    if (ds->host_stage) {
        cudaError_t e = cudaFree(ds->host_stage);
        ds->host_stage = nullptr;
        ds->host_stage_bytes = 0;
        if (e != cudaSuccess) return from_cuda(e);
    }
    void* p = nullptr;
    cudaError_t e = cudaMalloc(&p, bytes);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return NEST_ERR_OOM;
    }
    ds->host_stage = static_cast<unsigned char*>(p);
    ds->host_stage_bytes = bytes;
    return NEST_OK;
}

size_t round256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// The side stream, events and page-locked status word of
// nest_knn_step_host, created on first use.
nest_status_t ensure_aux(nest_datastore* ds)
{
    if (ds->aux) return NEST_OK;
    cudaError_t e = cudaStreamCreateWithFlags(&ds->aux, cudaStreamNonBlocking);
    for (int i = 0; i < 3 && e == cudaSuccess; ++i)
        e = cudaEventCreateWithFlags(&ds->aux_ev[i], cudaEventDisableTiming);
    if (e == cudaSuccess && !ds->host_status)
        e = cudaHostAlloc(reinterpret_cast<void**>(&ds->host_status), sizeof(int),
                          cudaHostAllocDefault);
    if (e != cudaSuccess) {
        for (cudaEvent_t& ev : ds->aux_ev) {
            if (ev) (void)cudaEventDestroy(ev);
            ev = nullptr;
        }
        if (ds->aux) (void)cudaStreamDestroy(ds->aux);
        ds->aux = nullptr;
        return from_cuda(e);
    }
    return NEST_OK;
}

// Device pointers only: plain host memory would fault on GPUs that cannot reach it.
bool is_device_pointer(const void* p)
{
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

nest_status_t check_search_args(const nest_datastore* ds, const void* q, int32_t B, int32_t r,
                                const int64_t* seg_off, const float* s_out,
                                const int64_t* idx_out)
{
    if (!ds || !q || !s_out || !idx_out) return NEST_ERR_INVALID_ARG;
    if (B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R) return NEST_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(s_out, 4) || !aligned(idx_out, 8)) return NEST_ERR_ALIGN;
    if (seg_off && !aligned(seg_off, 8)) return NEST_ERR_ALIGN;
    return NEST_OK;
}

// Kernels run on the current device and read the datastore's memory: a call
// made with another device current is refused before anything is launched.
nest_status_t check_device(const nest_datastore* ds)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return NEST_ERR_CUDA;
    }
    return dev == ds->device ? NEST_OK : NEST_ERR_INVALID_ARG;
}

nest_status_t check_mix_args(const nest_datastore* ds, const float* s_in, const int64_t* idx_in,
                             const float* p_lm, int32_t B, int32_t r, const float* p_knn_out,
                             const float* p_m_out)
{
    if (!ds || !s_in || !idx_in || !p_lm || !p_m_out) return NEST_ERR_INVALID_ARG;
    if (B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R) return NEST_ERR_INVALID_ARG;
    if (!aligned(s_in, 4) || !aligned(idx_in, 8) || !aligned(p_lm, 4) || !aligned(p_m_out, 4) ||
        (p_knn_out && !aligned(p_knn_out, 4)))
        return NEST_ERR_ALIGN;
    return NEST_OK;
}

// Large query batches: [sample pass, selection of the sample,] thresholded
// pass over all keys, selection of each query's rp candidates into the
// re-ranking region (fin, fin_cnt, state).
nest_status_t launch_wide(nest_datastore* ds, const SearchPlan& sp, const void* q, int32_t B,
                          const uint32_t* key_mask, uint64_t* scratch, uint64_t* fin,
                          int32_t* fin_cnt, uint32_t* state, unsigned long long* apair,
                          bool timed, cudaStream_t stream)
{
    const int32_t r = sp.rp;
    nest_status_t st;
    int32_t* cnt = reinterpret_cast<int32_t*>(scratch + sp.off_cnt);
    int32_t* flags = cnt + 2 * (size_t)B;  // kRecoverRounds rows of groups
    cudaError_t e = cudaMemsetAsync(cnt, 0, sizeof(int32_t) * sp.cnt_ints, stream);
    if (e != cudaSuccess) return from_cuda(e);
    CUtensorMap qmap;
    // a CTA of a pair stages 128 queries of each 256 of the group
    if (!encode_bf16_rows(&qmap, q, B, ds->d, sp.wpm.pair ? 128 : sp.wpm.nm, false))
        return NEST_ERR_CUDA;

    WideArgs wa{};
    wa.knorm = ds->knorm;
    wa.q = q;
    float* qn = reinterpret_cast<float*>(scratch + sp.off_qn);
    wa.qn = qn;
    wa.key_mask = key_mask;
    wa.status = ds->status;
    wa.r = r;
    wa.d = ds->d;
    wa.B = B;
    wa.groups = sp.wpm.groups;
    wa.stages = sp.wpm.stages;
    wa.kchunks = (ds->d + 63) / 64;
    e = launch_wide_qnorm(q, B, ds->d, qn, stream);
    if (e != cudaSuccess) return from_cuda(e);
    ++ds->launches;

    GselectArgs ga{};
    ga.r = r;
    ga.B = B;

    if (sp.single_pass) {
        // the "sample" is every key: its r nearest screened are the candidates
        wa.s_sample = nullptr;
        wa.cand = scratch + sp.off_cand_s;
        wa.cnt = cnt;
        wa.cap = sp.cap_s;
        wa.N = ds->N;
        wa.parts = sp.wpm.parts;
        wa.key_stride = 1;
        if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
        e = launch_tc_wide(sp.wpm, ds->keys_map, qmap, wa, stream);
        if (e != cudaSuccess) return from_cuda(e);
        if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
        ga.cand = wa.cand;
        ga.cnt = cnt;
        ga.cap = sp.cap_s;
        ga.words_out = fin;
        ga.words_cnt = fin_cnt;
        ga.refine_state = state;
        ga.refine_apair = apair;
        e = launch_gselect(ga, stream);
        if (e != cudaSuccess) return from_cuda(e);
        ds->launches += 2;
        return NEST_OK;
    }

    CUtensorMap smap;
    if (!encode_bf16_rows(&smap, ds->K, sp.sample_rows, ds->d, kTcTileKeys, true, sp.stride))
        return NEST_ERR_CUDA;
    float* s_s = reinterpret_cast<float*>(scratch + sp.off_s_s);
    int64_t* i_s = reinterpret_cast<int64_t*>(scratch + sp.off_i_s);
    // 1. sample pass: every sampled key is a candidate
    wa.s_sample = nullptr;
    wa.cand = scratch + sp.off_cand_s;
    wa.cnt = cnt;
    wa.cap = sp.cap_s;
    wa.N = sp.sample_rows;
    wa.parts = sp.wps.parts;
    wa.key_stride = sp.stride;
    e = launch_tc_wide(sp.wps, smap, qmap, wa, stream);
    if (e != cudaSuccess) return from_cuda(e);
    ga.cand = wa.cand;
    ga.cnt = cnt;
    ga.cap = sp.cap_s;
    ga.s_out = s_s;
    ga.idx_out = i_s;
    e = launch_gselect(ga, stream);
    if (e != cudaSuccess) return from_cuda(e);
    // 2. every key, admitted at or below the sample's thr_rank-th screened distance
    wa.s_sample = s_s;
    wa.thr_rank = sp.thr_rank;
    wa.cand = scratch + sp.off_cand_m;
    wa.cnt = cnt + B;
    wa.cap = sp.cap_m;
    wa.N = ds->N;
    wa.parts = sp.wpm.parts;
    wa.key_stride = 1;
    wa.resv = sp.resv;
    if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
    e = launch_tc_wide(sp.wpm, ds->keys_map, qmap, wa, stream);
    if (e != cudaSuccess) return from_cuda(e);
    if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
    // 3. Lists with fewer than r survivors (the threshold came out below
    // the query's r-th distance) are scanned again up to the sample's r-th
    // distance, a safe bound; lists that overflowed (more survivors than
    // their capacity: many keys tied at the threshold, say) are scanned
    // again with a tighter limit, the r-th smallest word each holds.  Both
    // kernels of a round return at once when no list needs it.
    uint64_t* lim = scratch + sp.off_lim;
    CUtensorMap rmap;
    if (!encode_bf16_rows(&rmap, q, B, ds->d, sp.wpr.nm, false)) return NEST_ERR_CUDA;
    for (int round = 0; round < kRecoverRounds; ++round) {
        GselectArgs gp{};
        gp.cand = wa.cand;
        gp.cnt = cnt + B;
        gp.cap = sp.cap_m;
        gp.r = r;
        gp.B = B;
        gp.lim_out = lim;
        gp.group_flag = flags + (size_t)round * sp.wpr.groups;
        gp.group_size = sp.wpr.nm;
        gp.s_sample = s_s;
        gp.check_underflow = round == 0 ? 1 : 0;
        e = launch_gselect(gp, stream);
        if (e != cudaSuccess) return from_cuda(e);
        WideArgs wr = wa;
        wr.resv = 0;
        wr.groups = sp.wpr.groups;
        wr.parts = sp.wpr.parts;
        wr.stages = sp.wpr.stages;
        wr.word_lim = lim;
        wr.group_flag = gp.group_flag;
        e = launch_tc_wide_recover(sp.wpr, ds->keys_map, rmap, wr, stream);
        if (e != cudaSuccess) return from_cuda(e);
        ds->launches += 2;
    }
    ga.cand = wa.cand;
    ga.cnt = cnt + B;
    ga.cap = sp.cap_m;
    ga.s_out = nullptr;
    ga.idx_out = nullptr;
    ga.status = ds->status;
    ga.words_out = fin;
    ga.words_cnt = fin_cnt;
    ga.refine_state = state;
    ga.refine_apair = apair;
    e = launch_gselect(ga, stream);
    if (e != cudaSuccess) return from_cuda(e);
    ds->launches += 4;
    return NEST_OK;
}

// Plan, check the scratch, launch the scan and the merge tree (or the
// large-batch passes), then the exact re-ranking.  The scratch (64-bit
// words) is the handle's own or the caller's; timing events are recorded
// around the scan when `timed`.
nest_status_t launch_search(nest_datastore* ds, const void* q, int32_t B, int32_t r_out,
                            const int64_t* seg_off, const uint32_t* key_mask, float* s_out,
                            int64_t* idx_out, uint64_t* scratch, size_t scratch_words,
                            bool timed, cudaStream_t stream)
{
    SearchPlan sp;
    nest_status_t st = plan_search(ds, B, r_out, seg_off != nullptr, &sp);
    if (st != NEST_OK) return st;
    if (sp.total_words > scratch_words) return NEST_ERR_OVERFLOW;
    const int32_t r = sp.rp;
    uint64_t* fin = scratch + sp.off_fin;
    int32_t* fin_cnt = reinterpret_cast<int32_t*>(fin + (size_t)B * r);
    uint32_t* state = reinterpret_cast<uint32_t*>(fin_cnt + B);
    auto* apair = reinterpret_cast<unsigned long long*>(fin + (size_t)B * r + (3 * (size_t)B + 1) / 2);

    cudaError_t e;
    if (sp.wide) {
        st = launch_wide(ds, sp, q, B, key_mask, scratch, fin, fin_cnt, state, apair, timed,
                         stream);
        if (st != NEST_OK) return st;
    } else {
        uint64_t* regionA = scratch;
        uint64_t* regionB = scratch + sp.cand_words;
        int32_t* cntA = reinterpret_cast<int32_t*>(scratch + sp.cand_words + sp.level_words);
        int32_t* cntB = cntA + ((size_t)sp.groups * sp.parts * sp.nq + 1) / 2 * 2;
        if (sp.tc) {
            CUtensorMap qmap;
            if (!encode_bf16_rows(&qmap, q, B, ds->d, 16, false)) return NEST_ERR_CUDA;
            TcScanArgs ta{};
            ta.knorm = ds->knorm;
            ta.q = q;
            ta.seg_off = seg_off;
            ta.key_mask = key_mask;
            ta.cand = regionA;
            ta.cand_cnt = cntA;
            ta.status = ds->status;
            ta.N = ds->N;
            ta.d = ds->d;
            ta.B = B;
            ta.r = r;
            ta.cap = sp.tcp.cap;
            ta.parts = sp.tcp.parts;
            ta.stages = sp.tcp.stages;
            ta.kchunks = (ds->d + 63) / 64;
            ta.key_stride = 1;
            if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
            e = launch_tc_scan(sp.tcp, ds->keys_map, qmap, ta, stream);
        } else {
            ScanArgs sa{};
            sa.K = ds->K;
            sa.knorm = ds->knorm;
            sa.q = q;
            sa.seg_off = seg_off;
            sa.key_mask = key_mask;
            sa.cand = regionA;
            sa.cand_cnt = cntA;
            sa.status = ds->status;
            sa.N = ds->N;
            sa.row_bytes = ds->row_bytes;
            sa.chunks = ds->row_bytes / 16;
            sa.B = B;
            sa.r = r;
            sa.cap = sp.scan.cap;
            sa.parts = sp.scan.parts;
            sa.stages = sp.scan.stages;
            sa.stage_bytes = sp.scan.stage_bytes;
            if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;
            e = sp.rows ? launch_scan_rows(sp.scan, sa, stream)
                        : launch_scan(ds->dtype, sp.scan, sa, stream);
        }
        if (e != cudaSuccess) return from_cuda(e);
        ++ds->launches;
        if (timed && (st = record_event(ds, stream)) != NEST_OK) return st;

        MergeArgs ma{};
        ma.in = regionA;
        ma.in_cnt = cntA;
        ma.list_stride = (int64_t)sp.nq * r;
        ma.nq_in = sp.nq;
        ma.lists = sp.parts;
        ma.B = B;
        ma.r = r;
        bool into_b = true;
        if (sp.two_phase) {
            // per-list summaries (their largest words first, then the words)
            ma.tsum = regionB;
            ma.sum = regionB + (size_t)B * sp.parts;
            ma.out = fin;
            ma.out_cnt = fin_cnt;
            ma.refine_state = state;
            ma.refine_apair = apair;
            e = launch_merge_two_phase(ma, stream);
            if (e != cudaSuccess) return from_cuda(e);
            ds->launches += 2;
        }
        for (; !sp.two_phase;) {
            ma.per_cta = merge_fanin(ma.lists, r);
            const int groups = (ma.lists + ma.per_cta - 1) / ma.per_cta;
            const bool last = groups == 1;
            ma.out = last ? fin : (into_b ? regionB : regionA);
            ma.out_cnt = last ? fin_cnt : (into_b ? cntB : cntA);
            ma.refine_state = last ? state : nullptr;
            ma.refine_apair = last ? apair : nullptr;
            e = launch_merge(ma, stream);
            if (e != cudaSuccess) return from_cuda(e);
            ++ds->launches;
            if (last) break;
            ma.in = ma.out;
            ma.in_cnt = ma.out_cnt;
            ma.list_stride = r;
            ma.nq_in = 1;
            ma.lists = groups;
            into_b = !into_b;
        }
    }

    RefineArgs ra{};
    ra.K = ds->K;
    ra.q = q;
    ra.row_bytes = ds->row_bytes;
    ra.cand = fin;
    ra.cand_cnt = fin_cnt;
    ra.state = state;
    ra.apair = apair;
    ra.status = ds->status;
    ra.B = B;
    ra.r = sp.r;
    ra.rp = r;
    ra.s_out = s_out;
    ra.idx_out = idx_out;
    e = launch_refine(ds->dtype, ra, stream);
    if (e != cudaSuccess) return from_cuda(e);
    ++ds->launches;
    return NEST_OK;
}

nest_status_t run_search(nest_datastore* ds, const void* q, int32_t B, int32_t r,
                         const int64_t* seg_off, float* s_out, int64_t* idx_out,
                         cudaStream_t stream, const uint32_t* key_mask = nullptr)
{
    SearchPlan sp;
    nest_status_t st = plan_search(ds, B, r, seg_off != nullptr, &sp);
    if (st != NEST_OK) return st;
    st = ensure_scratch(ds, sp.total_words);
    if (st != NEST_OK) return st;
    return launch_search(ds, q, B, r, seg_off, key_mask, s_out, idx_out, ds->scratch,
                         ds->scratch_words, ds->timing, stream);
}

nest_status_t run_mix(nest_datastore* ds, const float* s_in, const int64_t* idx_in,
                      const float* p_lm, int32_t B, int32_t r, float mu, float lambda, int rrc,
                      float alpha, float tau, float* lam_out, float* p_knn_out, float* p_m_out,
                      cudaStream_t stream)
{
    MixArgs m{};
    m.s = s_in;
    m.idx = idx_in;
    m.V = ds->V;
    m.p_lm = p_lm;
    m.p_knn = p_knn_out;
    m.p_m = p_m_out;
    m.lam_out = lam_out;
    m.status = ds->status;
    m.N = ds->N;
    m.vocab = ds->vocab;
    m.B = B;
    m.r = r;
    m.mu = mu;
    m.lambda = lambda;
    m.rrc = rrc;
    m.alpha = alpha;
    m.tau = tau;
    // Enough CTAs to stream the vocabulary rows, at least one per query.
    const int64_t want = std::max<int64_t>(1, (2LL * ds->num_sms + B - 1) / B);
    const int64_t by_vocab = std::max<int64_t>(1, ds->vocab / 2048);
    m.slices = (int32_t)std::max<int64_t>(mix_min_slices(ds->vocab),
                                          std::min<int64_t>(want, by_vocab));
    cudaError_t e = launch_mix(m, stream);
    if (e != cudaSuccess) return from_cuda(e);
    ++ds->launches;
    return NEST_OK;
}

}  // namespace

extern "C" {

nest_status_t nest_datastore_create(const void* K, const int32_t* V, int64_t N, int32_t d,
                                    nest_dtype_t dtype, int32_t vocab, void* stream,
                                    nest_datastore_t** out)
{
    if (!out) return NEST_ERR_INVALID_ARG;
    *out = nullptr;
    if (!K || !V) return NEST_ERR_INVALID_ARG;
    if (dtype != NEST_F32 && dtype != NEST_BF16) return NEST_ERR_DTYPE;
    if (N < 1 || N > kMaxKeys || d < 1 || vocab < 1) return NEST_ERR_INVALID_ARG;
    const int64_t row_bytes = (int64_t)d * element_size(dtype);
    if (row_bytes > NEST_MAX_ROW_BYTES) return NEST_ERR_UNSUPPORTED;
    if (row_bytes % 16 != 0 || !aligned(K, 16) || !aligned(V, 4)) return NEST_ERR_ALIGN;
    if (!is_device_pointer(K) || !is_device_pointer(V)) return NEST_ERR_INVALID_ARG;

    nest_datastore* ds = new (std::nothrow) nest_datastore();
    if (!ds) return NEST_ERR_OOM;
    ds->K = K;
    ds->V = V;
    ds->N = N;
    ds->d = d;
    ds->dtype = dtype;
    ds->vocab = vocab;
    ds->row_bytes = (int32_t)row_bytes;
    cudaError_t e = cudaGetDevice(&ds->device);
    int optin = 0;
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&ds->num_sms, cudaDevAttrMultiProcessorCount, ds->device);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ds->device);
    ds->smem_optin = (size_t)optin;
    if (e == cudaSuccess) e = cudaMalloc(reinterpret_cast<void**>(&ds->knorm), (size_t)N * sizeof(float));
    if (e == cudaSuccess) e = cudaMalloc(reinterpret_cast<void**>(&ds->status), sizeof(int));
    cudaStream_t st = as_stream(stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(ds->status, 0, sizeof(int), st);
    if (e == cudaSuccess) e = launch_key_norms(K, N, d, dtype, ds->knorm, st);
    if (e == cudaSuccess) e = launch_check_values(V, N, vocab, ds->status, st);
    int host_status = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&host_status, ds->status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        nest_datastore_destroy(ds);
        return e == cudaErrorMemoryAllocation ? NEST_ERR_OOM : NEST_ERR_CUDA;
    }
    ds->launches = 2;
    // Tensor-core scan: bf16 keys whose row indices fit TMA's 32-bit coordinates.
    if (dtype == NEST_BF16 && N <= (int64_t)0x7FFFFF00)
        ds->tc = encode_bf16_rows(&ds->keys_map, K, N, d, kTcTileKeys, true);
    ds->pairs_ok = ds->tc && wide_pair_clusters(ds->smem_optin) > 0;
    ds->pairs_mode = -1;  // automatic: nest_datastore_use_cta_pairs
    if (host_status != 0) {
        nest_datastore_destroy(ds);
        return static_cast<nest_status_t>(host_status);
    }
    *out = ds;
    return NEST_OK;
}

nest_status_t nest_datastore_destroy(nest_datastore_t* ds)
{
    if (!ds) return NEST_OK;
    cudaError_t first = cudaSuccess;
    auto keep = [&](cudaError_t e) {
        if (first == cudaSuccess) first = e;
    };
    if (ds->knorm) keep(cudaFree(ds->knorm));
    if (ds->status) keep(cudaFree(ds->status));
    if (ds->scratch) keep(cudaFree(ds->scratch));
    if (ds->host_stage) keep(cudaFree(ds->host_stage));
    if (ds->host_status) keep(cudaFreeHost(ds->host_status));
    for (cudaEvent_t ev : ds->aux_ev)
        if (ev) keep(cudaEventDestroy(ev));
    if (ds->aux) keep(cudaStreamDestroy(ds->aux));
    for (cudaEvent_t ev : ds->events) keep(cudaEventDestroy(ev));
    delete ds;
    return from_cuda(first);
}

nest_status_t nest_datastore_reserve(nest_datastore_t* ds, int32_t max_B, int32_t max_r,
                                     int32_t ragged)
{
    if (!ds || max_B < 1 || max_B > kMaxB || max_r < 1 || max_r > NEST_MAX_R)
        return NEST_ERR_INVALID_ARG;
    size_t need = 0;
    for (int r = 1; r <= max_r; r = (r == max_r) ? max_r + 1 : std::min(max_r, r * 2)) {
        for (int B = 1; B <= max_B; B = (B == max_B) ? max_B + 1 : std::min(max_B, B * 2)) {
            SearchPlan sp;
            if (plan_search(ds, B, r, ragged != 0, &sp) == NEST_OK)
                need = std::max(need, sp.total_words);
        }
    }
    return ensure_scratch(ds, need);
}

nest_status_t nest_datastore_use_cta_pairs(nest_datastore_t* ds, int32_t mode)
{
    if (!ds || mode < -1 || mode > 1) return NEST_ERR_INVALID_ARG;
    if (mode == 1 && !ds->pairs_ok) return NEST_ERR_UNSUPPORTED;
    ds->pairs_mode = mode;
    return NEST_OK;
}

nest_status_t nest_knn_search(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                              const int64_t* seg_off, float* s_out, int64_t* idx_out, void* stream)
{
    nest_status_t st = check_search_args(ds, q, B, r, seg_off, s_out, idx_out);
    if (st == NEST_OK) st = check_device(ds);
    if (st != NEST_OK) return st;
    return run_search(ds, q, B, r, seg_off, s_out, idx_out, as_stream(stream));
}

nest_status_t nest_knn_mix(nest_datastore_t* ds, const float* s_in, const int64_t* idx_in,
                           const float* p_lm, int32_t B, int32_t r, float mu, float lambda,
                           float* p_knn_out, float* p_m_out, void* stream)
{
    nest_status_t st = check_mix_args(ds, s_in, idx_in, p_lm, B, r, p_knn_out, p_m_out);
    if (st != NEST_OK) return st;
    if (!(lambda >= 0.f && lambda <= 1.f)) return NEST_ERR_INVALID_ARG;
    return run_mix(ds, s_in, idx_in, p_lm, B, r, mu, lambda, 0, 0.f, 1.f, nullptr, p_knn_out,
                   p_m_out, as_stream(stream));
}

nest_status_t nest_knn_mix_rrc(nest_datastore_t* ds, const float* s_in, const int64_t* idx_in,
                               const float* p_lm, int32_t B, int32_t r, float mu, float alpha,
                               float tau, float* lambda_out, float* p_knn_out, float* p_m_out,
                               void* stream)
{
    nest_status_t st = check_mix_args(ds, s_in, idx_in, p_lm, B, r, p_knn_out, p_m_out);
    if (st != NEST_OK) return st;
    if (!(tau > 0.f) || alpha != alpha) return NEST_ERR_INVALID_ARG;
    if (lambda_out && !aligned(lambda_out, 4)) return NEST_ERR_ALIGN;
    return run_mix(ds, s_in, idx_in, p_lm, B, r, mu, 0.f, 1, alpha, tau, lambda_out, p_knn_out,
                   p_m_out, as_stream(stream));
}

nest_status_t nest_knn_step(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                            const int64_t* seg_off, const float* p_lm, float mu, float lambda,
                            float* s_out, int64_t* idx_out, float* p_knn_out, float* p_m_out,
                            void* stream)
{
    nest_status_t st = check_search_args(ds, q, B, r, seg_off, s_out, idx_out);
    if (st != NEST_OK) return st;
    st = check_mix_args(ds, s_out, idx_out, p_lm, B, r, p_knn_out, p_m_out);
    if (st != NEST_OK) return st;
    if (!(lambda >= 0.f && lambda <= 1.f)) return NEST_ERR_INVALID_ARG;
    if ((st = check_device(ds)) != NEST_OK) return st;
    cudaStream_t s = as_stream(stream);
    st = run_search(ds, q, B, r, seg_off, s_out, idx_out, s);
    if (st != NEST_OK) return st;
    return run_mix(ds, s_out, idx_out, p_lm, B, r, mu, lambda, 0, 0.f, 1.f, nullptr, p_knn_out,
                   p_m_out, s);
}

nest_status_t nest_knn_step_host(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                                 const int64_t* seg_off, const float* p_lm, float mu,
                                 float lambda, float* s_out, int64_t* idx_out, float* p_m_out,
                                 void* stream)
{
    if (!ds || !q || !p_lm || !s_out || !idx_out || !p_m_out) return NEST_ERR_INVALID_ARG;
    if (B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R) return NEST_ERR_INVALID_ARG;
    if (!(lambda >= 0.f && lambda <= 1.f)) return NEST_ERR_INVALID_ARG;
    const size_t q_bytes = (size_t)B * ds->row_bytes;
    const size_t so_bytes = seg_off ? (size_t)(B + 1) * 8 : 0;
    const size_t v_bytes = (size_t)B * ds->vocab * 4;
    const size_t s_bytes = (size_t)B * r * 4, i_bytes = (size_t)B * r * 8;
    const size_t off_so = round256(q_bytes), off_p = off_so + round256(so_bytes);
    const size_t off_s = off_p + round256(v_bytes), off_i = off_s + round256(s_bytes);
    const size_t off_m = off_i + round256(i_bytes), total = off_m + round256(v_bytes);
    nest_status_t st = ensure_host_stage(ds, total);
    if (st == NEST_OK) st = ensure_aux(ds);
    if (st != NEST_OK) return st;
    unsigned char* d = ds->host_stage;
    const int64_t* d_so = seg_off ? reinterpret_cast<const int64_t*>(d + off_so) : nullptr;
    const float* d_p = reinterpret_cast<const float*>(d + off_p);
    float* d_s = reinterpret_cast<float*>(d + off_s);
    int64_t* d_i = reinterpret_cast<int64_t*>(d + off_i);
    float* d_m = reinterpret_cast<float*>(d + off_m);
    cudaStream_t s = as_stream(stream), x = ds->aux;
    cudaEvent_t ev_start = ds->aux_ev[0], ev_lm = ds->aux_ev[1], ev_search = ds->aux_ev[2];
    // the queries go in on `stream` ahead of the search; p_LM goes in on the
    // side stream while the search runs, and s / idx come back on it while
    // the mix runs
    cudaError_t e = cudaEventRecord(ev_start, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(x, ev_start, 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(d, q, q_bytes, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess && seg_off)
        e = cudaMemcpyAsync(d + off_so, seg_off, so_bytes, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(d + off_p, p_lm, v_bytes, cudaMemcpyHostToDevice, x);
    if (e == cudaSuccess) e = cudaEventRecord(ev_lm, x);
    if (e != cudaSuccess) return from_cuda(e);
    st = nest_knn_search(ds, d, B, r, d_so, d_s, d_i, stream);
    if (st != NEST_OK) {
        (void)cudaStreamSynchronize(x);
        return st;
    }
    e = cudaEventRecord(ev_search, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(x, ev_search, 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(s_out, d_s, s_bytes, cudaMemcpyDeviceToHost, x);
    if (e == cudaSuccess) e = cudaMemcpyAsync(idx_out, d_i, i_bytes, cudaMemcpyDeviceToHost, x);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ev_lm, 0);
    if (e != cudaSuccess) {
        (void)cudaStreamSynchronize(x);
        return from_cuda(e);
    }
    st = nest_knn_mix(ds, d_s, d_i, d_p, B, r, mu, lambda, nullptr, d_m, stream);
    if (st == NEST_OK) e = cudaMemcpyAsync(p_m_out, d_m, v_bytes, cudaMemcpyDeviceToHost, s);
    // the device status comes back with the results (and is cleared), so a
    // condition the kernels recorded is this call's return value
    if (st == NEST_OK && e == cudaSuccess)
        e = cudaMemcpyAsync(ds->host_status, ds->status, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (st == NEST_OK && e == cudaSuccess) e = cudaMemsetAsync(ds->status, 0, sizeof(int), s);
    const cudaError_t es = cudaStreamSynchronize(s);
    const cudaError_t ex = cudaStreamSynchronize(x);
    if (st != NEST_OK) return st;
    if (e == cudaSuccess) e = es;
    if (e == cudaSuccess) e = ex;
    if (e != cudaSuccess) return from_cuda(e);
    return static_cast<nest_status_t>(*ds->host_status);
}

nest_status_t nest_knn_search_masked(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                                     const int64_t* seg_off, const uint32_t* key_mask,
                                     float* s_out, int64_t* idx_out, void* stream)
{
    nest_status_t st = check_search_args(ds, q, B, r, seg_off, s_out, idx_out);
    if (st != NEST_OK) return st;
    if (!key_mask) return NEST_ERR_INVALID_ARG;
    if (!aligned(key_mask, 4)) return NEST_ERR_ALIGN;
    if ((st = check_device(ds)) != NEST_OK) return st;
    return run_search(ds, q, B, r, seg_off, s_out, idx_out, as_stream(stream), key_mask);
}

nest_status_t nest_mask_keys(nest_datastore_t* ds, uint32_t* key_mask, int64_t first_key,
                             int64_t count, void* stream)
{
    if (!ds || !key_mask || first_key < 0 || count < 0 || first_key > ds->N - count)
        return NEST_ERR_INVALID_ARG;
    if (!aligned(key_mask, 4)) return NEST_ERR_ALIGN;
    const cudaError_t e = launch_mask(key_mask, first_key, count, as_stream(stream));
    if (e != cudaSuccess) return from_cuda(e);
    if (count > 0) ++ds->launches;
    return NEST_OK;
}

nest_status_t nest_knn_decide(nest_datastore_t* ds, const float* p_m, const float* s_in,
                              const int64_t* idx_in, const float* lambda, int32_t B, int32_t r,
                              float delta, int32_t* token_out, float* p_max_out,
                              int64_t* span_key_out, int32_t* use_span_out, void* stream)
{
    if (!ds || !p_m || !s_in || !idx_in || !lambda || !token_out || !p_max_out || !span_key_out ||
        !use_span_out)
        return NEST_ERR_INVALID_ARG;
    if (B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R || delta != delta) return NEST_ERR_INVALID_ARG;
    if (!aligned(p_m, 4) || !aligned(s_in, 4) || !aligned(idx_in, 8) || !aligned(lambda, 4) ||
        !aligned(token_out, 4) || !aligned(p_max_out, 4) || !aligned(span_key_out, 8) ||
        !aligned(use_span_out, 4))
        return NEST_ERR_ALIGN;
    DecideArgs a{};
    a.p_m = p_m;
    a.s = s_in;
    a.idx = idx_in;
    a.V = ds->V;
    a.lambda = lambda;
    a.status = ds->status;
    a.N = ds->N;
    a.vocab = ds->vocab;
    a.B = B;
    a.r = r;
    a.delta = delta;
    a.token = token_out;
    a.p_max = p_max_out;
    a.span_key = span_key_out;
    a.use_span = use_span_out;
    const cudaError_t e = launch_decide(a, as_stream(stream));
    if (e != cudaSuccess) return from_cuda(e);
    ++ds->launches;
    return NEST_OK;
}

nest_status_t nest_verify_spans(nest_datastore_t* ds, const float* p_m, const int32_t* draft,
                                int32_t rows, const int32_t* span_off, int32_t spans, float gamma,
                                float* ratio_out, int32_t* accept_out, int32_t* n_accept_out,
                                void* stream)
{
    if (!ds || !p_m || !draft || !span_off || !ratio_out || !accept_out || !n_accept_out)
        return NEST_ERR_INVALID_ARG;
    if (rows < 1 || rows > kMaxB || spans < 1 || spans > kMaxB || !(gamma > 0.f))
        return NEST_ERR_INVALID_ARG;
    if (!aligned(p_m, 4) || !aligned(draft, 4) || !aligned(span_off, 4) || !aligned(ratio_out, 4) ||
        !aligned(accept_out, 4) || !aligned(n_accept_out, 4))
        return NEST_ERR_ALIGN;
    VerifyArgs a{};
    a.p_m = p_m;
    a.draft = draft;
    a.span_off = span_off;
    a.status = ds->status;
    a.vocab = ds->vocab;
    a.rows = rows;
    a.spans = spans;
    a.gamma = gamma;
    a.ratio = ratio_out;
    a.accept = accept_out;
    a.n_accept = n_accept_out;
    const cudaError_t e = launch_verify(a, as_stream(stream));
    if (e != cudaSuccess) return from_cuda(e);
    ds->launches += 2;
    return NEST_OK;
}

nest_status_t nest_selftest_bounded_wait(nest_datastore_t* ds, int64_t* waited_ns, void* stream)
{
    if (!ds) return NEST_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    int64_t* d_ns = nullptr;
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&d_ns), sizeof(int64_t));
    if (e == cudaSuccess) e = launch_wait_selftest(ds->status, d_ns, st);
    int64_t h_ns = 0;
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(&h_ns, d_ns, sizeof(int64_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (d_ns) (void)cudaFree(d_ns);
    if (e != cudaSuccess) return from_cuda(e);
    ++ds->launches;
    if (waited_ns) *waited_ns = h_ns;
    return NEST_OK;
}

nest_status_t nest_device_status(nest_datastore_t* ds, void* stream)
{
    if (!ds) return NEST_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    int h = 0;
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemcpy(&h, ds->status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(ds->status, 0, sizeof(int));
    if (e != cudaSuccess) return from_cuda(e);
    return static_cast<nest_status_t>(h);
}

nest_status_t nest_timing_enable(nest_datastore_t* ds, int32_t on)
{
    if (!ds) return NEST_ERR_INVALID_ARG;
    ds->timing = on != 0;
    return NEST_OK;
}

nest_status_t nest_timing_read(nest_datastore_t* ds, double* total_ms, int64_t* launches)
{
    if (!ds || !total_ms || !launches) return NEST_ERR_INVALID_ARG;
    double sum = 0.0;
    const size_t pairs = ds->events_used / 2;
    for (size_t i = 0; i < pairs; ++i) {
        cudaError_t e = cudaEventSynchronize(ds->events[2 * i + 1]);
        float ms = 0.f;
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, ds->events[2 * i], ds->events[2 * i + 1]);
        if (e != cudaSuccess) return from_cuda(e);
        sum += ms;
    }
    *total_ms = sum;
    *launches = (int64_t)pairs;
    ds->events_used = 0;
    return NEST_OK;
}

int64_t nest_launch_count(const nest_datastore_t* ds) { return ds ? ds->launches : 0; }

nest_status_t nest_plan_offline(int64_t N, int32_t d, nest_dtype_t dtype, int32_t B, int32_t r,
                                int32_t ragged, int32_t num_sms, int64_t smem_per_block,
                                int32_t cta_pairs, nest_plan_t* out)
{
    if (!out) return NEST_ERR_INVALID_ARG;
    if (dtype != NEST_F32 && dtype != NEST_BF16) return NEST_ERR_DTYPE;
    if (N < 1 || N > kMaxKeys || d < 1 || B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R ||
        num_sms < 2 || smem_per_block < 1)
        return NEST_ERR_INVALID_ARG;
    const int64_t row_bytes = (int64_t)d * element_size(dtype);
    if (row_bytes > NEST_MAX_ROW_BYTES) return NEST_ERR_UNSUPPORTED;
    if (row_bytes % 16 != 0) return NEST_ERR_ALIGN;
    nest_datastore ds;
    ds.N = N;
    ds.d = d;
    ds.dtype = dtype;
    ds.row_bytes = (int32_t)row_bytes;
    ds.num_sms = num_sms;
    ds.smem_optin = (size_t)smem_per_block;
    // the key tensor map encodes for every such bf16 datastore (16-byte rows)
    ds.tc = dtype == NEST_BF16 && N <= (int64_t)0x7FFFFF00;
    if (cta_pairs < -1 || cta_pairs > 1) return NEST_ERR_INVALID_ARG;
    ds.pairs_ok = ds.tc;
    ds.pairs_mode = cta_pairs;
    SearchPlan sp;
    const nest_status_t st = plan_search(&ds, B, r, ragged != 0, &sp);
    if (st != NEST_OK) return st;
    nest_plan_t p{};
    p.path = sp.wide ? (sp.wpm.pair ? 4 : (sp.wpm.mb == 2 ? 3 : 2)) : (sp.tc ? 1 : (sp.rows ? 5 : 0));
    if (sp.wide) {
        p.queries_per_group = sp.wpm.nm;
        p.groups = sp.wpm.groups;
        p.parts = sp.wpm.parts;
        p.stages = sp.wpm.stages;
        p.single_pass = sp.single_pass ? 1 : 0;
        p.sample_stride = sp.stride;
        p.list_capacity = sp.single_pass ? sp.cap_s : sp.cap_m;
    } else {
        p.queries_per_group = sp.nq;
        p.groups = sp.groups;
        p.parts = sp.parts;
        p.stages = sp.tc ? sp.tcp.stages : sp.scan.stages;
        p.list_capacity = sp.tc ? sp.tcp.cap : sp.scan.cap;
    }
    p.scratch_bytes = (int64_t)(sp.total_words * sizeof(uint64_t));
    *out = p;
    return NEST_OK;
}

int32_t nest_search_path(const nest_datastore_t* ds, int32_t B, int32_t r, int32_t ragged)
{
    if (!ds || B < 1 || B > kMaxB || r < 1 || r > NEST_MAX_R) return -(int32_t)NEST_ERR_INVALID_ARG;
    SearchPlan sp;
    const nest_status_t st = plan_search(ds, B, r, ragged != 0, &sp);
    if (st != NEST_OK) return -(int32_t)st;
    return sp.wide ? (sp.wpm.pair ? 4 : (sp.wpm.mb == 2 ? 3 : 2)) : (sp.tc ? 1 : (sp.rows ? 5 : 0));
}

const char* nest_status_string(nest_status_t s)
{
    switch (s) {
    case NEST_OK: return "ok";
    case NEST_ERR_INVALID_ARG: return "invalid argument";
    case NEST_ERR_DTYPE: return "unknown element type";
    case NEST_ERR_ALIGN: return "pointer or row not 16-byte aligned";
    case NEST_ERR_OOM: return "device allocation failed";
    case NEST_ERR_CUDA: return "CUDA runtime error";
    case NEST_ERR_VALUE_RANGE: return "token id or key index out of range";
    case NEST_ERR_OVERFLOW: return "device buffer overflow";
    case NEST_ERR_TIMEOUT: return "device wait timed out";
    case NEST_ERR_UNSUPPORTED: return "shape not supported";
    case NEST_ERR_MARGIN: return "exact re-ranking could not confirm the r-th neighbour";
    }
    return "unknown status";
}

int32_t nest_version(void) { return 300; }

}  // extern "C"

// ---------------------------------------------------------------- caller-provided scratch
// Used by the allocation-free search entry point (noalloc.cu): the same plan
// and kernels as nest_knn_search, with the candidate lists placed in memory
// the caller of these helpers owns.
namespace nest {

nest_status_t search_scratch_words(const nest_datastore* ds, int32_t B, int32_t r, bool ragged,
                                   size_t* words)
{
    SearchPlan sp;
    nest_status_t st = plan_search(ds, B, r, ragged, &sp);
    if (st != NEST_OK) return st;
    *words = sp.total_words;
    return NEST_OK;
}

nest_status_t check_search_call(const nest_datastore* ds, const void* q, int32_t B, int32_t r,
                                const int64_t* seg_off, const float* s_out,
                                const int64_t* idx_out)
{
    nest_status_t st = check_search_args(ds, q, B, r, seg_off, s_out, idx_out);
    if (st == NEST_OK) st = check_device(ds);
    return st;
}

nest_status_t search_with_scratch(nest_datastore* ds, const void* q, int32_t B, int32_t r,
                                  const int64_t* seg_off, float* s_out, int64_t* idx_out,
                                  uint64_t* scratch, size_t scratch_words, cudaStream_t stream)
{
    nest_status_t st = check_search_call(ds, q, B, r, seg_off, s_out, idx_out);
    if (st != NEST_OK) return st;
    return launch_search(ds, q, B, r, seg_off, nullptr, s_out, idx_out, scratch, scratch_words,
                         ds->timing, stream);
}

}  // namespace nest
