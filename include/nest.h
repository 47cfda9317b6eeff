/*
 * nest.h -- C ABI of the GB300 kNN-LM step of Nearest Neighbor Speculative
 * Decoding (NEST, arXiv 2405.19325).
 *
 * One step of the method, for a batch of B LM hidden states q (the queries):
 *
 *   search  s(q, k) = -||q - k||^2 against every datastore key k, or, for the
 *           second stage of NEST's two-stage search, against a per-query
 *           candidate segment of the keys (Sec. 2.2; Sec. 3.1; App. A), and
 *           keep the r nearest neighbours pi (Sec. 2.2; search step of
 *           Algorithm 1);
 *   mix     p_kNN(w) proportional to sum over pi of 1[w = v_i] exp(mu s_i)
 *           (Eq. 2), then p_M = lambda p_LM + (1 - lambda) p_kNN (Eq. 3), or
 *           with lambda replaced by the relative retrieval confidence
 *           lambda_t of Eq. 4.
 *
 * Conventions shared by every call:
 *   - Array arguments are DEVICE pointers on the current CUDA device, owned
 *     by the caller, unless a comment says otherwise.  Matrices are dense and
 *     row-major.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  All work is stream-ordered and no call synchronizes, except
 *     nest_datastore_create, nest_datastore_destroy, nest_knn_step_host,
 *     nest_device_status, nest_selftest_bounded_wait and nest_timing_read,
 *     and a call that allocates scratch (nest_datastore_reserve, or the
 *     first search of a larger shape without it); each says so.
 *   - Keys and queries are NEST_F32 or NEST_BF16 (IEEE bfloat16 bits).
 *     Distances, similarities and probabilities are fp32.
 *   - Argument errors are found on the host before anything is launched and
 *     are returned synchronously.  Conditions only the GPU can see (a bad
 *     segment offset, an out-of-range neighbour index, a wait that ran out
 *     of time) are recorded in a per-datastore device status word and
 *     reported by nest_device_status.
 *   - A datastore handle is not safe for concurrent calls from several
 *     streams or threads: its scratch memory is shared by its calls.
 */
#ifndef NEST_H
#define NEST_H

#include <stdint.h>

#if defined(__GNUC__)
#define NEST_API __attribute__((visibility("default")))
#else
#define NEST_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum nest_status {
    NEST_OK = 0,
    NEST_ERR_INVALID_ARG = 1,  /* null pointer, size out of range, bad lambda/tau */
    NEST_ERR_DTYPE = 2,        /* unknown element type */
    NEST_ERR_ALIGN = 3,        /* pointer or row not 16-byte aligned */
    NEST_ERR_OOM = 4,          /* device allocation failed */
    NEST_ERR_CUDA = 5,         /* a CUDA runtime call failed */
    NEST_ERR_VALUE_RANGE = 6,  /* token id outside [0, vocab) or key index outside [0, N) */
    NEST_ERR_OVERFLOW = 7,     /* a search needs more than a fixed-size scratch buffer holds */
    NEST_ERR_TIMEOUT = 8,      /* a device-side wait gave up */
    NEST_ERR_UNSUPPORTED = 9,  /* shape outside what the kernels handle */
    NEST_ERR_MARGIN = 10       /* exact re-ranking could not confirm a query's r-th neighbour */
} nest_status_t;

typedef enum nest_dtype { NEST_F32 = 0, NEST_BF16 = 1 } nest_dtype_t;

/* Largest r accepted by the search. */
#define NEST_MAX_R 4096
/* Largest row of a key or query, in bytes (d * element size). */
#define NEST_MAX_ROW_BYTES 16384

typedef struct nest_datastore nest_datastore_t;

/*
 * Register a key-value datastore (K, V) (Sec. 2.2, Eq. 1: key k_i = hidden
 * state f(c_i), value v_i = the next token w_i).
 *
 *   K      N x d keys, element type `dtype`; 16-byte aligned, and a row
 *          (d * element size bytes) must be a multiple of 16 bytes and at
 *          most NEST_MAX_ROW_BYTES.
 *   V      N token ids (int32), each in [0, vocab).
 *   N      number of keys, 1 <= N <= 2^32 - 2.
 *   vocab  vocabulary size of p_LM / p_kNN / p_M, >= 1.
 *   out    receives the handle.
 *
 * K and V are BORROWED: the caller keeps them alive and unchanged until
 * nest_datastore_destroy.  The handle owns the fp32 key norms ||k_i||^2
 * (computed here, N * 4 bytes), a device status word and the scratch memory
 * of later calls.  This call synchronizes `stream`: it checks every value
 * on the device and returns NEST_ERR_VALUE_RANGE if one is out of range.
 */
NEST_API nest_status_t nest_datastore_create(const void* K, const int32_t* V, int64_t N, int32_t d,
                                    nest_dtype_t dtype, int32_t vocab, void* stream,
                                    nest_datastore_t** out);

/* Free everything the handle owns (synchronizes the device).  NULL is a no-op. */
NEST_API nest_status_t nest_datastore_destroy(nest_datastore_t* ds);

/*
 * Allocate the handle's scratch memory for searches of up to max_B queries
 * and r <= max_r, so that such searches allocate nothing (for instance
 * before stream capture).  Without it the first search of a larger shape
 * allocates.  Synchronizes the device when it allocates.
 */
NEST_API nest_status_t nest_datastore_reserve(nest_datastore_t* ds, int32_t max_B, int32_t max_r,
                                     int32_t ragged);

/*
 * How searches of more than 128 queries are laid out on the SMs (search
 * paths 3 and 4 of nest_search_path).  Both return the same neighbours.
 *
 *   mode  1  always on CTA pairs (path 4): each 256-key tile is split over
 *            the two SMs of a pair and each CTA stages only half of each
 *            256-query block, so a pipeline stage carries the MMA work of a
 *            path-3 stage in three quarters of the shared memory (four
 *            stages instead of three).  Batches of 257 to 512 queries run as
 *            one group of 512 (one 256-key tile against both halves per
 *            stage); other batches as groups of 256 (two 256-key tiles per
 *            stage).
 *   mode  0  never: single CTAs with two 128-key tiles per stage and groups
 *            of 256 queries (path 3).
 *   mode -1  automatic, the default: pairs when the batch is one group
 *            (129 to 512 queries), single CTAs for more.  On a GB300, pairs
 *            made the main pass about 5 % faster at d = 8192, 8M keys,
 *            B = 256, and about 3 % faster at d = 4096, 4M keys, B = 512
 *            (every key read from DRAM once instead of once per group of
 *            256).  Two or more pair groups drift apart over the same keys
 *            and read them from DRAM again, so larger batches stay on single
 *            CTAs, whose four or more groups share the keys in L2.
 *
 * Pairs need two CTAs of about 220 KiB of shared memory each on the two SMs
 * of one TPC at the same time; mode 1 where the device cannot place them
 * returns NEST_ERR_UNSUPPORTED and changes nothing, and mode -1 there runs
 * single CTAs.  Any other mode returns NEST_ERR_INVALID_ARG.  Host only;
 * takes effect from the next search, which may need more scratch than
 * nest_datastore_reserve set aside.
 */
NEST_API nest_status_t nest_datastore_use_cta_pairs(nest_datastore_t* ds, int32_t mode);

/*
 * r-nearest-neighbour search (Sec. 2.2; Sec. 3.1 second stage; App. A).
 *
 *   q        B x d queries, the datastore's element type, 16-byte aligned.
 *   B        1 <= B <= 65535.
 *   r        1 <= r <= NEST_MAX_R.
 *   seg_off  NULL: every query scans all N keys.  Otherwise B + 1 int64
 *            offsets: query b scans only keys [seg_off[b], seg_off[b+1])
 *            (its on-the-fly datastore K', given as a segment of K).
 *            Offsets must satisfy 0 <= seg_off[b] <= seg_off[b+1] <= N; a
 *            violating segment is searched as empty and recorded as
 *            NEST_ERR_INVALID_ARG in the device status.
 *   s_out    B x r fp32: s = -||q - k||^2 of the neighbours, nearest first
 *            (s descending, ties by smaller key index).
 *   idx_out  B x r int64 global key indices of the neighbours.
 *
 * When a query has fewer than r candidate keys the tail of its row is
 * padded with s = -inf and idx = -1.
 *
 * Distances: every key is screened by ||q||^2 + ||k||^2 - 2 q.k evaluated in
 * fp32 (tensor cores for bf16 keys), whose rounding error is absolute in the
 * norms.  Each query keeps its r' = r + m nearest screened keys
 * (m = r / 16, at least 16 and at most 128), their distances are recomputed
 * as sums of squared differences of the stored elements in fp32 (error a
 * few units in the last place of the distance itself; exactly 0 for a key
 * equal to the query), and the r nearest by those are returned.  If more
 * than m keys lie within the screening error of the r-th distance, a key
 * outside the r' might belong to the r nearest: this is detected from the
 * screening errors seen among the r' (see refine.cu) and recorded as
 * NEST_ERR_MARGIN in the device status; the row then holds the r nearest of
 * the r' candidates.
 */
NEST_API nest_status_t nest_knn_search(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                              const int64_t* seg_off, float* s_out, int64_t* idx_out,
                              void* stream);

/*
 * nest_knn_search without any device allocation (the paper has no
 * counterpart: this is a deployment variant of the search above).
 *
 * nest_knn_search places its candidate lists in scratch memory that the
 * handle allocates with cudaMalloc on first use and re-allocates when a
 * larger search comes; cudaMalloc and cudaFree synchronize the device and
 * draw on memory that a framework's own allocator may already own.  Callers
 * that must not allocate -- for example a serving loop that may never stall
 * the device, or an application whose allocator owns all device memory --
 * call this instead.  It runs the same kernels and writes the same outputs,
 * with the candidate lists in one fixed 8 MiB array compiled into the
 * library, which every GPU that loads the library holds until the process
 * exits.
 *
 *   Arguments, outputs and device-side errors are those of nest_knn_search.
 *   Returns NEST_ERR_OVERFLOW, before launching anything, when the search
 *   needs more than the 2^20 candidate words (8 MiB) of the array; the
 *   decode and second-stage workloads need far less (1M keys, B = 4,
 *   r = 1024: about 0.65M words).
 *   The first call on each device looks up the array's device address
 *   (cudaGetSymbolAddress) with that device current; make that first call
 *   before any stream capture.
 *   All calls on a device share the one array and it keeps what the last
 *   call left in it (no call relies on it starting at zero): calls that
 *   overlap on the GPU, from different streams or threads, race with each
 *   other and must be serialized by the caller.
 */
NEST_API nest_status_t nest_knn_search_static(nest_datastore_t* ds, const void* q, int32_t B,
                                              int32_t r, const int64_t* seg_off, float* s_out,
                                              int64_t* idx_out, void* stream);

/*
 * Eq. 2 and Eq. 3 for each query row b < B:
 *
 *   p_kNN[b][w] = sum_{i : V[idx_in[b][i]] = w} exp(mu s_i) / sum_j exp(mu s_j)
 *   p_M[b][w]   = lambda p_LM[b][w] + (1 - lambda) p_kNN[b][w]
 *
 *   s_in, idx_in  B x r neighbours as written by nest_knn_search (entries
 *                 with idx < 0 or s = -inf carry no weight; an index >= N
 *                 is recorded as NEST_ERR_VALUE_RANGE and skipped).
 *   p_lm          B x vocab fp32.
 *   mu            inverse temperature (the paper uses 1/sqrt(d)).
 *   lambda        in [0, 1].
 *   p_knn_out     B x vocab fp32, or NULL when not wanted.
 *   p_m_out       B x vocab fp32.
 *
 * A row with no real neighbour gets p_kNN = 0 and p_M = p_LM (lambda is
 * taken as 1).  The softmax subtracts the largest s first, which leaves the
 * result unchanged in exact arithmetic.
 */
NEST_API nest_status_t nest_knn_mix(nest_datastore_t* ds, const float* s_in, const int64_t* idx_in,
                           const float* p_lm, int32_t B, int32_t r, float mu, float lambda,
                           float* p_knn_out, float* p_m_out, void* stream);

/*
 * As nest_knn_mix, with each row's lambda replaced by the relative
 * retrieval confidence of Eq. 4 (Sec. 3.2):
 *
 *   lambda_t = sigmoid((min_i |s_i| / max_i |s_i| - alpha) / tau)
 *
 * over the row's real neighbours (Eq. 4 takes absolute values, which the
 * restatement in Algorithm 1 drops; Eq. 4 is followed).  tau > 0.  A row
 * with no real neighbour gets lambda_t = 1; a row whose neighbours all have
 * s = 0 takes the ratio as 1.  lambda_out (B fp32, or NULL) receives
 * lambda_t.
 */
NEST_API nest_status_t nest_knn_mix_rrc(nest_datastore_t* ds, const float* s_in, const int64_t* idx_in,
                               const float* p_lm, int32_t B, int32_t r, float mu, float alpha,
                               float tau, float* lambda_out, float* p_knn_out, float* p_m_out,
                               void* stream);

/*
 * One kNN-LM step: nest_knn_search followed by nest_knn_mix on `stream`,
 * with the same arguments and outputs (s_out and idx_out are required; they
 * carry the neighbours from the search to the mix).
 */
NEST_API nest_status_t nest_knn_step(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                            const int64_t* seg_off, const float* p_lm, float mu, float lambda,
                            float* s_out, int64_t* idx_out, float* p_knn_out, float* p_m_out,
                            void* stream);

/*
 * nest_knn_step from host memory: the query batch, the segment offsets (or
 * NULL) and p_LM are copied to device buffers the handle owns, the step runs
 * on `stream`, and p_M, s and idx are copied back; the call returns once
 * `stream` has finished (or with the first error).  Same arguments as
 * nest_knn_step except that every pointer is a host pointer (page-locked
 * memory lets the copies run asynchronously; pageable memory works but the
 * driver stages it) and no p_kNN is returned.
 *
 * p_LM goes in, and s and idx come back, on a side stream the handle owns
 * (ordered with `stream` by events), so those copies overlap the search and
 * the mix.  The device buffers grow on demand with cudaMalloc, the side
 * stream is created on the first call, and nest_datastore_destroy frees
 * both; calls on one handle must not overlap.  The call also reads the
 * device status word once the step is done and returns the first condition
 * the kernels recorded (clearing it, as nest_device_status does), so an
 * overflow or a failed margin check is never returned as NEST_OK.  The paper's method is the same as nest_knn_step (Eq. 1-3);
 * only the data movement differs.
 */
NEST_API nest_status_t nest_knn_step_host(nest_datastore_t* ds, const void* q, int32_t B, int32_t r,
                                          const int64_t* seg_off, const float* p_lm, float mu,
                                          float lambda, float* s_out, int64_t* idx_out,
                                          float* p_m_out, void* stream);

/*
 * nest_knn_search over the keys not yet used in this generation: accepted
 * spans are masked out of the datastore and never retrieved again
 * (Sec. 3.4, last paragraph).
 *
 *   key_mask  ceil(N / 32) uint32 words on the device; bit (k % 32) of word
 *             k / 32 set means key k is never a candidate.  Owned by the
 *             caller (nest_mask_keys sets bits).
 * Other arguments and outputs are those of nest_knn_search.
 */
NEST_API nest_status_t nest_knn_search_masked(nest_datastore_t* ds, const void* q, int32_t B,
                                              int32_t r, const int64_t* seg_off,
                                              const uint32_t* key_mask, float* s_out,
                                              int64_t* idx_out, void* stream);

/*
 * Mark keys [first_key, first_key + count) as used in key_mask (atomic OR on
 * the device, stream-ordered): the keys of an accepted span, which are
 * consecutive in a passage's datastore.  0 <= first_key <= N - count.
 */
NEST_API nest_status_t nest_mask_keys(nest_datastore_t* ds, uint32_t* key_mask, int64_t first_key,
                                      int64_t count, void* stream);

/*
 * Greedy token, span start and span decision for each row b < B (Eq. 5 and
 * Eq. 6, Sec. 3.3; the span-selection steps of Algorithm 1):
 *
 *   token_out[b]    = argmax_w p_m[b][w]             (ties: smaller token id)
 *   p_max_out[b]    = p_m[b][token_out[b]]
 *   span_key_out[b] = the key index of the neighbour i of row b with
 *                     V[idx_i] = token whose own term exp(mu s_i) is largest,
 *                     i.e. the nearest such neighbour (ties: smaller key
 *                     index): the start of the n-gram continuation in the
 *                     corpus; -1 if no neighbour has that value.  (Eq. 5 and
 *                     Algorithm 1 write an argmax of p_kNN over neighbours
 *                     with value w_t, which is one shared number; the
 *                     max-pooling is read as pooling their own terms.)
 *   use_span_out[b] = 1 if lambda[b] <= delta and a span start exists (Eq. 6
 *                     emits the n-gram), else 0 (emit the token).
 *
 *   p_m        B x vocab fp32 (for example from nest_knn_mix_rrc).
 *   s_in/idx_in  B x r neighbours from the search.
 *   lambda     B fp32 per-row interpolation weights (lambda_t of Eq. 4).
 */
NEST_API nest_status_t nest_knn_decide(nest_datastore_t* ds, const float* p_m, const float* s_in,
                                       const int64_t* idx_in, const float* lambda, int32_t B,
                                       int32_t r, float delta, int32_t* token_out,
                                       float* p_max_out, int64_t* span_key_out,
                                       int32_t* use_span_out, void* stream);

/*
 * Relaxed speculative decoding of drafted spans (Eq. 7, Sec. 3.4; the
 * verification loop of Algorithm 1).  Row b of p_m (rows x vocab fp32) is
 * p_M at draft position b given the prefix and the drafted tokens before
 * it; draft[b] is the token drafted there.  Span j covers rows
 * [span_off[j], span_off[j+1]) (spans + 1 int32 offsets).
 *
 *   ratio_out[b]    = p_m[b][draft[b]] / (gamma * max_w p_m[b][w])  (0 if the max is 0)
 *   accept_out[b]   = 1 if min(1, ratio) > 1/2, else 0 (Algorithm 1 stops at
 *                     the first position whose acceptance is at most 1/2)
 *   n_accept_out[j] = number of leading accepted positions of span j
 *
 * 1 <= rows <= 65535 and 1 <= spans <= 65535; a span may be empty
 * (span_off[j] == span_off[j+1], n_accept = 0).
 * gamma > 0 is the relaxation factor (Sec. 3.4 relaxes with values in
 * (0, 1]; gamma <= 0 or NaN is refused).  A draft token outside
 * [0, vocab) is rejected and recorded as NEST_ERR_VALUE_RANGE; bad span
 * offsets give n_accept = 0 and NEST_ERR_INVALID_ARG in the device status.
 */
NEST_API nest_status_t nest_verify_spans(nest_datastore_t* ds, const float* p_m,
                                         const int32_t* draft, int32_t rows,
                                         const int32_t* span_off, int32_t spans, float gamma,
                                         float* ratio_out, int32_t* accept_out,
                                         int32_t* n_accept_out, void* stream);

/*
 * Check of the failure-detection path (no counterpart in the paper).  Runs
 * one kernel that waits on an mbarrier nothing arrives on, through the same
 * bounded wait the scan kernels use for their pipeline stages.  The wait
 * gives up after its limit (2 s) and records NEST_ERR_TIMEOUT in this
 * datastore's device status, which nest_device_status then returns; the
 * context stays usable.  Synchronizes `stream`.  waited_ns (host, may be
 * NULL) receives how long the kernel waited.  Returns NEST_OK when the
 * kernel ran.
 */
NEST_API nest_status_t nest_selftest_bounded_wait(nest_datastore_t* ds, int64_t* waited_ns,
                                                  void* stream);

/*
 * Synchronize `stream`, return the first condition the GPU recorded for
 * this datastore since the previous call (NEST_OK if none), and clear it.
 */
NEST_API nest_status_t nest_device_status(nest_datastore_t* ds, void* stream);

/*
 * Kernel timing: while enabled, every search records a pair of CUDA events
 * on its stream around its distance-scan kernel (the kernel that streams
 * the keys).  nest_timing_read synchronizes those events and returns the
 * summed milliseconds and the number of launches since the last read.
 */
NEST_API nest_status_t nest_timing_enable(nest_datastore_t* ds, int32_t on);
NEST_API nest_status_t nest_timing_read(nest_datastore_t* ds, double* total_ms, int64_t* launches);

/*
 * Which distance scan a search of this shape runs on this datastore:
 *   0  CUDA-core scan with per-CTA top-r (fp32 keys with rows over 2 KiB,
 *      or rows TMA cannot map)
 *   1  tensor-core scan with per-CTA top-r (bf16 keys, query groups of <= 16)
 *   2  tensor-core scan of large query batches against sampled admission
 *      thresholds (bf16 keys, more queries than one CTA keeps lists for)
 *   3  the same with two 128-key tiles per pipeline stage (groups of 256
 *      queries, when three 64 KiB stages fit in shared memory)
 *   4  the same on CTA pairs (groups of 256 or 512 queries, 256-key tiles
 *      split over two SMs): by default for 129 to 512 queries; see
 *      nest_datastore_use_cta_pairs
 *   5  CUDA-core scan of fp32 keys with rows of at most 2 KiB (d <= 512), one
 *      key row per thread, with per-CTA top-r
 * Returns a negative nest_status_t on a bad argument.  Host only, no launch.
 */
NEST_API int32_t nest_search_path(const nest_datastore_t* ds, int32_t B, int32_t r,
                                  int32_t ragged);

/*
 * The plan a search of this shape would run, computed on the host without
 * a GPU or a handle (no counterpart in the paper; for capacity planning and
 * for tests of the planning logic).  It runs the same planning code as
 * nest_knn_search on a datastore of N keys of d elements of `dtype`, on a
 * device with `num_sms` SMs and `smem_per_block` bytes of opt-in shared
 * memory per block (cudaDevAttrMaxSharedMemoryPerBlockOptin), with
 * nest_datastore_use_cta_pairs(ds, cta_pairs) in effect (1, 0 or -1, the
 * handle's default; the device is assumed able to place the pairs).  Arguments are checked as
 * nest_datastore_create and nest_knn_search check them.
 */
typedef struct nest_plan {
    int32_t path;               /* as nest_search_path */
    int32_t queries_per_group;  /* queries one CTA (or CTA pair) scans together */
    int32_t groups;             /* query groups */
    int32_t parts;              /* key-range parts per group (CTAs or CTA pairs) */
    int32_t stages;             /* pipeline stages of the scan kernel (1 for path 5) */
    int32_t single_pass;        /* paths 2-4: 1 when the sample is every key */
    int64_t sample_stride;      /* paths 2-4: the sample is every stride-th key */
    int64_t list_capacity;      /* words of a query's candidate list: in a CTA's shared
                                   memory (paths 0-1), or in global memory for the
                                   thresholded pass, or the whole datastore when
                                   single_pass (2-4) */
    int64_t scratch_bytes;      /* scratch the handle allocates for this search */
} nest_plan_t;

NEST_API nest_status_t nest_plan_offline(int64_t N, int32_t d, nest_dtype_t dtype, int32_t B,
                                         int32_t r, int32_t ragged, int32_t num_sms,
                                         int64_t smem_per_block, int32_t cta_pairs,
                                         nest_plan_t* out);

/* Kernels this handle has launched since it was created (all kinds). */
NEST_API int64_t nest_launch_count(const nest_datastore_t* ds);

/* Static text for a status code. */
NEST_API const char* nest_status_string(nest_status_t status);

/* ABI version: major * 10000 + minor * 100 + patch (0.2.0: CTA pairs and
 * the bounded-wait self-test added to 0.1.0; 0.3.0: CTA pairs with 48 KiB
 * stages and groups of up to 512 queries, chosen automatically for one
 * query group; search path 5 for narrow fp32 rows). */
NEST_API int32_t nest_version(void);

#ifdef __cplusplus
}
#endif

#endif /* NEST_H */
