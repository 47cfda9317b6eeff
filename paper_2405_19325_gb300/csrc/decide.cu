// decide.cu -- the per-step decisions that follow p_M in NEST:
//
//   decide_kernel  greedy token w_t = argmax p_M (ties: smaller token id) and
//                  the span start of Eq. 5 -- the neighbour with value w_t
//                  whose own term exp(mu s_i) is largest, i.e. the nearest
//                  one (ties: smaller key index) -- and the choice of Eq. 6
//                  between the token and its n-gram (span when lambda_t <= delta);
//   verify_kernel  relaxed speculative decoding (Eq. 7): for each drafted
//                  position, p_M(draft) / (gamma max_w p_M) and acceptance
//                  when min(1, ratio) > 1/2 (Algorithm 1's cut);
//   cut_kernel     leading accepted positions of each drafted span;
//   mask_kernel    marks a run of keys as used (accepted spans are masked
//                  out of the datastore for the rest of a generation, Sec. 3.4).
#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace nest {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;

// (value, index) with "better" = larger value, then smaller index.
struct Best {
    float v;
    int64_t i;
};

__device__ __forceinline__ Best better(Best a, Best b)
{
    if (b.v > a.v || (b.v == a.v && b.i < a.i)) return b;
    return a;
}

__device__ __forceinline__ Best warp_best(Best x)
{
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        Best y;
        y.v = __shfl_xor_sync(~0u, x.v, o);
        y.i = __shfl_xor_sync(~0u, x.i, o);
        x = better(x, y);
    }
    return x;
}

// Block-wide best; every thread gets the result.
__device__ Best block_best(Best x, Best* scratch)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    x = warp_best(x);
    if (lane == 0) scratch[warp] = x;
    __syncthreads();
    Best r = scratch[0];
    for (int w = 1; w < kWarps; ++w) r = better(r, scratch[w]);
    __syncthreads();
    return r;
}

// Largest entry of a row of n floats (ties: smaller index).
__device__ Best row_argmax(const float* row, int n, Best* scratch)
{
    Best b{-INFINITY, (int64_t)n};
    for (int w = threadIdx.x; w < n; w += kThreads) {
        const float v = row[w];
        if (v > b.v) {  // increasing w within a thread: first maximum kept
            b.v = v;
            b.i = w;
        }
    }
    return block_best(b, scratch);
}

__global__ void __launch_bounds__(kThreads) decide_kernel(const DecideArgs a)
{
    __shared__ Best scratch[kWarps];
    const int b = blockIdx.x;
    const Best top = row_argmax(a.p_m + (int64_t)b * a.vocab, a.vocab, &scratch[0]);
    const int32_t token = (int32_t)top.i;
    // span start: nearest neighbour whose value is the token
    Best sp{-INFINITY, INT64_MAX};
    for (int i = threadIdx.x; i < a.r; i += kThreads) {
        const int64_t k = a.idx[(int64_t)b * a.r + i];
        const float s = a.s[(int64_t)b * a.r + i];
        if (k < 0 || !(s > -INFINITY)) continue;
        if (k >= a.N) {
            record_status(a.status, NEST_ERR_VALUE_RANGE);
            continue;
        }
        if (a.V[k] != token) continue;
        sp = better(sp, Best{s, k});
    }
    sp = block_best(sp, &scratch[0]);
    if (threadIdx.x == 0) {
        const bool have = sp.i != INT64_MAX;
        const float lam = a.lambda[b];
        a.token[b] = token;
        a.p_max[b] = top.v;
        a.span_key[b] = have ? sp.i : -1;
        a.use_span[b] = (have && lam <= a.delta) ? 1 : 0;
    }
}

__global__ void __launch_bounds__(kThreads) verify_kernel(const VerifyArgs a)
{
    __shared__ Best scratch[kWarps];
    const int b = blockIdx.x;
    const float* row = a.p_m + (int64_t)b * a.vocab;
    const Best top = row_argmax(row, a.vocab, &scratch[0]);
    if (threadIdx.x == 0) {
        const int32_t t = a.draft[b];
        float ratio = 0.f;
        if (t < 0 || t >= a.vocab) {
            record_status(a.status, NEST_ERR_VALUE_RANGE);
        } else if (top.v > 0.f) {
            ratio = row[t] / (a.gamma * top.v);
        }
        a.ratio[b] = ratio;
        a.accept[b] = fminf(1.f, ratio) > 0.5f ? 1 : 0;
    }
}

__global__ void cut_kernel(const VerifyArgs a)
{
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= a.spans) return;
    const int32_t lo = a.span_off[j], hi = a.span_off[j + 1];
    if (lo < 0 || hi < lo || hi > a.rows) {
        record_status(a.status, NEST_ERR_INVALID_ARG);
        a.n_accept[j] = 0;
        return;
    }
    int32_t n = 0;
    while (lo + n < hi && a.accept[lo + n]) ++n;
    a.n_accept[j] = n;
}

__global__ void mask_kernel(uint32_t* mask, int64_t first, int64_t count)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= count) return;
    const int64_t k = first + i;
    atomicOr(&mask[k >> 5], 1u << (k & 31));
}

}  // namespace

cudaError_t launch_decide(const DecideArgs& a, cudaStream_t stream)
{
    decide_kernel<<<a.B, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_verify(const VerifyArgs& a, cudaStream_t stream)
{
    if (a.rows > 0) {
        verify_kernel<<<a.rows, kThreads, 0, stream>>>(a);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (a.spans > 0) cut_kernel<<<(a.spans + 127) / 128, 128, 0, stream>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_mask(uint32_t* mask, int64_t first, int64_t count, cudaStream_t stream)
{
    if (count <= 0) return cudaSuccess;
    const int64_t blocks = (count + 255) / 256;
    mask_kernel<<<(unsigned)blocks, 256, 0, stream>>>(mask, first, count);
    return cudaGetLastError();
}

}  // namespace nest
