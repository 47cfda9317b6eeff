// mix.cu -- Eq. 2 (p_kNN from the neighbours' similarities), Eq. 3 (fixed
// lambda mix) or Eq. 4 (relative retrieval confidence lambda_t) for each
// query row.
//
// Grid (slices, B).  Every CTA of a row reads the row's r neighbours,
// gathers their token ids V[idx] once into shared memory, and forms the
// softmax weights
// w_i = exp(mu (s_i - s_max)) / Z.  Weights of tokens inside the CTA's
// vocabulary slice are summed per token in shared memory as 48-bit fixed
// point: integer addition is associative, so the sums do not depend on the
// order of the atomics and are exact to 2^-49 per term.  One streaming pass
// over the slice then writes p_M[w] = lambda p_LM[w] + (1 - lambda) p_kNN[w].
#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace nest {
namespace {

constexpr int kMixThreads = 512;
constexpr int kMixMaxSliceTokens = 16384;  // 128 KiB of fixed-point sums
constexpr int kWarps = kMixThreads / 32;
constexpr float kFixScale = 281474976710656.0f;  // 2^48
constexpr float kFixInv = 1.0f / 281474976710656.0f;

struct Red {
    float v[kWarps];
    float w[kWarps];
    float x[kWarps];
    int c[kWarps];
};

__device__ __forceinline__ float warp_sum(float x)
{
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(~0u, x, o);
    return x;
}
__device__ __forceinline__ float warp_max(float x)
{
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x = fmaxf(x, __shfl_xor_sync(~0u, x, o));
    return x;
}
__device__ __forceinline__ float warp_min(float x)
{
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x = fminf(x, __shfl_xor_sync(~0u, x, o));
    return x;
}

__global__ void __launch_bounds__(kMixThreads) mix_kernel(const MixArgs a)
{
    // The row's neighbours, gathered once (token id, -1 for no weight; s),
    // then the slice's fixed-point sums.
    extern __shared__ __align__(16) unsigned long long smem_mix[];
    int32_t* tok = reinterpret_cast<int32_t*>(smem_mix);
    float* sim = reinterpret_cast<float*>(tok + a.r);
    unsigned long long* acc = smem_mix + a.r;
    __shared__ Red red;
    __shared__ float bc[4];
    __shared__ int bci;

    grid_dependency_wait();
    grid_dependents_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.y, slice = blockIdx.x;
    // Slice boundaries fall on multiples of 4 when the vocabulary allows it.
    const int unit = (a.vocab & 3) == 0 ? 4 : 1;
    const int64_t units = a.vocab / unit;
    const int w0 = unit * (int)(units * slice / a.slices);
    const int w1 = unit * (int)(units * (slice + 1) / a.slices);
    const float* s = a.s + (int64_t)b * a.r;
    const int64_t* id = a.idx + (int64_t)b * a.r;

    for (int w = tid; w < w1 - w0; w += kMixThreads) acc[w] = 0ull;

    // Real neighbours: max s, min/max |s|, count (Eq. 2 and Eq. 4 inputs).
    float smax = -INFINITY, amin = INFINITY, amax = 0.f;
    int count = 0;
    for (int i = tid; i < a.r; i += kMixThreads) {
        const int64_t k = id[i];
        const float si = s[i];
        int32_t v = -1;
        if (k >= 0 && si > -INFINITY) {
            if (k >= a.N) {
                record_status(a.status, NEST_ERR_VALUE_RANGE);
            } else {
                const int32_t t = a.V[k];
                if (t < 0 || t >= a.vocab) record_status(a.status, NEST_ERR_VALUE_RANGE);
                else v = t;
            }
        }
        tok[i] = v;  // each thread reads back only the entries it wrote
        sim[i] = si;
        if (v < 0) continue;
        smax = fmaxf(smax, si);
        amin = fminf(amin, fabsf(si));
        amax = fmaxf(amax, fabsf(si));
        ++count;
    }
    smax = warp_max(smax);
    amin = warp_min(amin);
    amax = warp_max(amax);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) count += __shfl_xor_sync(~0u, count, o);
    if (lane == 0) {
        red.v[warp] = smax;
        red.w[warp] = amin;
        red.x[warp] = amax;
        red.c[warp] = count;
    }
    __syncthreads();
    if (tid == 0) {
        float m = -INFINITY, lo = INFINITY, hi = 0.f;
        int c = 0;
        for (int w = 0; w < kWarps; ++w) {
            m = fmaxf(m, red.v[w]);
            lo = fminf(lo, red.w[w]);
            hi = fmaxf(hi, red.x[w]);
            c += red.c[w];
        }
        bc[0] = m;
        bc[1] = lo;
        bc[2] = hi;
        bci = c;
    }
    __syncthreads();
    smax = bc[0];
    const int nreal = bci;

    // Z = sum of exp(mu (s_i - s_max)) over real neighbours (fixed-order tree).
    float zpart = 0.f;
    for (int i = tid; i < a.r; i += kMixThreads) {
        if (tok[i] < 0) continue;
        zpart += expf(a.mu * (sim[i] - smax));
    }
    zpart = warp_sum(zpart);
    if (lane == 0) red.v[warp] = zpart;
    __syncthreads();
    if (tid == 0) {
        float z = 0.f;
        for (int w = 0; w < kWarps; ++w) z += red.v[w];
        float lam = a.lambda;
        if (a.rrc) {
            const float ratio = (bc[2] > 0.f) ? bc[1] / bc[2] : 1.f;
            lam = 1.f / (1.f + expf(-(ratio - a.alpha) / a.tau));
        }
        if (nreal == 0) lam = 1.f;
        bc[3] = z;
        bc[0] = lam;
        if (a.lam_out != nullptr && slice == 0) a.lam_out[b] = lam;
    }
    __syncthreads();
    const float lam = bc[0];
    const float z = bc[3];

    // p_kNN of the slice's tokens: w_i / Z summed per token in fixed point.
    for (int i = tid; i < a.r; i += kMixThreads) {
        const int32_t v = tok[i];
        if (v < w0 || v >= w1) continue;  // also skips v = -1 (w0 >= 0)
        const float p = expf(a.mu * (sim[i] - smax)) / z;
        atomicAdd(&acc[v - w0], (unsigned long long)__float2ull_rn(p * kFixScale));
    }
    __syncthreads();

    // One pass over the slice: p_M = lambda p_LM + (1 - lambda) p_kNN.
    const float* plm = a.p_lm + (int64_t)b * a.vocab;
    float* pm = a.p_m + (int64_t)b * a.vocab;
    float* pk = a.p_knn ? a.p_knn + (int64_t)b * a.vocab : nullptr;
    const float one_m = 1.f - lam;
    const bool vec = ((a.vocab & 3) == 0) && ((reinterpret_cast<uintptr_t>(a.p_lm) & 15) == 0) &&
                     ((reinterpret_cast<uintptr_t>(a.p_m) & 15) == 0) &&
                     (pk == nullptr || (reinterpret_cast<uintptr_t>(a.p_knn) & 15) == 0) &&
                     ((w0 & 3) == 0);
    if (vec) {
        const int n4 = (w1 - w0) >> 2;
        const float4* src = reinterpret_cast<const float4*>(plm + w0);
        float4* dst = reinterpret_cast<float4*>(pm + w0);
        float4* dk = pk ? reinterpret_cast<float4*>(pk + w0) : nullptr;
        for (int i = tid; i < n4; i += kMixThreads) {
            const float4 x = __ldg(src + i);
            const float k0 = __ull2float_rn(acc[4 * i]) * kFixInv;
            const float k1 = __ull2float_rn(acc[4 * i + 1]) * kFixInv;
            const float k2 = __ull2float_rn(acc[4 * i + 2]) * kFixInv;
            const float k3 = __ull2float_rn(acc[4 * i + 3]) * kFixInv;
            dst[i] = make_float4(lam * x.x + one_m * k0, lam * x.y + one_m * k1,
                                 lam * x.z + one_m * k2, lam * x.w + one_m * k3);
            if (dk) dk[i] = make_float4(k0, k1, k2, k3);
        }
    } else {
        for (int w = w0 + tid; w < w1; w += kMixThreads) {
            const float kk = __ull2float_rn(acc[w - w0]) * kFixInv;
            pm[w] = lam * plm[w] + one_m * kk;
            if (pk) pk[w] = kk;
        }
    }
}

}  // namespace

cudaError_t launch_mix(const MixArgs& a, cudaStream_t stream)
{
    // the widest slice of the grid, in tokens
    const int unit = (a.vocab & 3) == 0 ? 4 : 1;
    const int64_t units = a.vocab / unit;
    const int widest = unit * (int)((units + a.slices - 1) / a.slices) + unit;
    // r gathered neighbours (token id and s, 8 bytes) + the slice's sums
    const size_t smem = ((size_t)a.r + widest) * sizeof(unsigned long long);
    cudaError_t e =
        raise_smem_limit(reinterpret_cast<const void*>(mix_kernel), (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid(a.slices, a.B);
    return launch_pdl(mix_kernel, grid, dim3(kMixThreads), smem, stream, a);
}

int mix_min_slices(int vocab) { return (vocab + kMixMaxSliceTokens - 1) / kMixMaxSliceTokens; }

}  // namespace nest
