// mix.cu -- Eq. 2 (p_kNN from the neighbours' similarities), Eq. 3 (fixed
// lambda mix) or Eq. 4 (relative retrieval confidence lambda_t) for each
// query row.
//
// Grid (slices, B).  Every CTA of a row gathers the row's r neighbours'
// token ids V[idx], forms the softmax weights exp(mu (s_i - s_max)) and
// their sum Z (a fixed-order reduction), and sorts (token, slot) pairs so
// that equal tokens are adjacent; it then writes its vocabulary slice:
// p_M[w] = lambda p_LM[w] everywhere, and, after a block barrier, the
// entries of the slice that received neighbour mass,
// p_M[v] = lambda p_LM[v] + (1 - lambda) p_kNN[v].  Sums over equal tokens
// run in slot order, so results do not depend on scheduling.
#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace nest {
namespace {

constexpr int kMixThreads = 512;
constexpr int kWarps = kMixThreads / 32;

__host__ __device__ inline int next_pow2_mix(int x)
{
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

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
    extern __shared__ __align__(16) unsigned char smem[];
    const int P2 = next_pow2_mix(a.r);
    uint64_t* keys = reinterpret_cast<uint64_t*>(smem);        // P2: (token << 32) | slot
    float* wts = reinterpret_cast<float*>(keys + P2);          // r: s, then weights
    __shared__ Red red;
    __shared__ float bc[4];
    __shared__ int bci;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.y, slice = blockIdx.x;
    // Slice boundaries fall on multiples of 4 when the vocabulary allows it.
    const int unit = (a.vocab & 3) == 0 ? 4 : 1;
    const int64_t units = a.vocab / unit;
    const int w0 = unit * (int)(units * slice / a.slices);
    const int w1 = unit * (int)(units * (slice + 1) / a.slices);
    const float* s = a.s + (int64_t)b * a.r;
    const int64_t* id = a.idx + (int64_t)b * a.r;

    // Gather token ids, mark real neighbours, and reduce max s, min s, min/max |s|.
    float smax = -INFINITY, amin = INFINITY, amax = 0.f;
    int count = 0;
    for (int i = tid; i < P2; i += kMixThreads) {
        uint64_t key = kNoCandidate;
        if (i < a.r) {
            const int64_t k = id[i];
            const float si = s[i];
            if (k >= 0 && si > -INFINITY) {
                if (k >= a.N) {
                    record_status(a.status, NEST_ERR_VALUE_RANGE);
                } else {
                    const int32_t v = a.V[k];
                    if (v < 0 || v >= a.vocab) {
                        record_status(a.status, NEST_ERR_VALUE_RANGE);
                    } else {
                        key = ((uint64_t)(uint32_t)v << 32) | (uint32_t)i;
                        smax = fmaxf(smax, si);
                        amin = fminf(amin, fabsf(si));
                        amax = fmaxf(amax, fabsf(si));
                        ++count;
                    }
                }
            }
            wts[i] = si;
        }
        keys[i] = key;
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

    // Weights exp(mu (s_i - s_max)) of real neighbours and their sum Z.
    float zpart = 0.f;
    for (int i = tid; i < a.r; i += kMixThreads) {
        const float w = keys[i] != kNoCandidate ? expf(a.mu * (wts[i] - smax)) : 0.f;
        wts[i] = w;
        zpart += w;
    }
    zpart = warp_sum(zpart);
    if (lane == 0) red.v[warp] = zpart;
    __syncthreads();
    float lam = a.lambda;
    if (tid == 0) {
        float z = 0.f;
        for (int w = 0; w < kWarps; ++w) z += red.v[w];
        if (a.rrc) {
            const float ratio = (bc[2] > 0.f) ? bc[1] / bc[2] : 1.f;
            lam = 1.f / (1.f + expf(-(ratio - a.alpha) / a.tau));
        }
        if (nreal == 0) lam = 1.f;
        bc[3] = z;
        bc[0] = lam;
        if (a.lam_out != nullptr && slice == 0) a.lam_out[b] = lam;
    }

    // Sort (token, slot) ascending so equal tokens are adjacent, slots in order.
    __syncthreads();
    for (int k = 2; k <= P2; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = tid; i < P2; i += kMixThreads) {
                const int l = i ^ j;
                if (l > i) {
                    const uint64_t x = keys[i], y = keys[l];
                    if ((x > y) == ((i & k) == 0)) {
                        keys[i] = y;
                        keys[l] = x;
                    }
                }
            }
            __syncthreads();
        }
    }
    lam = bc[0];
    const float z = bc[3];

    // Dense part of this vocabulary slice.
    const float* plm = a.p_lm + (int64_t)b * a.vocab;
    float* pm = a.p_m + (int64_t)b * a.vocab;
    float* pk = a.p_knn ? a.p_knn + (int64_t)b * a.vocab : nullptr;
    const bool vec = ((a.vocab & 3) == 0) && ((reinterpret_cast<uintptr_t>(a.p_lm) & 15) == 0) &&
                     ((reinterpret_cast<uintptr_t>(a.p_m) & 15) == 0) &&
                     (pk == nullptr || (reinterpret_cast<uintptr_t>(a.p_knn) & 15) == 0) &&
                     ((w0 & 3) == 0);
    if (vec) {
        const int n4 = (w1 - w0) >> 2;
        const float4* src = reinterpret_cast<const float4*>(plm + w0);
        float4* dst = reinterpret_cast<float4*>(pm + w0);
        for (int i = tid; i < n4; i += kMixThreads) {
            float4 x = __ldg(src + i);
            x.x *= lam;
            x.y *= lam;
            x.z *= lam;
            x.w *= lam;
            dst[i] = x;
            if (pk) reinterpret_cast<float4*>(pk + w0)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        for (int w = w0 + 4 * n4 + tid; w < w1; w += kMixThreads) {
            pm[w] = lam * plm[w];
            if (pk) pk[w] = 0.f;
        }
    } else {
        for (int w = w0 + tid; w < w1; w += kMixThreads) {
            pm[w] = lam * plm[w];
            if (pk) pk[w] = 0.f;
        }
    }
    __syncthreads();

    // Tokens of this slice that received neighbour mass.
    for (int i = tid; i < P2; i += kMixThreads) {
        const uint64_t key = keys[i];
        if (key == kNoCandidate) continue;
        const uint32_t v = (uint32_t)(key >> 32);
        if (i > 0 && (uint32_t)(keys[i - 1] >> 32) == v) continue;  // not the first of its token
        if ((int)v < w0 || (int)v >= w1) continue;
        float sum = 0.f;
        for (int j = i; j < P2 && keys[j] != kNoCandidate && (uint32_t)(keys[j] >> 32) == v; ++j)
            sum += wts[(uint32_t)keys[j]];
        const float p = sum / z;
        pm[v] = lam * plm[v] + (1.f - lam) * p;
        if (pk) pk[v] = p;
    }
}

}  // namespace

cudaError_t launch_mix(const MixArgs& a, cudaStream_t stream)
{
    const int P2 = next_pow2_mix(a.r);
    const size_t smem = (size_t)P2 * 8 + (size_t)a.r * 4;
    cudaError_t e =
        cudaFuncSetAttribute(mix_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid(a.slices, a.B);
    mix_kernel<<<grid, kMixThreads, smem, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace nest
