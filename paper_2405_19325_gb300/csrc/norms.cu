// norms.cu -- datastore set-up kernels: fp32 key norms ||k_i||^2 (the
// ||k||^2 term of ||q - k||^2 = ||q||^2 + ||k||^2 - 2 q.k, Sec. 2.2) and the
// token-id range check of V.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace nest {
namespace {

constexpr int kNormThreads = 256;

// One warp per key row; each lane sums squares of 16-byte chunks in fp32.
template <int DT>
__global__ void __launch_bounds__(kNormThreads) key_norms_kernel(const unsigned char* K, int64_t N,
                                                                 int row_bytes, float* out)
{
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (kNormThreads / 32);
    const int chunks = row_bytes / 16;
    for (int64_t row = (int64_t)blockIdx.x * (kNormThreads / 32) + (threadIdx.x >> 5); row < N;
         row += warps) {
        const unsigned char* p = K + row * row_bytes;
        float acc = 0.f;
#pragma unroll 4
        for (int c = lane; c < chunks; c += 32) {
            const uint4 v = ld_global_nc_v4(p + (size_t)c * 16);
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
            if constexpr (DT == NEST_BF16) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float lo = __uint_as_float(w[i] << 16);
                    const float hi = __uint_as_float(w[i] & 0xffff0000u);
                    acc = fmaf(lo, lo, acc);
                    acc = fmaf(hi, hi, acc);
                }
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float x = __uint_as_float(w[i]);
                    acc = fmaf(x, x, acc);
                }
            }
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(~0u, acc, o);
        if (lane == 0) out[row] = acc;
    }
}

__global__ void check_values_kernel(const int32_t* V, int64_t N, int32_t vocab, int* status)
{
    bool bad = false;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t v = V[i];
        bad |= (v < 0) | (v >= vocab);
    }
    if (__any_sync(~0u, bad) && (threadIdx.x & 31) == 0) record_status(status, NEST_ERR_VALUE_RANGE);
}

int grid_for(int64_t work, int per_block)
{
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (work + per_block - 1) / per_block;
    const int64_t cap = (int64_t)sms * 16;
    return (int)(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

cudaError_t launch_key_norms(const void* K, int64_t N, int32_t d, int dtype, float* knorm,
                             cudaStream_t stream)
{
    const int esize = dtype == NEST_BF16 ? 2 : 4;
    const int row_bytes = d * esize;
    const int grid = grid_for(N, kNormThreads / 32);
    if (dtype == NEST_BF16)
        key_norms_kernel<NEST_BF16><<<grid, kNormThreads, 0, stream>>>(
            static_cast<const unsigned char*>(K), N, row_bytes, knorm);
    else
        key_norms_kernel<NEST_F32><<<grid, kNormThreads, 0, stream>>>(
            static_cast<const unsigned char*>(K), N, row_bytes, knorm);
    return cudaGetLastError();
}

cudaError_t launch_check_values(const int32_t* V, int64_t N, int32_t vocab, int* status,
                                cudaStream_t stream)
{
    const int grid = grid_for(N, 256);
    check_values_kernel<<<grid, 256, 0, stream>>>(V, N, vocab, status);
    return cudaGetLastError();
}

}  // namespace nest
