// noalloc.cu -- nest_knn_search_static: the r-nearest-neighbour search with
// no device allocation at all.
//
// nest_knn_search keeps its candidate lists in scratch memory the datastore
// handle allocates with cudaMalloc on first use (and frees and re-allocates
// when a larger search comes).  Some callers cannot allow that: a framework
// whose own allocator owns the device memory, or a serving loop that must
// never run a call which synchronizes the whole device (cudaMalloc and
// cudaFree do).  For them this entry point runs the same kernels with the
// candidate lists in one fixed array that is part of the library's device
// image, so nothing is allocated when it is called.
//
// The array is a file-scope __device__ variable: every GPU on which the
// library is loaded holds its kStaticScratchWords * 8 bytes (8 MiB) until the
// process exits.  In host code the variable's name is only a host-side
// stand-in, so its device address is looked up with cudaGetSymbolAddress
// once per device (with that device current) and cached.
#include <mutex>

#include "internal.h"

namespace {

// 2^20 64-bit candidate words = 8 MiB per device.
constexpr size_t kStaticScratchWords = size_t(1) << 20;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint64_t g_static_scratch[kStaticScratchWords];

std::mutex g_scratch_mutex;
uint64_t* g_scratch_addr[kMaxDevices] = {};

// Device address of this device's copy of g_static_scratch (looked up once).
nest_status_t static_scratch(uint64_t** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return NEST_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return NEST_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess || p == nullptr) {
            (void)cudaGetLastError();
            return NEST_ERR_CUDA;
        }
        g_scratch_addr[dev] = static_cast<uint64_t*>(p);
    }
    *out = g_scratch_addr[dev];
    return NEST_OK;
}

}  // namespace

extern "C" nest_status_t nest_knn_search_static(nest_datastore_t* ds, const void* q, int32_t B,
                                                int32_t r, const int64_t* seg_off, float* s_out,
                                                int64_t* idx_out, void* stream)
{
    // the argument, alignment and device checks of nest_knn_search come first
    nest_status_t st = nest::check_search_call(ds, q, B, r, seg_off, s_out, idx_out);
    if (st != NEST_OK) return st;
    size_t need = 0;
    st = nest::search_scratch_words(ds, B, r, seg_off != nullptr, &need);
    if (st != NEST_OK) return st;
    if (need > kStaticScratchWords) return NEST_ERR_OVERFLOW;
    uint64_t* scratch = nullptr;
    st = static_scratch(&scratch);
    if (st != NEST_OK) return st;
    // Nothing in the array has to start at zero: every word a call reads was
    // written earlier in the same call.
    return nest::search_with_scratch(ds, q, B, r, seg_off, s_out, idx_out, scratch,
                                     kStaticScratchWords, static_cast<cudaStream_t>(stream));
}
