// select.cuh -- block-cooperative exact top-r selection over 64-bit
// candidate words (distance bits : key index) held in shared memory.
//
// MSB-first radix select, 8 bits per pass: a histogram of the next 8 bits of
// the words that still match the selected prefix locates those bits of the
// r-th smallest word.  The first pass starts below the leading bits that
// all words share (found from the least and greatest distance halves), so
// distances of similar size do not pile into a few bins.  The loop stops
// as soon as the chosen bucket holds exactly the words still needed (at the
// latest once all 64 bits are fixed, since the words are distinct), so
// every word <= (prefix | ~mask) is kept: that is exactly the r smallest.
// A stable in-place compaction then keeps them.
#pragma once

#include "internal.h"
#include "ptx.cuh"

namespace nest {

template <int NT, int NQ>
struct SelectSmem {
    uint32_t hist[NQ][256];
    uint64_t prefix[NQ];
    uint64_t mask[NQ];
    uint32_t krem[NQ];
    uint32_t hmin[NQ];  // least and greatest distance half (bits 63..32)
    uint32_t hmax[NQ];
    int shift[NQ];      // lowest bit of the next 8-bit digit
    int done[NQ];
    int wcnt[2][NT / 32];
};

// For every list b < NQ holding more than r words, keep its r smallest words
// (in their original relative order) at buf[b * stride + 0 .. r), set
// cnt[b] = r and thr[b] to an inclusive upper bound of the kept words; any
// word > thr[b] can never enter list b's r smallest later.  Lists with
// cnt[b] <= r are left alone.  Words of one list must be distinct.  All NT
// threads of the caller's group call this; bar() synchronizes exactly them.
template <int NT, int NQ, class Bar>
__device__ __forceinline__ void select_smallest(uint64_t* buf, int stride, int* cnt,
                                                uint64_t* thr, int r, SelectSmem<NT, NQ>& s,
                                                int tid, Bar bar)
{
    const int lane = tid & 31, warp = tid >> 5;
    if (tid < NQ) {
        s.prefix[tid] = 0;
        s.mask[tid] = 0;
        s.krem[tid] = (uint32_t)r;
        s.hmin[tid] = ~0u;
        s.hmax[tid] = 0;
        s.done[tid] = cnt[tid] <= r;
    }
    bar();
    // leading bits shared by every word of each list
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
        if (s.done[b]) continue;
        const int n = cnt[b];
        const uint64_t* src = buf + (size_t)b * stride;
        uint32_t lo = ~0u, hi = 0;
        for (int j = tid; j < n; j += NT) {
            const uint32_t h = (uint32_t)(src[j] >> 32);
            lo = h < lo ? h : lo;
            hi = h > hi ? h : hi;
        }
        lo = __reduce_min_sync(~0u, lo);
        hi = __reduce_max_sync(~0u, hi);
        if (lane == 0) {
            atomicMin(&s.hmin[b], lo);
            atomicMax(&s.hmax[b], hi);
        }
    }
    bar();
    if (tid < NQ && !s.done[tid]) {
        const uint32_t x = s.hmin[tid] ^ s.hmax[tid];
        const int L = x ? __clz(x) : 32;
        if (L > 0) {
            s.mask[tid] = ~0ull << (64 - L);
            s.prefix[tid] = ((uint64_t)s.hmin[tid] << 32) & s.mask[tid];
        }
        s.shift[tid] = 56 - L;  // L <= 32, so the first digit lies within the word
    }
    bar();
    for (int pass = 0; pass < 8; ++pass) {
        bool all_done = true;
#pragma unroll
        for (int b = 0; b < NQ; ++b) all_done &= (s.done[b] != 0);
        if (all_done) break;
        for (int i = tid; i < NQ * 256; i += NT) (&s.hist[0][0])[i] = 0;
        bar();
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            if (s.done[b]) continue;
            const int shift = s.shift[b];
            const uint64_t pre = s.prefix[b], m = s.mask[b];
            const int n = cnt[b];
            const uint64_t* src = buf + (size_t)b * stride;
            for (int base = 0; base < n; base += NT) {
                const int j = base + tid;
                bool in = false;
                uint32_t bin = 0;
                if (j < n) {
                    const uint64_t e = src[j];
                    in = ((e ^ pre) & m) == 0;
                    bin = (uint32_t)(e >> shift) & 255u;
                }
                if (in) atomicAdd(&s.hist[b][bin], 1u);
            }
        }
        bar();
        for (int b = warp; b < NQ; b += NT / 32) {
            if (s.done[b]) continue;
            const int shift = s.shift[b];
            uint32_t h[8];
            uint32_t local = 0;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                h[k] = s.hist[b][lane * 8 + k];
                local += h[k];
            }
            uint32_t incl = local;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(~0u, incl, o);
                if (lane >= o) incl += y;
            }
            const uint32_t before = incl - local;
            const uint32_t krem = s.krem[b];
            if (before < krem && krem <= incl) {
                uint32_t cum = before;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    if (cum + h[k] >= krem) {
                        const uint32_t bin = (uint32_t)(lane * 8 + k);
                        const uint32_t left = krem - cum;
                        s.prefix[b] |= (uint64_t)bin << shift;
                        s.mask[b] |= 0xFFull << shift;
                        s.krem[b] = left;
                        s.done[b] = (h[k] == left);
                        // the last digit may overlap bits already fixed: the
                        // words that match the prefix agree on those
                        s.shift[b] = shift >= 8 ? shift - 8 : 0;
                        break;
                    }
                    cum += h[k];
                }
            }
        }
        bar();
    }
#pragma unroll
    for (int b = 0; b < NQ; ++b) {
        const int n = cnt[b];
        if (n <= r) continue;
        const uint64_t T = s.prefix[b] | ~s.mask[b];
        uint64_t* p = buf + (size_t)b * stride;
        int out = 0;
        for (int base = 0, t = 0; base < n; base += NT, ++t) {
            const int j = base + tid;
            uint64_t e = 0;
            bool keep = false;
            if (j < n) {
                e = p[j];
                keep = e <= T;
            }
            const uint32_t bal = __ballot_sync(~0u, keep);
            if (lane == 0) s.wcnt[t & 1][warp] = __popc(bal);
            bar();
            // exclusive prefix of the warps' counts by a shuffle scan in every warp
            int c = lane < NT / 32 ? s.wcnt[t & 1][lane] : 0;
#pragma unroll
            for (int o = 1; o < NT / 32; o <<= 1) {
                const int y = __shfl_up_sync(~0u, c, o);
                if (lane >= o) c += y;
            }
            const int tot = __shfl_sync(~0u, c, NT / 32 - 1);
            const int before = warp > 0 ? __shfl_sync(~0u, c, warp - 1) : 0;
            // Every word this tile writes lands at or below where it was read,
            // and every word of this tile was read before the barrier above.
            if (keep) p[out + before + __popc(bal & lanemask_lt())] = e;
            out += tot;
        }
        bar();
        if (tid == 0) {
            cnt[b] = out;
            thr[b] = T;
        }
    }
    bar();
}

// One compare-exchange of a bitonic sorting network done through a warp
// shuffle: element i and element i ^ jj (jj < 32, same warp) keep the smaller
// and the larger word, in ascending order where bit k of i is clear.
__device__ __forceinline__ uint64_t bitonic_shfl(uint64_t x, int i, int jj, int k)
{
    const uint64_t y = __shfl_xor_sync(~0u, x, jj);
    const bool keep_min = ((i & jj) == 0) == ((i & k) == 0);
    return keep_min ? (x < y ? x : y) : (x > y ? x : y);
}

// Sorts buf[0 .. P2) ascending, P2 a power of two.  Stages whose partner
// distance is below 32 run in registers with warp shuffles; only the wider
// ones go through shared memory, with a barrier each.  All NT threads (a
// multiple of 32) call this; bar() synchronizes exactly them.
template <int NT, class Bar>
__device__ __forceinline__ void bitonic_sort(uint64_t* buf, int P2, int tid, Bar bar)
{
    if (P2 < 64) {
        for (int k = 2; k <= P2; k <<= 1) {
            for (int jj = k >> 1; jj > 0; jj >>= 1) {
                for (int i = tid; i < P2; i += NT) {
                    const int l = i ^ jj;
                    if (l > i) {
                        const uint64_t x = buf[i], y = buf[l];
                        if ((x > y) == ((i & k) == 0)) {
                            buf[i] = y;
                            buf[l] = x;
                        }
                    }
                }
                bar();
            }
        }
        return;
    }
    // P2 >= 64: whole warps own 32 consecutive elements
    for (int i = tid; i < P2; i += NT) {
        uint64_t x = buf[i];
#pragma unroll
        for (int k = 2; k <= 32; k <<= 1)
#pragma unroll
            for (int jj = k >> 1; jj > 0; jj >>= 1) x = bitonic_shfl(x, i, jj, k);
        buf[i] = x;
    }
    bar();
    for (int k = 64; k <= P2; k <<= 1) {
        for (int jj = k >> 1; jj >= 32; jj >>= 1) {
            for (int i = tid; i < P2; i += NT) {
                const int l = i ^ jj;
                if (l > i) {
                    const uint64_t x = buf[i], y = buf[l];
                    if ((x > y) == ((i & k) == 0)) {
                        buf[i] = y;
                        buf[l] = x;
                    }
                }
            }
            bar();
        }
        for (int i = tid; i < P2; i += NT) {
            uint64_t x = buf[i];
#pragma unroll
            for (int jj = 16; jj > 0; jj >>= 1) x = bitonic_shfl(x, i, jj, k);
            buf[i] = x;
        }
        bar();
    }
}

}  // namespace nest
