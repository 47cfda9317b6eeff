// select.cuh -- block-cooperative exact top-r selection over 64-bit
// candidate words (distance bits : key index) held in shared memory.
//
// MSB-first radix select, 8 bits per pass: a histogram of the next byte of
// the words that still match the selected prefix locates the byte of the
// r-th smallest word.  The loop stops as soon as the chosen bucket holds
// exactly the words still needed (at the latest after the last byte, since
// the words are distinct), so every word <= (prefix | ~mask) is kept: that
// is exactly the r smallest.  A stable in-place compaction then keeps them.
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
        s.done[tid] = cnt[tid] <= r;
    }
    bar();
    for (int pass = 0; pass < 8; ++pass) {
        bool all_done = true;
#pragma unroll
        for (int b = 0; b < NQ; ++b) all_done &= (s.done[b] != 0);
        if (all_done) break;
        const int shift = 56 - 8 * pass;
        for (int i = tid; i < NQ * 256; i += NT) (&s.hist[0][0])[i] = 0;
        bar();
#pragma unroll
        for (int b = 0; b < NQ; ++b) {
            if (s.done[b]) continue;
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
                const uint32_t active = __ballot_sync(~0u, in);
                if (in) {
                    // one shared-memory atomic per distinct bin of the warp
                    const uint32_t peers = __match_any_sync(active, bin);
                    if (lane == __ffs(peers) - 1) atomicAdd(&s.hist[b][bin], (uint32_t)__popc(peers));
                }
            }
        }
        bar();
        for (int b = warp; b < NQ; b += NT / 32) {
            if (s.done[b]) continue;
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
            int before = 0, tot = 0;
#pragma unroll
            for (int w = 0; w < NT / 32; ++w) {
                const int c = s.wcnt[t & 1][w];
                before += (w < warp) ? c : 0;
                tot += c;
            }
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

}  // namespace nest
