// Block-wide selection building blocks shared by the calibration kernel and
// the adaptive (per-layer) selection kernel.
//
// "The k best" always means: larger value first, equal values -> lower index
// first.  Values are compared through order-preserving 32-bit keys
// (float_key).  A radix select (4 x 8-bit digits, warp-aggregated histogram
// updates) finds the k-th best key tau and how many elements equal to tau
// are taken; index-ordered sweeps then decide membership: key > tau, or
// key == tau among the first `need` equal keys.  The sweeps are
// warp-segmented (warp w owns a contiguous index range, its lanes take
// consecutive elements) so that reads are conflict-free while ballots keep
// the index order inside a warp.
//
// A key accessor `key_of(i, key)` returns false for elements excluded from a
// selection (they are neither counted nor taken).
#pragma once

#include "common.cuh"

namespace bacon {
namespace sel {

struct SelectResult {
    uint32_t tau;  // key of the k-th best element
    int need;      // how many elements with key == tau are taken
};

// k-th best key over the included elements of [0, n) (1 <= k <= their
// count).  Every thread returns the same result.
template <typename KeyFn>
__device__ SelectResult radix_select_by(int n, int k, KeyFn key_of, int* hist, int* bcast)
{
    uint32_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        // warp-aggregated: lanes that fall into the same bin add once together
        const int n_round = (n + 31) & ~31;
        for (int i = threadIdx.x; i < n_round; i += blockDim.x) {
            uint32_t key = 0u;
            const bool in = i < n && key_of(i, key);
            const bool hit = in && (key & mask) == prefix;
            const int bin = hit ? (int)((key >> shift) & 255u) : -1;
            const uint32_t peers = __match_any_sync(0xffffffffu, bin);
            if (hit && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
        }
        __syncthreads();
        if (threadIdx.x < 32) {
            // bins high to low: find the bin where the running count from the
            // top reaches `remaining`
            const int lane = threadIdx.x;
            int cum = 0, found_bin = -1, found_rem = 0;
            for (int base = 255; base >= 0 && found_bin < 0; base -= 32) {
                const int b = base - lane;
                const int c = hist[b];
                int incl = c;  // inclusive scan from the top (lane 0 = highest bin)
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const uint32_t ballot = __ballot_sync(0xffffffffu, cum + incl >= remaining);
                if (ballot) {
                    const int first = __ffs(ballot) - 1;
                    const int excl = __shfl_sync(0xffffffffu, incl - c, first);
                    found_bin = base - first;
                    found_rem = remaining - (cum + excl);
                }
                cum += __shfl_sync(0xffffffffu, incl, 31);
            }
            if (lane == 0) {
                bcast[0] = found_bin;
                bcast[1] = found_rem;
            }
        }
        __syncthreads();
        prefix |= (uint32_t)bcast[0] << shift;
        mask |= 255u << shift;
        remaining = bcast[1];
        __syncthreads();
    }
    return {prefix, remaining};
}

struct Segment {
    int lo, hi;
};

// This warp's contiguous share of [0, n), a multiple of 32 long.
__device__ __forceinline__ Segment warp_segment(int n)
{
    const int nw = blockDim.x >> 5;
    const int per = ((n + nw - 1) / nw + 31) & ~31;
    const int lo = min(n, (int)(threadIdx.x >> 5) * per);
    return {lo, min(n, lo + per)};
}

__device__ __forceinline__ int warp_sum(int v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Exclusive scan of one value per warp (lane 0's `v`), returned to every
// lane; *total receives the sum.
__device__ inline int warp_exclusive_scan(int v, int* warp_sums, int* total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        const int w = lane < nw ? warp_sums[lane] : 0;
        int incl = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane < nw) warp_sums[lane] = incl - w;
        if (lane == 31) *total = incl;
    }
    __syncthreads();
    const int r = warp_sums[warp];
    __syncthreads();
    return r;
}

// Included keys equal to tau before this warp's segment.
template <typename KeyFn>
__device__ int eq_before_segment_by(Segment sg, uint32_t tau, KeyFn key_of, int* warp_sums,
                                    int* total)
{
    int eq = 0;
    for (int i = sg.lo + (threadIdx.x & 31); i < sg.hi; i += 32) {
        uint32_t key = 0u;
        eq += key_of(i, key) && key == tau;
    }
    return warp_exclusive_scan(warp_sum(eq), warp_sums, total);
}

// Walks this warp's segment in index order and calls f(i, valid, in), in =
// membership in the k best.  Every lane of the warp calls f the same number
// of times (valid = false past the segment end), so f may use warp votes.
template <typename KeyFn, typename F>
__device__ __forceinline__ void walk_topk_by(Segment sg, SelectResult sel, int eq_before,
                                             KeyFn key_of, F f)
{
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    int running = eq_before;
    for (int base = sg.lo; base < sg.hi; base += 32) {
        const int i = base + lane;
        uint32_t key = 0u;
        const bool valid = i < sg.hi && key_of(i, key);
        const bool eq = valid && key == sel.tau;
        const uint32_t ball = __ballot_sync(0xffffffffu, eq);
        const int rank = running + __popc(ball & lt);
        const bool in = valid && (key > sel.tau || (eq && rank < sel.need));
        f(i, i < sg.hi, in);
        running += __popc(ball);
    }
}

// Plain float arrays (every element included).
struct FloatKeys {
    const float* v;
    __device__ __forceinline__ bool operator()(int i, uint32_t& key) const
    {
        key = float_key(v[i]);
        return true;
    }
};

__device__ inline SelectResult radix_select(const float* vals, int n, int k, int* hist, int* bcast)
{
    return radix_select_by(n, k, FloatKeys{vals}, hist, bcast);
}
__device__ inline int eq_before_segment(const float* vals, Segment sg, uint32_t tau,
                                        int* warp_sums, int* total)
{
    return eq_before_segment_by(sg, tau, FloatKeys{vals}, warp_sums, total);
}
template <typename F>
__device__ __forceinline__ void walk_topk(const float* vals, Segment sg, SelectResult sel,
                                          int eq_before, F f)
{
    walk_topk_by(sg, sel, eq_before, FloatKeys{vals}, f);
}

}  // namespace sel
}  // namespace bacon
