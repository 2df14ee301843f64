// Block-wide selection building blocks shared by the calibration kernel and
// the adaptive (per-layer) selection kernel.
//
// "The k best" always means: larger value first, equal values -> lower index
// first.  Values are compared through order-preserving 32-bit keys
// (float_key).  A range-adaptive radix select finds the k-th best key tau
// and how many elements equal to tau are taken; index-ordered sweeps then
// decide membership: key > tau, or key == tau among the first `need` equal
// keys.  The sweeps are warp-segmented (warp w owns a contiguous index
// range, its lanes take consecutive elements) so that reads are
// conflict-free while ballots keep the index order inside a warp.
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
    int count_eq;  // how many included elements have key == tau
    // every element equal to tau is taken: membership is key >= tau and
    // needs no index-ordered counting
    __device__ __forceinline__ bool all_ties_in() const { return need == count_eq; }
};

// Histogram bins of one select pass; the caller's shared array `hist` holds
// kSelHist ints: the bins, 32 warp totals, a counter and a buffer of up to
// kSelCap keys.
constexpr int kSelBits = 11;
constexpr int kSelBins = 1 << kSelBits;
constexpr int kSelCap = 2048;
constexpr int kSelHist = kSelBins + 64 + kSelCap;

// k-th best key over the included elements of [0, n) (1 <= k <= their
// count).  First the range [kmin, kmax] of the included keys, then passes
// over it: each pass histograms the keys of the current range into
// kSelBins bins of 2^shift keys (plain shared-memory adds: the bins follow
// the data's own range, so few keys share one), takes the bin where the
// count from the top reaches k, and narrows the range to it, until a bin is
// one key, or until it holds at most 32 keys, which one warp then sorts.
// At most three passes for 32-bit keys.  Every thread returns the
// same result; blockDim.x must be a power of two from 64 to 1024.
// kmin / kmax: this thread's share of the key range (the callers that know
// it from an earlier pass over the keys pass it in; see radix_select_by).
template <typename KeyFn>
__device__ SelectResult radix_select_range(int n, int k, KeyFn key_of, int* hist, int* bcast,
                                           uint32_t kmin, uint32_t kmax)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    kmin = __reduce_min_sync(0xffffffffu, kmin);
    kmax = __reduce_max_sync(0xffffffffu, kmax);
    if (lane == 0) {
        hist[warp] = (int)kmin;
        hist[32 + warp] = (int)kmax;
    }
    __syncthreads();
    if (warp == 0) {
        // only the first nwarps entries were written: the other lanes take
        // the neutral element of each reduction
        const bool held = lane < (int)(blockDim.x >> 5);
        const uint32_t a = __reduce_min_sync(0xffffffffu, held ? (uint32_t)hist[lane] : 0xffffffffu);
        const uint32_t b = __reduce_max_sync(0xffffffffu, held ? (uint32_t)hist[32 + lane] : 0u);
        if (lane == 0) {
            bcast[0] = (int)a;
            bcast[1] = (int)b;
        }
    }
    __syncthreads();
    uint32_t lo = (uint32_t)bcast[0];
    const uint64_t span = (uint64_t)(uint32_t)bcast[1] - lo + 1u;
    int shift = 0;
    while (((span - 1u) >> shift) >= (uint64_t)kSelBins) ++shift;  // top bin index < kSelBins
    uint64_t width = span;  // keys of the current range: [lo, lo + width)
    int remaining = k;
    // Once the current range holds at most kSelCap keys, the next pass also
    // copies them into the buffer and the passes after it read only that.
    int* bufcnt = hist + kSelBins + 32;
    uint32_t* buf = reinterpret_cast<uint32_t*>(hist + kSelBins + 64);
    int in_range = -1, nbuf = -1;  // unknown / not compacted
    __syncthreads();
    while (true) {
        for (int b = threadIdx.x; b < kSelBins; b += blockDim.x) hist[b] = 0;
        const bool collect = nbuf < 0 && in_range >= 0 && in_range <= kSelCap;
        if (threadIdx.x == 0) *bufcnt = 0;
        __syncthreads();
        if (nbuf >= 0) {
            for (int i = threadIdx.x; i < nbuf; i += blockDim.x) {
                const uint32_t key = buf[i];
                if (key >= lo && (uint64_t)(key - lo) < width) atomicAdd(&hist[(key - lo) >> shift], 1);
            }
        } else {
            for (int i0 = threadIdx.x; i0 < n; i0 += 4 * blockDim.x) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int i = i0 + q * (int)blockDim.x;
                    uint32_t key = 0u;
                    if (i < n && key_of(i, key) && key >= lo && (uint64_t)(key - lo) < width) {
                        atomicAdd(&hist[(key - lo) >> shift], 1);
                        if (collect) buf[atomicAdd(bufcnt, 1)] = key;
                    }
                }
            }
        }
        __syncthreads();
        if (collect) nbuf = *bufcnt;
        // bins from the top: warp w holds the w-th slice of bpw bins and its
        // lane l the bpl bins just below the top l bpl of that slice; warp
        // totals first, then the boundary warp's lanes, then the lane's bins
        const int nwarps = (int)(blockDim.x >> 5);
        const int bpw = kSelBins / nwarps, bpl = bpw / 32;
        const int ltop = bpw * (warp + 1) - 1 - bpl * lane;  // this lane's highest bin
        int mine = 0;
        for (int q = 0; q < bpl; ++q) mine += hist[ltop - q];
        int incl = mine;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) hist[kSelBins + warp] = incl;  // warp total
        __syncthreads();
        if (warp == 0) {
            // warps from the top: above[w] = totals of warps w + 1 .. nwarps - 1
            const int tot = lane < nwarps ? hist[kSelBins + nwarps - 1 - lane] : 0;
            int cum = tot;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, cum, o);
                if (lane >= o) cum += y;
            }
            const uint32_t hit = __ballot_sync(0xffffffffu, cum >= remaining);
            const int first = __ffs(hit) - 1;  // the boundary warp is nwarps - 1 - first
            const int above = __shfl_sync(0xffffffffu, cum - tot, first);
            if (lane == 0) {
                bcast[2] = nwarps - 1 - first;
                bcast[3] = above;
            }
        }
        __syncthreads();
        if (warp == bcast[2]) {
            const int rem = remaining - bcast[3];
            const uint32_t hit = __ballot_sync(0xffffffffu, incl >= rem);
            const int first = __ffs(hit) - 1;
            if (lane == first) {
                int before = incl - mine;  // bins above this lane's
                for (int q = 0; q < bpl; ++q) {
                    const int c = hist[ltop - q];
                    if (before + c >= rem) {
                        bcast[0] = ltop - q;
                        bcast[1] = rem - before;
                        bcast[4] = c;
                        break;
                    }
                    before += c;
                }
            }
        }
        __syncthreads();
        lo += (uint32_t)bcast[0] << shift;
        remaining = bcast[1];
        const int in_bin = bcast[4];
        in_range = in_bin;
        width = (uint64_t)1 << shift;
        __syncthreads();
        if (shift == 0) return {lo, remaining, in_bin};
        if (in_bin <= 32) {
            // few keys left in the range: gather them (the bins are free
            // now) and let one warp sort them instead of more passes
            int* few = hist;
            if (threadIdx.x == 0) *bufcnt = 0;
            __syncthreads();
            if (nbuf >= 0) {
                for (int i = threadIdx.x; i < nbuf; i += blockDim.x) {
                    const uint32_t key = buf[i];
                    if (key >= lo && (uint64_t)(key - lo) < width) few[atomicAdd(bufcnt, 1)] = (int)key;
                }
            } else {
                for (int i = threadIdx.x; i < n; i += blockDim.x) {
                    uint32_t key = 0u;
                    if (key_of(i, key) && key >= lo && (uint64_t)(key - lo) < width)
                        few[atomicAdd(bufcnt, 1)] = (int)key;
                }
            }
            __syncthreads();
            if (warp == 0) {
                // (valid, key) pairs sorted descending by a bitonic network
                // across the lanes; invalid lanes sink to the end
                unsigned long long v =
                    lane < in_bin ? ((1ull << 32) | (uint32_t)few[lane]) : 0ull;
#pragma unroll
                for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
                    for (int j = k >> 1; j > 0; j >>= 1) {
                        const unsigned long long o = __shfl_xor_sync(0xffffffffu, v, j);
                        const bool keep_max = ((lane & k) == 0) == ((lane & j) == 0);
                        v = keep_max ? (v > o ? v : o) : (v < o ? v : o);
                    }
                }
                const uint32_t tau = (uint32_t)__shfl_sync(0xffffffffu, v, remaining - 1);
                const bool valid = (v >> 32) != 0ull;
                const uint32_t key = (uint32_t)v;
                const int eq = __popc(__ballot_sync(0xffffffffu, valid && key == tau));
                const int gt = __popc(__ballot_sync(0xffffffffu, valid && key > tau));
                if (lane == 0) {
                    bcast[0] = (int)tau;
                    bcast[1] = remaining - gt;
                    bcast[4] = eq;
                }
            }
            __syncthreads();
            const SelectResult r = {(uint32_t)bcast[0], bcast[1], bcast[4]};
            __syncthreads();
            return r;
        }
        shift = shift > kSelBits ? shift - kSelBits : 0;
    }
}

template <typename KeyFn>
__device__ SelectResult radix_select_by(int n, int k, KeyFn key_of, int* hist, int* bcast)
{
    uint32_t kmin = 0xffffffffu, kmax = 0u;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        uint32_t key;
        if (key_of(i, key)) {
            kmin = min(kmin, key);
            kmax = max(kmax, key);
        }
    }
    return radix_select_range(n, k, key_of, hist, bcast, kmin, kmax);
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

// Included keys equal to tau before this warp's segment (0 without a pass
// when every tie is taken: the walks then never need the count).
template <typename KeyFn>
__device__ int eq_before_segment_by(Segment sg, SelectResult sel, KeyFn key_of, int* warp_sums,
                                    int* total)
{
    if (sel.all_ties_in()) return 0;
    const uint32_t tau = sel.tau;
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

// walk_topk_by over this warp's segment that keeps each 32-element step's
// membership ballot in masks[0, MAXSTEPS) (0 past the segment's end) and
// returns the segment's member count, so that a later pass can emit the
// members without reading the keys again.  MAXSTEPS must cover the segment
// (its length / 32).
template <int MAXSTEPS, typename KeyFn>
__device__ __forceinline__ int walk_topk_masks_by(Segment sg, SelectResult sel, int eq_before,
                                                  KeyFn key_of, uint32_t* masks)
{
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    int running = eq_before, total = 0;
#pragma unroll
    for (int st = 0; st < MAXSTEPS; ++st) {
        const int base = sg.lo + 32 * st;
        uint32_t m = 0u;
        if (base < sg.hi) {
            const int i = base + lane;
            uint32_t key = 0u;
            const bool valid = i < sg.hi && key_of(i, key);
            const bool eq = valid && key == sel.tau;
            const uint32_t ball = __ballot_sync(0xffffffffu, eq);
            const int rank = running + __popc(ball & lt);
            const bool in = valid && (key > sel.tau || (eq && rank < sel.need));
            running += __popc(ball);
            m = __ballot_sync(0xffffffffu, in);
        }
        masks[st] = m;
        total += __popc(m);
    }
    return total;
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
__device__ inline int eq_before_segment(const float* vals, Segment sg, SelectResult sel,
                                        int* warp_sums, int* total)
{
    return eq_before_segment_by(sg, sel, FloatKeys{vals}, warp_sums, total);
}
template <typename F>
__device__ __forceinline__ void walk_topk(const float* vals, Segment sg, SelectResult sel,
                                          int eq_before, F f)
{
    walk_topk_by(sg, sel, eq_before, FloatKeys{vals}, f);
}

}  // namespace sel
}  // namespace bacon
