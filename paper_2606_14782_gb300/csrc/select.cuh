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

// Histogram bins of one select pass; the caller's shared array `hist` (16-
// byte aligned) holds sel_hist_ints(CAP) ints: two bin buffers (passes
// alternate, so a pass zeroes the next one's bins while it counts), 128 ints
// for the reductions and the buffer counter, and a buffer of up to CAP keys
// (kSelCap, or fewer when a caller never selects among more keys: a smaller
// array lets more CTAs share an SM).
constexpr int kSelBits = 11;
constexpr int kSelBins = 1 << kSelBits;
constexpr int kSelCap = 2048;
__host__ __device__ constexpr int sel_hist_ints(int cap) { return 2 * kSelBins + 128 + cap; }
constexpr int kSelHist = sel_hist_ints(kSelCap);

// k-th best key over the included elements of [0, n) (1 <= k <= their
// count).  First the range [kmin, kmax] of the included keys, then passes
// over it: each pass histograms the keys of the current range into
// kSelBins bins of 2^shift keys (plain shared-memory adds: the bins follow
// the data's own range, so few keys share one), one warp finds the bin
// where the count from the top reaches k, and the range narrows to it,
// until a bin is one key, or until it holds at most 32 keys, which one warp
// then sorts.  At most three passes for 32-bit keys, two block-wide
// barriers each.  Every thread returns the same result; blockDim.x must be
// a multiple of 32 from 64 to 1024.  kmin / kmax: this thread's share of the
// key range (the callers know it from an earlier pass over the keys).  With
// fsum, the block-wide sum of every thread's fval is reduced on the same
// barriers and written to *fsum for every thread.
template <int CAP = kSelCap, typename KeyFn>
__device__ __noinline__ SelectResult radix_select_range(int n, int k, KeyFn key_of, int* hist, int* bcast,
                                           uint32_t kmin, uint32_t kmax, float fval = 0.f,
                                           float* fsum = nullptr)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = (int)(blockDim.x >> 5);
    int* const bins0 = hist;
    int* const red = hist + 2 * kSelBins;  // [0, 32) min, [32, 64) max, [64, 96) sums, [96] counter
    int* const bufcnt = red + 96;
    uint32_t* const buf = reinterpret_cast<uint32_t*>(hist + 2 * kSelBins + 128);
    kmin = __reduce_min_sync(0xffffffffu, kmin);
    kmax = __reduce_max_sync(0xffffffffu, kmax);
    if (fsum) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) fval += __shfl_xor_sync(0xffffffffu, fval, o);
    }
    if (lane == 0) {
        red[warp] = (int)kmin;
        red[32 + warp] = (int)kmax;
        reinterpret_cast<float*>(red)[64 + warp] = fval;
    }
    for (int b = threadIdx.x; b < kSelBins; b += blockDim.x) bins0[b] = 0;
    __syncthreads();
    if (warp == 0) {
        // only the first nwarps entries were written: the other lanes take
        // the neutral element of each reduction
        const bool held = lane < nwarps;
        const uint32_t a = __reduce_min_sync(0xffffffffu, held ? (uint32_t)red[lane] : 0xffffffffu);
        const uint32_t b = __reduce_max_sync(0xffffffffu, held ? (uint32_t)red[32 + lane] : 0u);
        float f = held ? reinterpret_cast<const float*>(red)[64 + lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) f += __shfl_xor_sync(0xffffffffu, f, o);
        if (lane == 0) {
            bcast[0] = (int)a;
            bcast[1] = (int)b;
            reinterpret_cast<float*>(bcast)[5] = f;
            *bufcnt = 0;
        }
    }
    __syncthreads();
    if (fsum) *fsum = reinterpret_cast<const float*>(bcast)[5];
    uint32_t lo = (uint32_t)bcast[0];
    const uint64_t span = (uint64_t)(uint32_t)bcast[1] - lo + 1u;
    int shift = 0;
    while (((span - 1u) >> shift) >= (uint64_t)kSelBins) ++shift;  // top bin index < kSelBins
    uint64_t width = span;  // keys of the current range: [lo, lo + width)
    int remaining = k;
    // Once the current range holds at most CAP keys, the next pass also
    // copies them into the buffer and the passes after it read only that.
    int in_range = -1, nbuf = -1;  // unknown / not compacted
    for (int pass = 0;; ++pass) {
        int* const h = hist + (pass & 1) * kSelBins;          // zeroed
        int* const hn = hist + ((pass + 1) & 1) * kSelBins;   // the next pass's
        const bool collect = nbuf < 0 && in_range >= 0 && in_range <= CAP;
        // the bins of the pass before this one were last read before the
        // barrier that ended it: free to zero for the next pass
        for (int b = threadIdx.x; b < kSelBins; b += blockDim.x) hn[b] = 0;
        if (nbuf >= 0) {
            for (int i = threadIdx.x; i < nbuf; i += blockDim.x) {
                const uint32_t key = buf[i];
                if (key >= lo && (uint64_t)(key - lo) < width) atomicAdd(&h[(key - lo) >> shift], 1);
            }
        } else {
            const uint32_t last = (uint32_t)(width - 1u);  // width <= 2^32
            for (int i0 = threadIdx.x; i0 < n; i0 += 4 * blockDim.x) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int i = i0 + q * (int)blockDim.x;
                    uint32_t key = 0u;
                    if (i < n && key_of(i, key) && key >= lo && key - lo <= last) {
                        atomicAdd(&h[(key - lo) >> shift], 1);
                        if (collect) buf[atomicAdd(bufcnt, 1)] = key;
                    }
                }
            }
        }
        __syncthreads();
        if (warp == 0) {
            // lane l owns bins [64 l, 64 l + 64); counts from the top are
            // suffix sums over the lanes (16-byte reads in a rotated order)
            const int4* h4 = reinterpret_cast<const int4*>(h) + 16 * lane;
            int mine = 0;
#pragma unroll
            for (int q = 0; q < 16; ++q) {
                const int4 v = h4[(q + lane) & 15];
                mine += v.x + v.y + v.z + v.w;
            }
            int incl = mine;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_down_sync(0xffffffffu, incl, o);
                if (lane + o < 32) incl += y;
            }
            // the boundary lane: the highest one whose count from the top
            // reaches `remaining`
            const uint32_t hit = __ballot_sync(0xffffffffu, incl >= remaining);
            const int lb = hit ? 31 - __clz(hit) : 0;
            const int above = __shfl_sync(0xffffffffu, incl - mine, lb);
            // its 64 bins: two per lane, suffix sums again
            const int b0 = 64 * lb + 2 * lane;
            const int c0 = h[b0], c1 = h[b0 + 1];
            const int pair = c0 + c1;
            int inc2 = pair;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_down_sync(0xffffffffu, inc2, o);
                if (lane + o < 32) inc2 += y;
            }
            const uint32_t hit2 = __ballot_sync(0xffffffffu, above + inc2 >= remaining);
            const int l2 = hit2 ? 31 - __clz(hit2) : 0;
            if (lane == l2) {
                const int before = above + inc2 - pair;  // bins above this pair
                const bool top = before + c1 >= remaining;
                bcast[0] = top ? b0 + 1 : b0;
                bcast[1] = top ? remaining - before : remaining - before - c1;
                bcast[4] = top ? c1 : c0;
                bcast[3] = collect ? *bufcnt : -1;
                *bufcnt = 0;
            }
        }
        __syncthreads();
        if (collect) nbuf = bcast[3];
        lo += (uint32_t)bcast[0] << shift;
        remaining = bcast[1];
        const int in_bin = bcast[4];
        in_range = in_bin;
        width = (uint64_t)1 << shift;
        if (shift == 0) return {lo, remaining, in_bin};
        if (in_bin <= 32) {
            // few keys left in the range: gather them (this pass's bins are
            // free now) and let one warp sort them instead of more passes
            int* few = h;
            if (nbuf >= 0) {
                for (int i = threadIdx.x; i < nbuf; i += blockDim.x) {
                    const uint32_t key = buf[i];
                    if (key >= lo && (uint64_t)(key - lo) < width) few[atomicAdd(bufcnt, 1)] = (int)key;
                }
            } else {
                // four keys per iteration, as in the histogram pass: the
                // loads of a thread's keys are in flight together
                const uint32_t last = (uint32_t)(width - 1u);
                for (int i0 = threadIdx.x; i0 < n; i0 += 4 * blockDim.x) {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int i = i0 + q * (int)blockDim.x;
                        uint32_t key = 0u;
                        if (i < n && key_of(i, key) && key >= lo && key - lo <= last)
                            few[atomicAdd(bufcnt, 1)] = (int)key;
                    }
                }
            }
            __syncthreads();
            if (warp == 0) {
                // (valid, key) pairs sorted descending by a bitonic network
                // across the lanes; invalid lanes sink to the end
                unsigned long long v =
                    lane < in_bin ? ((1ull << 32) | (uint32_t)few[lane]) : 0ull;
#pragma unroll
                for (int kk = 2; kk <= 32; kk <<= 1) {
#pragma unroll
                    for (int j = kk >> 1; j > 0; j >>= 1) {
                        const unsigned long long o = __shfl_xor_sync(0xffffffffu, v, j);
                        const bool keep_max = ((lane & kk) == 0) == ((lane & j) == 0);
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
                    *bufcnt = 0;
                }
            }
            __syncthreads();
            return {(uint32_t)bcast[0], bcast[1], bcast[4]};
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
