// Calibration and selection, one CTA per (request, layer, kv-head):
//   V = E + L + T                (Sec. 4.3, Eqs. 5-11)
//   B~ = max-pool of B over the candidates
//   M = min(rho K, |I|), the M best candidates by B~, lambda =
//       gamma Std(B~) / (Std(V) + eps) over them      (Sec. 4.4, Eqs. 12-15)
//   S = B~ + lambda V                                 (Eq. 16)
//   the K best candidates by S, ascending, then the window (Eq. 17)
// Both "best k" sets use one order: larger value first, equal values ->
// lower position first.  A range-adaptive radix select (select.cuh) finds
// the k-th best key and how many of the keys equal to it are taken; the
// members are then decided thread by thread in position order.
//
// Each thread owns PER consecutive positions [t PER, t PER + PER), so the
// pooling and coherence windows slide along a thread's own positions and
// the position order of the members is (thread, slot) order: one
// block-wide exclusive scan gives every thread its tie rank or its output
// offset.  The one per-position array in shared memory (the pooled
// backbone, then the final score: the keys of the two selections) is
// stored slot-major, element (slot k, thread t) at k T + t, so the radix
// select's passes, which walk the storage index s = k T + t, read
// consecutive words, and those are the thread's own slots.  V lives in
// registers; the windows' neighbours come from the adjacent lanes' runs by
// warp shuffles (from global memory at a warp's two ends).
//
// The standard deviations are fp32 sums over the members: B~'s moments
// about the M-th value (one walk), V's mean and then its squared
// deviations from it (two walks); neither loses precision to cancellation.
#include "common.cuh"
#include "select.cuh"

namespace bacon {
namespace {

using namespace sel;

// Threads per CTA and positions per thread depend on the prompt length only
// (so that every call on the same shape reduces in the same order and gives
// the same bits), sized so that threads x positions stays close to N (the
// selections walk every storage slot): 8 positions per thread on 128, 256,
// 512 or 1024 threads up to 1024, 2048, 4096 or 8192 tokens (several CTAs
// share an SM below 1024 threads), then 1024 threads of 16 positions up to
// 16384 tokens and of 24 up to 24576.
constexpr int kMaxPrompt = 24576;

// Four block-wide fp32 sums in one round (red holds 4 x 33 floats), by a
// shuffle tree (pairwise, so the rounding error grows with log2 of the
// count).  FP64 is avoided: its rate on this part is a small fraction of fp32.
__device__ float4 block_sum4(float4 v, float* red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
        v.z += __shfl_xor_sync(0xffffffffu, v.z, o);
        v.w += __shfl_xor_sync(0xffffffffu, v.w, o);
    }
    if (lane == 0) {
        red[warp] = v.x;
        red[33 + warp] = v.y;
        red[66 + warp] = v.z;
        red[99 + warp] = v.w;
    }
    __syncthreads();
    if (warp < 4) {
        const int nw = (int)(blockDim.x >> 5);
        float t = lane < nw ? red[33 * warp + lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) red[33 * warp + 32] = t;
    }
    __syncthreads();
    const float4 tot = make_float4(red[32], red[65], red[98], red[131]);
    __syncthreads();
    return tot;
}

// Exclusive prefix sum of one int per thread, in thread order; *total
// receives the sum.  warp_sums holds 32 ints.
__device__ int block_exclusive_scan(int v, int* warp_sums, int* total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int nw = (int)(blockDim.x >> 5);
        const int w = lane < nw ? warp_sums[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        if (lane < nw) warp_sums[lane] = wi - w;
        if (lane == 31) *total = wi;
    }
    __syncthreads();
    const int r = warp_sums[warp] + incl - v;
    __syncthreads();
    return r;
}

// Ask L2 to fetch the n floats at p (one prefetch per 128-byte line, every
// address inside the array), so that later loads of them hit L2.
__device__ __forceinline__ void prefetch_l2(const float* p, int n)
{
    for (int i = (int)threadIdx.x * 32; i < n; i += (int)blockDim.x * 32)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(p + i));
}

// x[k] = src[i0 + k] for the thread's PER positions (0 at and past n), with
// 16-byte loads when the run is whole and aligned (n % 4 == 0).
template <int PER>
__device__ __forceinline__ void load_run(const float* __restrict__ src, int i0, int n, float* x)
{
    if ((n & 3) == 0 && i0 + PER <= n) {
        const float4* s4 = reinterpret_cast<const float4*>(src + i0);
#pragma unroll
        for (int q = 0; q < PER / 4; ++q) {
            const float4 v = __ldg(s4 + q);
            x[4 * q] = v.x;
            x[4 * q + 1] = v.y;
            x[4 * q + 2] = v.z;
            x[4 * q + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int k = 0; k < PER; ++k) x[k] = i0 + k < n ? src[i0 + k] : 0.f;
    }
}

// dst[i0 + k] = x[k] for the positions below n.
template <int PER>
__device__ __forceinline__ void store_run(float* dst, int i0, int n, const float* x)
{
    if ((n & 3) == 0 && i0 + PER <= n) {
        float4* d4 = reinterpret_cast<float4*>(dst + i0);
#pragma unroll
        for (int q = 0; q < PER / 4; ++q)
            d4[q] = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
    } else {
#pragma unroll
        for (int k = 0; k < PER; ++k)
            if (i0 + k < n) dst[i0 + k] = x[k];
    }
}

// Slot-major shared-memory array of T threads x PER positions.
template <int T, int PER>
struct Slots {
    float* a;
    // storage index of position i, and the position held at storage index s
    __device__ static __forceinline__ int at(int i) { return (i % PER) * T + i / PER; }
    __device__ static __forceinline__ int pos(int s) { return (s % T) * PER + s / T; }
    __device__ __forceinline__ float& own(int k) const { return a[k * T + (int)threadIdx.x]; }
    __device__ __forceinline__ float operator[](int i) const { return a[at(i)]; }
};

// Keys of the candidates [0, n_cand) of a slot-major array, walked by
// storage index (the radix select's passes read consecutive words).
template <int T, int PER>
struct SlotKeys {
    const float* a;
    int n_cand;
    __device__ __forceinline__ bool operator()(int s, uint32_t& key) const
    {
        if (Slots<T, PER>::pos(s) >= n_cand) return false;
        key = float_key(a[s]);
        return true;
    }
};

// Membership of the thread's candidates in the k best (bit k of the result):
// key > tau, or key == tau among the first `need` such keys in position
// order.  eq_before = keys equal to tau at lower positions (other threads).
template <int T, int PER>
__device__ __forceinline__ uint32_t members(const Slots<T, PER>& arr, int i0, int n_cand,
                                            const SelectResult& sel, int eq_before)
{
    uint32_t m = 0u;
    int rank = eq_before;
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        if (i0 + k < n_cand) {
            const uint32_t key = float_key(arr.own(k));
            const bool eq = key == sel.tau;
            if (key > sel.tau || (eq && rank < sel.need)) m |= 1u << k;
            rank += eq;
        }
    }
    return m;
}

// Keys equal to tau at lower positions than this thread's run (0 without a
// scan when every tie is taken: membership then never needs the rank).
template <int T, int PER>
__device__ __forceinline__ int ties_before(const Slots<T, PER>& arr, int i0, int n_cand,
                                           const SelectResult& sel, int* warp_sums, int* total)
{
    if (sel.all_ties_in()) return 0;
    int eq = 0;
#pragma unroll
    for (int k = 0; k < PER; ++k)
        eq += (i0 + k < n_cand) && float_key(arr.own(k)) == sel.tau;
    return block_exclusive_scan(eq, warp_sums, total);
}

// The residual E of the thread's run into x (0 at and past N), added to v
// when use_E, and the coherence (Eqs. 5-7) with the radius R a constant:
// v[k] += the mean of E over [i - R, i + R] clipped to [0, N), for the run's
// positions i = i0 + k < N.  The R values on either side come from the
// neighbouring lanes' runs by shuffles (from global memory at a warp's two
// ends, loaded together with the run) and count as 0 outside [0, N).  The
// window sum slides along the run: drop i - R, add i + 1 + R.  Needs
// R <= PER and every lane of the warp.
template <int PER, int R>
__device__ __forceinline__ void coherence_run(const float* __restrict__ Ec, int i0, int N,
                                              bool use_E, float* x, float* v)
{
    static_assert(R <= PER, "the halo must come from the adjacent run");
    const int lane = threadIdx.x & 31;
    load_run<PER>(Ec, i0, N, x);
    float gl[R], gh[R];
#pragma unroll
    for (int m = 0; m < R; ++m) {
        const int jl = i0 - R + m, jh = i0 + PER + m;
        gl[m] = (lane == 0 && jl >= 0 && jl < N) ? __ldg(Ec + jl) : 0.f;
        gh[m] = (lane == 31 && jh < N) ? __ldg(Ec + jh) : 0.f;
    }
    if (use_E) {
#pragma unroll
        for (int k = 0; k < PER; ++k) v[k] += x[k];
    }
    float e[PER + 2 * R];
#pragma unroll
    for (int m = 0; m < R; ++m) {
        const int jl = i0 - R + m, jh = i0 + PER + m;
        const float lo = __shfl_up_sync(0xffffffffu, x[PER - R + m], 1);
        const float hi = __shfl_down_sync(0xffffffffu, x[m], 1);
        e[m] = lane == 0 ? gl[m] : (jl >= 0 ? lo : 0.f);
        e[R + PER + m] = lane == 31 ? gh[m] : (jh < N ? hi : 0.f);
    }
#pragma unroll
    for (int k = 0; k < PER; ++k) e[R + k] = x[k];
    const float inv_full = 1.f / (float)(2 * R + 1);  // windows away from the ends
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j <= 2 * R; ++j) sum += e[j];
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int i = i0 + k;
        if (i < N) {
            const int cnt = min(N - 1, i + R) - max(0, i - R) + 1;
            float w = inv_full;
            if (cnt != 2 * R + 1) w = 1.f / (float)cnt;
            // the window sum of non-negative values: rounding in the slide
            // can leave ~1e-9 below zero after a large value leaves the
            // window, so it is clamped
            v[k] += fmaxf(sum, 0.f) * w;
        }
        if (k + 1 < PER) {
            sum -= e[k];
            sum += e[k + 2 * R + 1];
        }
    }
}

// The same for any radius, reading the window from global memory (L1).
template <int PER>
__device__ __forceinline__ void coherence_any(const float* __restrict__ Ec, int i0, int N, int r,
                                              float* v)
{
    const float inv_full = 1.f / (float)(2 * r + 1);
    int lo = max(0, i0 - r), hi = min(N - 1, i0 + r);
    float sum = 0.f;
    for (int j = lo; j <= hi; ++j) sum += __ldg(Ec + j);
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int i = i0 + k;
        if (i < N) {
            const int cnt = hi - lo + 1;
            v[k] += fmaxf(sum, 0.f) * (cnt == 2 * r + 1 ? inv_full : 1.f / (float)cnt);
            if (i - r >= 0) sum -= __ldg(Ec + i - r);
            if (i + 1 + r <= N - 1) sum += __ldg(Ec + i + 1 + r);
            lo = max(0, i + 1 - r);
            hi = min(N - 1, i + 1 + r);
        }
    }
}

// Whether the run with its halo (PER + 2 R floats) and V (PER floats) fit
// in the 64 registers a thread has, with room for the rest.
__host__ __device__ constexpr bool run_fits(int PER, int R) { return R <= PER && 2 * PER + 2 * R <= 56; }

// E (added to v when use_E) and its coherence, with the paper's radii (3, 5,
// 7, 9) compiled as constants where the registers allow.
template <int PER>
__device__ __forceinline__ void residual_and_coherence(const float* __restrict__ Ec, int i0, int N,
                                                       int r, bool use_E, float* x, float* v)
{
    if constexpr (run_fits(PER, 3))
        if (r == 3) return coherence_run<PER, 3>(Ec, i0, N, use_E, x, v);
    if constexpr (run_fits(PER, 5))
        if (r == 5) return coherence_run<PER, 5>(Ec, i0, N, use_E, x, v);
    if constexpr (run_fits(PER, 7))
        if (r == 7) return coherence_run<PER, 7>(Ec, i0, N, use_E, x, v);
    if constexpr (run_fits(PER, 9))
        if (r == 9) return coherence_run<PER, 9>(Ec, i0, N, use_E, x, v);
    load_run<PER>(Ec, i0, N, x);
    if (use_E) {
#pragma unroll
        for (int k = 0; k < PER; ++k) v[k] += x[k];
    }
    coherence_any<PER>(Ec, i0, N, r, v);
}

// One unit (request, layer, kv-head) u under hyper-parameters c.  lam_out
// (may be null) receives lambda; idx_pair is the pair's [Hkv][kept] output.
// N <= T PER.  One slot-major array in shared memory holds the pooled
// backbone and then the final score; V stays in the thread's registers
// (every later read of it is the thread's own), and the pooling and
// coherence windows read their neighbours from global memory (L1), so a
// unit needs T PER floats of shared memory and two CTAs share an SM at the
// 512-thread classes.
template <int T, int PER>
__device__ __forceinline__ void calibrate_unit(const Shape& s, const Calib& c, const CalibArgs& a,
                                               int u, float* lam_out, int32_t* idx_pair)
{
    extern __shared__ __align__(16) float sm[];
    const Slots<T, PER> A{sm};  // pooled backbone B~, then the final score S
    // the selections never look at more than T PER keys
    constexpr int kCap = T * PER < kSelCap ? T * PER : kSelCap;
    __shared__ __align__(16) int hist[sel_hist_ints(kCap)];
    __shared__ int bcast[8];
    __shared__ int warp_sums[32];
    __shared__ float red[4 * 33];
    __shared__ int total_s;

    const int N = s.N, W = s.W;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const int rq = pair / s.layers;
    const int layer = a.layer0 + (pair - rq * s.layers);
    const int win = c.keep_window ? W : 0;
    const int n_cand = N - win;
    const int kept_total = min(a.budget[pair], N);
    const int keep = kept_total - win;
    const int i0 = (int)threadIdx.x * PER;

    uint32_t skmin = 0xffffffffu, skmax = 0u;  // key range of S over the candidates
    auto Eof = [&](int j) -> const float* {
        return a.Ering + (long long)rq * a.ring_req_stride +
               (long long)(j % a.ring) * s.hkv * N + (long long)h * N;
    };

    if (a.compute_scores) {
        const float* Bu = a.B + (size_t)u * N;
        const float* Ec = Eof(layer);
        const int nprev = min(c.m, layer);
        const float inv_prev = nprev > 0 ? 1.f / (float)nprev : 0.f;
        // the residuals are read only after the pooling and the first
        // selection: start bringing them into L2 now
        prefetch_l2(Ec, N);
        if (c.use_T)
            for (int j = layer - nprev; j < layer; ++j) prefetch_l2(Eof(j), N);

        // ---- pooled backbone over the candidates (max over [i - half, i + half])
        float x[PER];
        load_run<PER>(Bu, i0, N, x);
        uint32_t kmin = 0xffffffffu, kmax = 0u;  // key range of B~ over the candidates
        const int half = c.pool / 2;
        if (half == 3) {
            // width 7 (the default): the run and three positions either side
            // in registers (-inf outside the candidates; the neighbours'
            // values by shuffles, from global memory at a warp's two ends),
            // each output a maximum of seven by three max3
            const int lane = threadIdx.x & 31;
            float hl[3], hr[3];
#pragma unroll
            for (int m = 0; m < 3; ++m) {
                const int jl = i0 - 3 + m, jr = i0 + PER + m;
                hl[m] = (lane == 0 && jl >= 0 && jl < n_cand) ? __ldg(Bu + jl) : -INFINITY;
                hr[m] = (lane == 31 && jr < n_cand) ? __ldg(Bu + jr) : -INFINITY;
            }
#pragma unroll
            for (int k = 0; k < PER; ++k)
                if (i0 + k >= n_cand) x[k] = -INFINITY;
#pragma unroll
            for (int m = 0; m < 3; ++m) {
                const float lo = __shfl_up_sync(0xffffffffu, x[PER - 3 + m], 1);
                const float hi = __shfl_down_sync(0xffffffffu, x[m], 1);
                if (lane != 0) hl[m] = lo;
                if (lane != 31) hr[m] = hi;
            }
            auto at = [&](int j) -> float { return j < 0 ? hl[j + 3] : (j >= PER ? hr[j - PER] : x[j]); };
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                float mx = 0.f;
                if (i0 + k < n_cand) {
                    mx = max3f(max3f(at(k - 3), at(k - 2), at(k - 1)),
                               max3f(at(k), at(k + 1), at(k + 2)), at(k + 3));
                    kmin = min(kmin, float_key(mx));
                    kmax = max(kmax, float_key(mx));
                }
                A.own(k) = mx;
            }
        } else {
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                const int i = i0 + k;
                float mx = 0.f;
                if (i < n_cand) {
                    mx = -INFINITY;
                    const int lo = max(0, i - half), hi = min(n_cand - 1, i + half);
                    for (int v = lo; v <= hi; ++v) mx = fmaxf(mx, __ldg(Bu + v));
                    kmin = min(kmin, float_key(mx));
                    kmax = max(kmax, float_key(mx));
                }
                A.own(k) = mx;
            }
        }
        if (a.Bp) {
#pragma unroll
            for (int k = 0; k < PER; ++k) x[k] = A.own(k);
            store_run<PER>(a.Bp + (size_t)u * N, i0, N, x);
        }

        // ---- the M best candidates by B~ (Eq. 12); V is computed after this
        // selection, so that it is not held across it
        const int calib_keep = min(a.calib_budget[pair], N) - win;
        const long long Ml = (long long)c.rho * (long long)(calib_keep > 0 ? calib_keep : 0);
        const int M = (int)(Ml < n_cand ? Ml : n_cand);
        uint32_t mem = 0u;
        float pb = 0.f;
        if (M > 0) {
            const SelectResult sel = radix_select_range<kCap>(T * PER, M, SlotKeys<T, PER>{A.a, n_cand},
                                                        hist, bcast, kmin, kmax);
            const int eqb = ties_before(A, i0, n_cand, sel, warp_sums, &total_s);
            mem = members(A, i0, n_cand, sel, eqb);
            pb = key_float(sel.tau);
        }

        // ---- persistence: mean of E over the preceding min(m, l) layers (Eqs. 8-9)
        float v[PER];
#pragma unroll
        for (int k = 0; k < PER; ++k) v[k] = 0.f;
        if (c.use_T) {
            // a layer's run in chunks of at most 16 (V and one chunk in
            // registers)
            constexpr int CH = PER <= 16 ? PER : PER / 2;
            static_assert(PER % CH == 0 && CH % 4 == 0, "chunks of whole 16-byte loads");
            for (int j = layer - nprev; j < layer; ++j) {
#pragma unroll
                for (int c0 = 0; c0 < PER; c0 += CH) {
                    float e[CH];
                    load_run<CH>(Eof(j), i0 + c0, N, e);
#pragma unroll
                    for (int k = 0; k < CH; ++k) v[c0 + k] += e[k];
                }
            }
#pragma unroll
            for (int k = 0; k < PER; ++k) v[k] *= inv_prev;
        }
        // ---- E, and the coherence: truncated radius-r box mean of E (Eqs. 5-7)
        if (c.use_L) {
            residual_and_coherence<PER>(Ec, i0, N, c.r, c.use_E, x, v);
        } else if (c.use_E) {
            load_run<PER>(Ec, i0, N, x);
#pragma unroll
            for (int k = 0; k < PER; ++k) v[k] += x[k];
        }
#pragma unroll
        for (int k = 0; k < PER; ++k)
            if (i0 + k >= N) v[k] = 0.f;
        if (a.V) store_run<PER>(a.V + (size_t)u * N, i0, N, v);

        // ---- lambda over the M members (Eqs. 13-15).  B~ by moments about
        // the M-th value (every member is at or above it, so the fp32
        // differences stay small); V by its members' mean, then the mean
        // square deviation from it (two reductions).
        float lam = 0.f;
        if (M > 0) {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                if ((mem >> k) & 1u) {
                    const float db = A.own(k) - pb;
                    acc.x += db;
                    acc.y = fmaf(db, db, acc.y);
                    acc.z += v[k];
                }
            }
            const float4 tot = block_sum4(acc, red);
            const float inv_m = 1.f / (float)M;
            const float mb = tot.x * inv_m, mv = tot.z * inv_m;
            float4 dev = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                if ((mem >> k) & 1u) {
                    const float dv = v[k] - mv;
                    dev.x = fmaf(dv, dv, dev.x);
                }
            }
            const float varv = block_sum4(dev, red).x * inv_m;
            const float stdb = sqrtf(fmaxf(tot.y * inv_m - mb * mb, 0.f));
            const float stdv = sqrtf(varv);
            lam = c.gamma * stdb / (stdv + c.eps);
        }
        if (threadIdx.x == 0 && lam_out) *lam_out = lam;
        // ---- Eq. 16 over the candidates (0 elsewhere)
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            float sv = 0.f;
            if (i0 + k < n_cand) {
                sv = fmaf(lam, v[k], A.own(k));
                skmin = min(skmin, float_key(sv));
                skmax = max(skmax, float_key(sv));
            }
            A.own(k) = sv;
            x[k] = sv;
        }
        if (a.write_S) store_run<PER>(a.S + (size_t)u * N, i0, N, x);
        __syncthreads();
    } else {
        float x[PER];
        load_run<PER>(a.S + (size_t)u * N, i0, N, x);
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            A.own(k) = x[k];
            if (i0 + k < n_cand) {
                skmin = min(skmin, float_key(x[k]));
                skmax = max(skmax, float_key(x[k]));
            }
        }
        __syncthreads();
    }

    if (!a.do_select) return;
    // ---- Eq. 17: the K best candidates by S, ascending, then the window
    int32_t* out = idx_pair + (size_t)h * kept_total;
    if (keep >= n_cand) {
        for (int i = threadIdx.x; i < n_cand; i += blockDim.x) out[i] = i;
    } else if (keep > 0) {
        const SelectResult sel = radix_select_range<kCap>(T * PER, keep, SlotKeys<T, PER>{A.a, n_cand},
                                                    hist, bcast, skmin, skmax);
        const int eqb = ties_before(A, i0, n_cand, sel, warp_sums, &total_s);
        const uint32_t mem = members(A, i0, n_cand, sel, eqb);
        int pos = block_exclusive_scan(__popc(mem), warp_sums, &total_s);
#pragma unroll
        for (int k = 0; k < PER; ++k)
            if ((mem >> k) & 1u) out[pos++] = i0 + k;
        if (threadIdx.x == 0 && total_s != keep && a.err) atomicCAS(a.err, 0, 2);
    }
    for (int w = threadIdx.x; w < win; w += blockDim.x) out[keep + w] = N - W + w;
}

template <int T, int PER>
__global__ void __launch_bounds__(T, 1024 / T)
calibrate_select_kernel(Shape s, Calib c, CalibArgs a)
{
    const int u = blockIdx.x;
    calibrate_unit<T, PER>(s, c, a, u, a.lambda + u, a.idx[u / s.hkv]);
}

// Several hyper-parameter sets over the same B and residuals: CTA (u, v)
// runs unit u under variant v; variant v's indices start v *
// idx_variant_stride elements after the single-variant layout and its
// lambdas v * units after a.lambda.
template <int T, int PER>
__global__ void __launch_bounds__(T, 1024 / T)
calibrate_sweep_kernel(Shape s, CalibTable t, CalibArgs a)
{
    const int u = blockIdx.x, v = blockIdx.y;
    float* lam = a.lambda ? a.lambda + (size_t)v * s.units + u : nullptr;
    calibrate_unit<T, PER>(s, t.c[v], a, u, lam,
                           a.idx[u / s.hkv] + (size_t)v * a.idx_variant_stride);
}

template <int T, int PER>
constexpr size_t smem_bytes()
{
    return (size_t)T * PER * sizeof(float);
}

template <int T, int PER>
cudaError_t launch_select_t(const Shape& s, const Calib& c, const CalibArgs& a, cudaStream_t st)
{
    constexpr size_t sm = smem_bytes<T, PER>();
    cudaError_t e = cudaFuncSetAttribute(calibrate_select_kernel<T, PER>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    calibrate_select_kernel<T, PER><<<s.units, T, sm, st>>>(s, c, a);
    return cudaGetLastError();
}

template <int T, int PER>
cudaError_t launch_sweep_t(const Shape& s, const CalibTable& t, int variants, const CalibArgs& a,
                           cudaStream_t st)
{
    constexpr size_t sm = smem_bytes<T, PER>();
    cudaError_t e = cudaFuncSetAttribute(calibrate_sweep_kernel<T, PER>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    calibrate_sweep_kernel<T, PER><<<dim3(s.units, variants), T, sm, st>>>(s, t, a);
    return cudaGetLastError();
}

// The launch for a prompt of N tokens: F(T, PER) with the size class above.
template <typename F>
cudaError_t by_size(int N, F f)
{
    if (N <= 1024) return f.template run<128, 8>();
    if (N <= 2048) return f.template run<256, 8>();
    if (N <= 4096) return f.template run<512, 8>();
    if (N <= 8192) return f.template run<1024, 8>();
    if (N <= 16384) return f.template run<1024, 16>();
    if (N <= kMaxPrompt) return f.template run<1024, 24>();
    return cudaErrorInvalidValue;
}

struct SelectLaunch {
    const Shape& s;
    const Calib& c;
    const CalibArgs& a;
    cudaStream_t st;
    template <int T, int PER>
    cudaError_t run() const { return launch_select_t<T, PER>(s, c, a, st); }
};

struct SweepLaunch {
    const Shape& s;
    const CalibTable& t;
    int variants;
    const CalibArgs& a;
    cudaStream_t st;
    template <int T, int PER>
    cudaError_t run() const { return launch_sweep_t<T, PER>(s, t, variants, a, st); }
};

}  // namespace

cudaError_t launch_calibrate_select(const Shape& s, const Calib& c, const CalibArgs& a,
                                    cudaStream_t st)
{
    return by_size(s.N, SelectLaunch{s, c, a, st});
}

cudaError_t launch_calibrate_sweep(const Shape& s, const CalibTable& t, int variants,
                                   const CalibArgs& a, cudaStream_t st)
{
    return by_size(s.N, SweepLaunch{s, t, variants, a, st});
}

}  // namespace bacon
