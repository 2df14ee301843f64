// Window scores (Eqs. 1, 2, 4) in one pass over K, for units whose logits fit
// in tensor memory: at most 32 window rows (G W <= 32) and at most 1024
// tokens, i.e. 8 tiles x 32 columns, so that two units' logits (2 x 256 of
// the 512 TMEM columns) are resident at once.
//
// The two-pass kernels (window_tc.cu) stream K twice because a softmax row
// must be normalised over all N keys before any token's share is final.
// When a whole unit's logits stay in TMEM, the normaliser is computed from
// them and the same logits are read again for the shares, so K is read once:
//   * warp 0 loads the unit's window rows (one of two slots) and its K tiles
//     (a ring of stages) by TMA;
//   * warp 1 computes D[token][row] = K Q^T (M = 128 tokens per tile, N = 32
//     rows) for every tile of the unit into the unit's half of TMEM and
//     commits it;
//   * eight epilogue warps (two groups x four lane quarters; group g takes
//     the tiles t = g mod 2) reduce each row's maximum over their tokens by a
//     butterfly transpose across the warp's lanes, meet at a CTA-wide
//     mbarrier, write p = 2^(x - max) over the logits in TMEM while reducing
//     the rows' sums of p the same way, meet again, and then each thread
//     sums its token's p times 1 / (row sum x G W) over the rows (B) and
//     over the last-position rows (Q), and stores E = [Q - B]_+.  Padding
//     rows and the two row sets enter through per-row constants (a -inf
//     shift, zero weights), so no row test runs per logit.
// Every wait is bounded (abort flag, clock limit): on timeout the CTA records
// BACON_ETIMEOUT, drains its own copies and MMAs, frees TMEM and returns.
#include <cuda_bf16.h>

#include "tc.cuh"
#include "window_tc.h"

namespace bacon {
namespace {

constexpr int kTok = 128;        // tokens per K tile (TMEM lanes)
constexpr int kRows = 32;        // window rows per unit, padded (MMA N)
constexpr int kMaxTiles = 8;     // tiles per unit
constexpr int kSlotCols = 256;   // TMEM columns of one unit
constexpr int kEpiWarps = 8;      // two groups of four lane quarters
constexpr int kGroups = kEpiWarps / 4;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kStages = 4;
constexpr float kLog2e = 1.4426950408889634f;

struct Layout {
    uint32_t q_half, q_slot, k_stage;  // bytes
    uint32_t q, k, xr, xs, fm, fw, bars, total;
};

template <int D>
__host__ __device__ inline Layout layout()
{
    constexpr int H = D / 64;
    Layout L;
    L.q_half = (uint32_t)kTcQBoxRows * 128u;  // one 64-row box (rows beyond 32 unused)
    L.q_slot = H * L.q_half;
    L.k_stage = (uint32_t)H * kTok * 128u;
    L.q = 0;
    L.k = L.q + 2 * L.q_slot;
    L.xr = L.k + kStages * L.k_stage;             // [warp][row] partial maxima
    L.xs = L.xr + kEpiWarps * kRows * 4u;          // [warp][row] partial sums
    L.fm = L.xs + kEpiWarps * kRows * 4u;          // [warp][row] -c max (this warp's copy)
    L.fw = L.fm + kEpiWarps * kRows * 4u;          // [warp][row] (B weight, Q weight)
    L.bars = L.fw + kEpiWarps * kRows * 8u;
    L.total = L.bars + 96u + 16u * kStages;
    return L;
}

// Barrier block (8-byte slots): q_full[2], q_empty[2], t_full[2], t_empty[2],
// e_sync, drain, TMEM base word, abort word, k_full[kStages], k_empty[kStages].
struct Bars {
    uint32_t base;
    __device__ __forceinline__ uint32_t q_full(int s) const { return base + 8u * s; }
    __device__ __forceinline__ uint32_t q_empty(int s) const { return base + 16u + 8u * s; }
    __device__ __forceinline__ uint32_t t_full(int s) const { return base + 32u + 8u * s; }
    __device__ __forceinline__ uint32_t t_empty(int s) const { return base + 48u + 8u * s; }
    __device__ __forceinline__ uint32_t e_sync() const { return base + 64u; }
    __device__ __forceinline__ uint32_t drain() const { return base + 72u; }
    __device__ __forceinline__ uint32_t tmem_slot() const { return base + 80u; }
    __device__ __forceinline__ uint32_t abort() const { return base + 88u; }
    __device__ __forceinline__ uint32_t k_full(int st) const { return base + 96u + 8u * st; }
    __device__ __forceinline__ uint32_t k_empty(int st) const
    {
        return base + 96u + 8u * (kStages + st);
    }
};

__device__ inline void raise_abort(const Bars& b, int* err)
{
    tc::st_shared_volatile(b.abort(), 1u);
    if (err) atomicCAS(err, 0, tc::kErrTimeout);
}

__device__ inline void unit_range(int units, int* u0, int* u1)
{
    *u0 = (int)(((long long)blockIdx.x * units) / gridDim.x);
    *u1 = (int)(((long long)(blockIdx.x + 1) * units) / gridDim.x);
}

// ---------------------------------------------------------------- producer

template <int D>
__device__ void produce(const TcArgs& a, const Layout& L, uint8_t* sm, const Bars& b)
{
    constexpr int H = D / 64;
    const Shape& s = a.s;
    const int lane = threadIdx.x & 31;
    const int ntiles = (s.N + kTok - 1) / kTok;
    int u0, u1;
    unit_range(s.units, &u0, &u1);
    int n = 0, kt = 0;
    bool ok = true;
    if (lane == 0) {
        const uint64_t kpol = tc::l2_evict_first_policy();  // K is read once
        for (int u = u0; u < u1 && ok; ++u, ++n) {
            const int pair = u / s.hkv, h = u - pair * s.hkv;
            const int slot = n & 1, use = n >> 1;
            if (!tc::mbar_wait(b.q_empty(slot), (use & 1) ^ 1, b.abort())) { ok = false; break; }
            tc::mbar_arrive_expect_tx(b.q_full(slot), L.q_slot);
            for (int kh = 0; kh < H; ++kh)
                tc::tma_load_2d(sm + L.q + slot * L.q_slot + kh * L.q_half, a.qmaps + pair, kh * 64,
                                h * s.rows, b.q_full(slot));
            for (int t = 0; t < ntiles; ++t, ++kt) {
                const int st = kt % kStages, m = kt / kStages;
                if (!tc::mbar_wait(b.k_empty(st), (m & 1) ^ 1, b.abort())) { ok = false; break; }
                tc::mbar_arrive_expect_tx(b.k_full(st), L.k_stage);
                for (int kh = 0; kh < H; ++kh)
                    tc::tma_load_2d_hint(sm + L.k + st * L.k_stage + kh * kTok * 128, a.kmaps + pair,
                                         kh * 64, h * s.N + t * kTok, b.k_full(st), kpol);
            }
        }
        if (!ok) raise_abort(b, a.err);
        // the last load of every stage and slot must land before the CTA exits
        for (int st = 0; st < kStages && st < kt; ++st) {
            const int last = kt - 1 - ((kt - 1 - st) % kStages);
            tc::mbar_wait(b.k_full(st), (last / kStages) & 1, 0u);
        }
        for (int slot = 0; slot < 2 && slot < n; ++slot) {
            const int last = n - 1 - ((n - 1 - slot) & 1);
            tc::mbar_wait(b.q_full(slot), (last >> 1) & 1, 0u);
        }
    }
}

// ------------------------------------------------------------- MMA issuer

template <int D>
__device__ void issue(const TcArgs& a, const Layout& L, uint8_t* sm, const Bars& b)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTok - 1) / kTok;
    const uint32_t tmem = tc::ld_shared(b.tmem_slot());
    const uint32_t sbase = smem_u32(sm);
    const uint32_t idesc = tc::idesc_bf16(kTok, kRows);
    int u0, u1;
    unit_range(s.units, &u0, &u1);
    int n = 0, kt = 0;
    bool ok = true;
    for (int u = u0; u < u1 && ok; ++u, ++n) {
        const int slot = n & 1, use = n >> 1;
        if (!tc::mbar_wait(b.q_full(slot), use & 1, b.abort()) ||
            !tc::mbar_wait(b.t_empty(slot), (use & 1) ^ 1, b.abort())) {
            ok = false;
            break;
        }
        tc::fence_after_sync();
        const uint32_t qaddr = sbase + L.q + slot * L.q_slot;
        for (int t = 0; t < ntiles; ++t, ++kt) {
            const int st = kt % kStages, m = kt / kStages;
            if (!tc::mbar_wait(b.k_full(st), m & 1, b.abort())) { ok = false; break; }
            tc::fence_after_sync();
            const uint32_t kaddr = sbase + L.k + st * L.k_stage;
            const uint32_t d_tmem = tmem + slot * kSlotCols + t * kRows;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                const int kh = kk / 4;
                const uint32_t koff = (kk % 4) * 32;
                tc::umma_bf16(d_tmem, tc::sdesc_sw128(kaddr + kh * kTok * 128 + koff),
                              tc::sdesc_sw128(qaddr + kh * L.q_half + koff), idesc, kk > 0);
            }
            tc::umma_commit(b.k_empty(st));
        }
        if (!ok) break;
        tc::umma_commit(b.t_full(slot));   // the unit's logits are complete
        tc::umma_commit(b.q_empty(slot));  // and its window rows may be replaced
    }
    if (!ok) raise_abort(b, a.err);
    tc::umma_commit(b.drain());
    tc::mbar_wait(b.drain(), 0, 0u);
}

// ---------------------------------------------------------------- epilogue

// After the call, lane l of the warp holds op over the warp's 32 lanes of
// v[l] (a butterfly transpose: 31 shuffles for 32 values).
template <bool MAX>
__device__ __forceinline__ float transpose_reduce(float* v)
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
        const bool upper = (lane & w) != 0;
#pragma unroll
        for (int j = 0; j < w; ++j) {
            const float send = upper ? v[j] : v[j + w];
            const float keep = upper ? v[j + w] : v[j];
            const float recv = __shfl_xor_sync(0xffffffffu, send, w);
            v[j] = MAX ? fmaxf(keep, recv) : keep + recv;
        }
    }
    return v[0];
}

// Raw logits of one tile for this thread's token (its TMEM lane); in tiles
// that reach into the window (or past N) the rows the token is hidden from
// become -inf: row r sits at position N - W + r mod W, and tokens past N are
// hidden from every row.  Padding rows (beyond the unit's window rows) are
// left as they are: their per-row constants below make every p of theirs 0.
__device__ __forceinline__ void load_visible(uint32_t taddr, int N, int W, int tile, int tok,
                                             float* v)
{
    tc::tmem_ld32(taddr, v);
    tc::tmem_ld_wait_regs32(v);
    if (tile * kTok + kTok - 1 <= N - W) return;  // whole tile before the window
    const int lim = tok < N ? tok - (N - W) : W;  // rows with r mod W < lim are hidden
    int rm = 0;                                    // r mod W
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
        if (rm < lim) v[r] = -INFINITY;
        rm = rm + 1 == W ? 0 : rm + 1;
    }
}

__device__ __forceinline__ bool epi_sync(const Bars& b, int& nsync)
{
    __syncwarp();
    if ((threadIdx.x & 31) == 0) tc::mbar_arrive(b.e_sync());
    const bool ok = tc::mbar_wait(b.e_sync(), nsync & 1, b.abort());
    ++nsync;
    return ok;
}

// SPEC: the multi-head 1024-token unit (N = 1024, W = 32, 32 window rows)
// with its sizes as constants: the tile loops unroll and the mask test runs
// only where a tile can reach into the window.
template <int D, bool SPEC>
__device__ void epilogue(const TcArgs& a, const Layout& L, uint8_t* sm, const Bars& b)
{
    const Shape& s = a.s;
    const int N = SPEC ? 1024 : s.N, W = SPEC ? 32 : s.W, rows = SPEC ? kRows : s.rows;
    const int ntiles = (N + kTok - 1) / kTok;
    constexpr int kSpecPerGroup = 1024 / kTok / kGroups;  // tiles per group (SPEC)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ew = warp - 2;               // epilogue warp 0 .. kEpiWarps - 1
    const int quarter = warp & 3;          // TMEM lanes this warp may access
    const int group = ew >> 2;             // tiles t = group mod kGroups
    const uint32_t tl = tc::ld_shared(b.tmem_slot()) + ((uint32_t)(quarter * 32) << 16);
    float* xr = reinterpret_cast<float*>(sm + L.xr);
    float* xs = reinterpret_cast<float*>(sm + L.xs);
    // this warp's copies of the per-row constants
    float* ncm = reinterpret_cast<float*>(sm + L.fm) + ew * kRows;     // -c max_r
    float2* wbq = reinterpret_cast<float2*>(sm + L.fw) + ew * kRows;   // (B, Q) weights
    const float c = kLog2e * rsqrtf((float)D);
    const unsigned long long c2 = tc::pack2(c, c);
    // bit r: row r is a window row / a last-position row (r mod W = W - 1)
    uint32_t real = 0u, last = 0u;
    for (int r = 0; r < kRows && r < rows; ++r) {
        real |= 1u << r;
        if (r % W == W - 1) last |= 1u << r;
    }
    int u0, u1;
    unit_range(s.units, &u0, &u1);
    int n = 0, nsync = 0;
    bool ok = true;
    for (int u = u0; u < u1 && ok; ++u, ++n) {
        const int slot = n & 1, use = n >> 1;
        if (!tc::mbar_wait(b.t_full(slot), use & 1, b.abort())) { ok = false; break; }
        tc::fence_after_sync();
        const uint32_t tbase = tl + slot * kSlotCols;
        // (1) each row's maximum logit over the unit's visible tokens (c > 0,
        // so c max_r is the maximum of the scaled logits)
        float v[kRows], acc[kRows];
#pragma unroll
        for (int r = 0; r < kRows; ++r) acc[r] = -INFINITY;
#pragma unroll
        for (int i = 0; i < (SPEC ? kSpecPerGroup : kMaxTiles / kGroups); ++i) {
            const int t = group + kGroups * i;
            if (!SPEC && t >= ntiles) break;
            load_visible(tbase + t * kRows, N, W, t, t * kTok + quarter * 32 + lane, v);
#pragma unroll
            for (int r = 0; r < kRows; ++r) acc[r] = fmaxf(acc[r], v[r]);
        }
        xr[ew * kRows + lane] = transpose_reduce<true>(acc);
        if (!epi_sync(b, nsync)) { ok = false; break; }
        float mrow = -INFINITY;
        for (int w = 0; w < kEpiWarps; ++w) mrow = fmaxf(mrow, xr[w * kRows + lane]);
        // p = 2^(c x - c max_r); a padding row takes -inf, so all its p are 0
        // (every window row sees at least the tokens before the window)
        ncm[lane] = (real >> lane) & 1u ? -(c * mrow) : -INFINITY;
        __syncwarp();
        // (2) each row's sum of p; p replaces the logit in TMEM (hidden tokens
        // give -inf, so p = 0)
        unsigned long long acc2[kRows / 2];
#pragma unroll
        for (int r = 0; r < kRows / 2; ++r) acc2[r] = 0ull;
#pragma unroll
        for (int i = 0; i < (SPEC ? kSpecPerGroup : kMaxTiles / kGroups); ++i) {
            const int t = group + kGroups * i;
            if (!SPEC && t >= ntiles) break;
            load_visible(tbase + t * kRows, N, W, t, t * kTok + quarter * 32 + lane, v);
#pragma unroll
            for (int r = 0; r < kRows; r += 2) {
                const float2 nb = *reinterpret_cast<const float2*>(ncm + r);
                const float2 x = tc::unpack2(tc::fma2(tc::pack2(v[r], v[r + 1]), c2,
                                                      tc::pack2(nb.x, nb.y)));
                v[r] = fast_exp2(x.x);
                v[r + 1] = fast_exp2(x.y);
                acc2[r >> 1] = tc::add2(acc2[r >> 1], tc::pack2(v[r], v[r + 1]));
            }
            tc::tmem_st32(tbase + t * kRows, v);
        }
        tc::tmem_st_wait();
#pragma unroll
        for (int r = 0; r < kRows; r += 2) {
            const float2 z2 = tc::unpack2(acc2[r >> 1]);
            acc[r] = z2.x;
            acc[r + 1] = z2.y;
        }
        xs[ew * kRows + lane] = transpose_reduce<false>(acc);
        if (!epi_sync(b, nsync)) { ok = false; break; }
        float z = 0.f;
        for (int w = 0; w < kEpiWarps; ++w) z += xs[w * kRows + lane];
        // a token's share of row r is p / (Z_r G W) (= A / (G W)): its weight
        // in B, and in Q for the last-position rows; padding rows weigh 0
        const float wr = z > 0.f ? 1.f / (z * (float)rows) : 0.f;
        wbq[lane] = make_float2(wr, (last >> lane) & 1u ? wr : 0.f);
        __syncwarp();
        // (3) the token's B (all rows), Q (last-position rows) and E: one
        // packed fma per row accumulates both
#pragma unroll
        for (int i = 0; i < (SPEC ? kSpecPerGroup : kMaxTiles / kGroups); ++i) {
            const int t = group + kGroups * i;
            if (!SPEC && t >= ntiles) break;
            const int tok = t * kTok + quarter * 32 + lane;
            tc::tmem_ld32(tbase + t * kRows, v);
            tc::tmem_ld_wait_regs32(v);
            unsigned long long bq[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
            for (int r = 0; r < kRows; ++r) {
                const float2 w2 = wbq[r];
                bq[r & 3] = tc::fma2(tc::pack2(v[r], v[r]), tc::pack2(w2.x, w2.y), bq[r & 3]);
            }
            const float2 s2 = tc::unpack2(tc::add2(tc::add2(bq[0], bq[1]), tc::add2(bq[2], bq[3])));
            const float bsum = s2.x, qsum = s2.y * (float)W;
            if (tok < N) {
                const size_t idx = (size_t)u * N + tok;
                a.B[idx] = bsum;
                a.Q[idx] = qsum;
                a.E[idx] = fmaxf(qsum - bsum, 0.f);
            }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(b.t_empty(slot));  // this unit's TMEM half is read
    }
    if (!ok) raise_abort(b, a.err);
}

template <int D, bool SPEC>
__global__ void __launch_bounds__(kThreads, 1) window_onepass_kernel(TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const Layout L = layout<D>();
    Bars b;
    b.base = smem_u32(sm + L.bars);
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(b.q_full(i), 1);
            tc::mbar_init(b.q_empty(i), 1);
            tc::mbar_init(b.t_full(i), 1);
            tc::mbar_init(b.t_empty(i), kEpiWarps);  // one arrival per epilogue warp
        }
        for (int i = 0; i < kStages; ++i) {
            tc::mbar_init(b.k_full(i), 1);
            tc::mbar_init(b.k_empty(i), 1);
        }
        tc::mbar_init(b.e_sync(), kEpiWarps);
        tc::mbar_init(b.drain(), 1);
        tc::st_shared_volatile(b.abort(), 0u);
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(b.tmem_slot(), 512);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();

    if (warp == 0)
        produce<D>(a, L, sm, b);
    else if (warp == 1) {
        if (tc::elect_one()) issue<D>(a, L, sm, b);
    } else {
        epilogue<D, SPEC>(a, L, sm, b);
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tc::ld_shared(b.tmem_slot()), 512);
    }
}

int num_sms_onepass()
{
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

template <int D, bool SPEC>
cudaError_t launch_d(const TcArgs& a, cudaStream_t st)
{
    const Layout L = layout<D>();
    size_t bytes = L.total + 1024;
    if (bytes < 116 * 1024) bytes = 116 * 1024;  // one CTA (one TMEM allocation) per SM
    cudaError_t e = cudaFuncSetAttribute(window_onepass_kernel<D, SPEC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    const int sms = num_sms_onepass();
    const int grid = a.s.units < sms ? a.s.units : sms;
    window_onepass_kernel<D, SPEC><<<grid, kThreads, bytes, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

bool window_onepass_fits(const Shape& s)
{
    return s.rows <= kRows && (s.d == 64 || s.d == 128) && (s.N + kTok - 1) / kTok <= kMaxTiles;
}

cudaError_t launch_window_onepass(const TcArgs& a, cudaStream_t st)
{
    if (!window_onepass_fits(a.s)) return cudaErrorInvalidValue;
    const bool spec = a.s.N == 1024 && a.s.W == 32 && a.s.rows == kRows;
    if (a.s.d == 128) return spec ? launch_d<128, true>(a, st) : launch_d<128, false>(a, st);
    return spec ? launch_d<64, true>(a, st) : launch_d<64, false>(a, st);
}

}  // namespace bacon
