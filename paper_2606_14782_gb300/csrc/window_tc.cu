// Window scores (Eqs. 1, 2, 4) on the 5th-generation tensor cores.
//
// A softmax row must be normalised over all N keys before any B_i is final,
// so K is streamed twice, by two persistent kernels built for sm_103a:
//   * K tiles (128 tokens x d) and the kv-head's G*W window rows are brought
//     into shared memory by TMA in the 128-byte-swizzled K-major layout that
//     tcgen05.mma reads directly;
//   * one thread issues tcgen05.mma (bf16 x bf16 -> fp32) into TMEM; the
//     accumulators never visit registers until the epilogue reads them;
//   * sixteen epilogue warps (four groups, each with one warp per TMEM lane
//     quarter) turn logits into softmax statistics (pass 1) or per-token
//     sums (pass 2) while the MMA of the next job runs into another TMEM
//     accumulator; exp2 runs on the SFU.
// Pass 1 (stats):  D[row][token], 128 rows x 128 tokens per job, four
//                  128-column accumulators; a thread owns one window row and
//                  32 tokens of every job.
// Pass 2 (scores): D[token][row], 128 tokens x up to 256 rows per job, two
//                  256-column accumulators (four of 128 when shared memory
//                  is short); the accumulator starts from each row's
//                  -lse2 / c (one extra MMA against a constant operand) and
//                  a thread owns one token and a share of a job's columns
//                  (32-column slices, or one 64-column range of a 224-column
//                  job).
// Each CTA takes a contiguous range of 1024-token chunks of the flattened
// (unit, chunk) space, so it reloads the window rows only when its range
// crosses into the next (request, layer, kv-head).  The epilogue groups meet
// through shared-memory slots and arrival counters, never at a barrier.
// The epilogues are bound by instruction issue, so the common plans are
// compiled with their job counts, job sizes and window as constants.
// Every wait is bounded: on timeout the CTA raises an abort flag, records
// kErrTimeout in the error word, drains its own copies and MMAs, frees TMEM
// and returns.
#include <cuda_bf16.h>

#include "tc.cuh"
#include "window_tc.h"

namespace bacon {
namespace {

constexpr int kTileTok = 128;          // tokens per K tile
constexpr int kChunk = 1024;           // tokens per work chunk (8 tiles)
constexpr int kTilesPerChunk = kChunk / kTileTok;
constexpr int kGroups = 4;             // epilogue warp groups (4 warps each, one per lane quarter)
constexpr int kEpiThreads = 128 * kGroups;
constexpr int kThreads = 64 + kEpiThreads;  // warp 0 TMA, warp 1 MMA, then the epilogue
constexpr int kQBox = 64;              // rows per TMA box of the window rows
constexpr int kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;

struct Smem {
    // offsets in bytes from the 1024-aligned dynamic shared memory base
    uint32_t q, k, ones, bias, xchg, bars;
    uint32_t q_half;      // bytes of one 64-column half of the window rows
    uint32_t q_slot;      // bytes of one slot of window rows (both halves)
    uint32_t bias_slot;   // bytes of one slot of the pass-2 bias operand
    uint32_t k_stage;     // bytes of one K tile
    uint32_t total;
};

// How a launch cuts the work: the window rows in shared memory (whole 64-row
// TMA boxes), the jobs of a tile (n_jobs jobs over `granules` 16-row
// granules), the number of K stages and of TMEM accumulator buffers
// (2^nbuf_log2 buffers of 512 >> nbuf_log2 columns).
//
// Pass 2 adds two bf16 operands in the same swizzled layout: a constant one
// for every token (columns 0-2) and, per job j, the row bias -lse2 / c split
// into three bf16 parts (columns 16 j .. 16 j + 2), so that one extra
// K = 16 MMA subtracts each row's normaliser inside the accumulator.  The
// bias operand has bias_rows rows (the largest job) x 64 columns.  The
// constant operand is 128 identical rows; when shared memory is short only
// its first 8-row atom is stored and its descriptor's 8-row stride is zero,
// so every group of 8 token rows reads the same atom.
struct Plan {
    int q_rows, n_jobs, granules, stages, nbuf_log2, bias_rows, ones_atom;
    int q_slots;   // 2: the next unit's window rows load while this unit's MMAs run
    int last_m64;  // pass 1: the last row block holds 64 window rows (an M = 64 job)
};

constexpr uint32_t kOnesBytes = 128u * 128u;
constexpr uint32_t kOnesAtomBytes = 8u * 128u;

template <int D, int PASS>
__host__ __device__ inline Smem smem_layout(const Plan& p)
{
    Smem s;
    constexpr int H = D / 64;
    s.q_half = (uint32_t)p.q_rows * 128u;
    s.q_slot = H * s.q_half;
    s.bias_slot = PASS == 2 ? (uint32_t)p.bias_rows * 128u : 0u;
    s.k_stage = (uint32_t)H * kTileTok * 128u;
    s.q = 0;
    s.k = s.q + (uint32_t)p.q_slots * s.q_slot;
    s.ones = s.k + (uint32_t)p.stages * s.k_stage;
    s.bias = s.ones + (PASS == 2 ? (p.ones_atom ? kOnesAtomBytes : kOnesBytes) : 0u);
    s.xchg = s.bias + (uint32_t)p.q_slots * s.bias_slot;
    // every group's partials: pass 1 per row block of a chunk, pass 2 for
    // two tiles
    s.bars = s.xchg + (PASS == 1 ? 4u : 2u) * kGroups * 128u * 8u;
    s.bars = (s.bars + 7u) & ~7u;
    s.total = s.bars + 272u + 16u * (uint32_t)p.stages;  // barriers, TMEM base, abort flag
    return s;
}

// Barrier block, 8-byte slots from `base` (a shared-memory address):
// t_full[4], t_empty[4], q_full[0], q_empty[0], drain, q_full[1],
// q_empty[1], three spare slots, the
// TMEM base word, the abort word, x_full[2][4], x_empty[2][4] (fixed
// offsets, so the epilogue's barrier addresses need no stage count), then
// k_full[stages], k_empty[stages].
struct Bars {
    uint32_t base;
    int stages;
    __device__ __forceinline__ uint32_t t_full(int i) const { return base + 8u * i; }
    __device__ __forceinline__ uint32_t t_empty(int i) const { return base + 32u + 8u * i; }
    __device__ __forceinline__ uint32_t q_full(int slot) const { return base + (slot ? 88u : 64u); }
    __device__ __forceinline__ uint32_t q_empty(int slot) const { return base + (slot ? 96u : 72u); }
    __device__ __forceinline__ uint32_t drain() const { return base + 80u; }
    __device__ __forceinline__ uint32_t tmem_slot() const { return base + 128u; }
    __device__ __forceinline__ uint32_t abort() const { return base + 136u; }
    // exchange slot p of lane quarter q (pass 1: p = 0 only): the three
    // non-merging groups' partials are in it / the merging group has read it
    __device__ __forceinline__ uint32_t x_full(int p, int q) const { return base + 144u + 8u * (4 * p + q); }
    __device__ __forceinline__ uint32_t x_empty(int p, int q) const
    {
        return base + 208u + 8u * (4 * p + q);
    }
    __device__ __forceinline__ uint32_t k_full(int st) const { return base + 272u + 8u * st; }
    __device__ __forceinline__ uint32_t k_empty(int st) const
    {
        return base + 272u + 8u * (stages + st);
    }
};

__device__ inline Bars bars_at(uint8_t* p, int stages)
{
    Bars b;
    b.base = smem_u32(p);
    b.stages = stages;
    return b;
}

__device__ inline void raise_abort(const Bars& b, int* err)
{
    tc::st_shared_volatile(b.abort(), 1u);
    if (err) atomicCAS(err, 0, tc::kErrTimeout);
}

// Range of global chunks [c0, c1) owned by this CTA.
__device__ inline void chunk_range(int total, int* c0, int* c1)
{
    *c0 = (int)(((long long)blockIdx.x * total) / gridDim.x);
    *c1 = (int)(((long long)(blockIdx.x + 1) * total) / gridDim.x);
}

// Jobs of one tile: the window rows, in 16-row granules, split into n_jobs
// jobs of at most 128 rows (8 granules) as evenly as granules allow; job j
// has n(j) rows starting at row0(j).  Pass 1 uses whole 128-row blocks
// (8 granules per job).
struct JobTable {
    int n_jobs;
    int q, rem;  // granules per job, and how many jobs take one more
    __device__ __forceinline__ int n(int j) const { return 16 * (q + (j < rem ? 1 : 0)); }
    __device__ __forceinline__ int row0(int j) const { return 16 * (j * q + min(j, rem)); }
};

__device__ __forceinline__ JobTable make_jobs(int n_jobs, int granules)
{
    JobTable jt;
    jt.n_jobs = n_jobs;
    jt.q = granules / n_jobs;
    jt.rem = granules - jt.q * n_jobs;
    return jt;
}

// --------------------------------------------------- producer (TMA, warp 0)

// Byte offset of element (row, col) of a 128-row x 64-column bf16 operand in
// the 128-byte-swizzled K-major layout (8-row atoms of 1024 bytes; the
// 16-byte chunks of a row are permuted by the row's position in its atom).
__device__ __forceinline__ uint32_t sw128_offset(int row, int col)
{
    return (uint32_t)((row >> 3) * 1024 + (row & 7) * 128 + ((((col * 2) >> 4) ^ (row & 7)) << 4) +
                      ((col * 2) & 15));
}

// Pass 2 bias operand of unit u: for job j and its row l (window row
// row0_j + l), columns 16 j .. 16 j + 2 hold -lse2 / c as three bf16 parts
// whose sum is the fp32 value to about 2^-24; rows beyond the window rows
// get a huge negative bias so their exponentials vanish.  Written by the 32
// lanes of the producer warp; columns 16 j + 3 .. stay zero.
__device__ __forceinline__ void write_bias(const TcArgs& a, uint8_t* bias, int u, const JobTable& jt,
                                           float inv_c)
{
    const Shape& s = a.s;
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (j >= jt.n_jobs) break;
        for (int l = lane; l < jt.n(j); l += 32) {
            const int r = jt.row0(j) + l;
            const float x = r < s.rows ? -a.lse2[(size_t)u * s.rows + r] * inv_c : -1.0e38f;
            const __nv_bfloat16 hi = __float2bfloat16_rn(x);
            const float r1 = x - __bfloat162float(hi);
            const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
            const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
            const uint32_t off = sw128_offset(l, 16 * j);
            *reinterpret_cast<uint32_t*>(bias + off) =
                (uint32_t)__bfloat16_as_ushort(hi) | ((uint32_t)__bfloat16_as_ushort(mid) << 16);
            *reinterpret_cast<uint32_t*>(bias + off + 4) = (uint32_t)__bfloat16_as_ushort(lo);
        }
    }
}

// All 32 lanes run the loop; lane 0 issues the copies.  At each new unit the
// window rows are reloaded once the previous unit's MMAs have released them
// (pass 2 also rewrites the bias operand, a second arrival on q_full).
template <int D, int PASS>
__device__ __forceinline__ void produce(const TcArgs& a, const Smem& L, uint8_t* sm, const Bars& b,
                                        int stages, int q_rows, int q_slots, const JobTable& jt)
{
    constexpr int H = D / 64;
    const Shape& s = a.s;
    const int lane = threadIdx.x & 31;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const float inv_c = sqrtf((float)D) / kLog2e;
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int cur_u = -1, qloads = 0, kt = 0;
    bool ok = true;
    const uint64_t kpol = tc::l2_evict_first_policy();  // K is read once per pass
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        const int pair = u / s.hkv, h = u - pair * s.hkv;
        if (u != cur_u) {
            const int slot = qloads % q_slots, use = qloads / q_slots;
            ok = __all_sync(0xffffffffu, tc::mbar_wait(b.q_empty(slot), (use & 1) ^ 1, b.abort()));
            if (!ok) break;
            uint8_t* qdst = sm + L.q + slot * L.q_slot;
            if (lane == 0) {
                tc::mbar_arrive_expect_tx(b.q_full(slot), L.q_slot);
                for (int kh = 0; kh < H; ++kh)
                    for (int rb = 0; rb < q_rows / kQBox; ++rb)
                        tc::tma_load_2d(qdst + kh * L.q_half + rb * kQBox * 128, a.qmaps + pair,
                                        kh * 64, h * s.rows + rb * kQBox, b.q_full(slot));
            }
            if (PASS == 2) {
                write_bias(a, sm + L.bias + slot * L.bias_slot, u, jt, inv_c);
                tc::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.q_full(slot));
            }
            ++qloads;
            cur_u = u;
        }
        if (lane == 0) {
            const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
            for (int t = ci * kTilesPerChunk; t < t1; ++t, ++kt) {
                const int st = kt % stages, n = kt / stages;
                if (!tc::mbar_wait(b.k_empty(st), (n & 1) ^ 1, b.abort())) { ok = false; break; }
                // injected fault (tests only): the first load never arrives, so
                // the MMA thread's bounded wait runs out and the CTA aborts
                if (PASS == 1 && a.fault == 1 && blockIdx.x == 0 && kt == 0) continue;
                tc::mbar_arrive_expect_tx(b.k_full(st), L.k_stage);
                for (int kh = 0; kh < H; ++kh)
                    tc::tma_load_2d_hint(sm + L.k + st * L.k_stage + kh * kTileTok * 128,
                                         a.kmaps + pair, kh * 64, h * s.N + t * kTileTok,
                                         b.k_full(st), kpol);
            }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    if (!ok) raise_abort(b, a.err);
    if (lane != 0) return;
    // drain: the last load of every stage (and of Q) must have landed before
    // this CTA's shared memory can be released
    for (int st = 0; st < stages && st < kt; ++st) {
        const int last = kt - 1 - ((kt - 1 - st) % stages);
        tc::mbar_wait(b.k_full(st), (last / stages) & 1, 0u);
    }
    for (int slot = 0; slot < q_slots && slot < qloads; ++slot) {
        const int last = qloads - 1 - ((qloads - 1 - slot) % q_slots);
        tc::mbar_wait(b.q_full(slot), (last / q_slots) & 1, 0u);
    }
}

// ------------------------------------------------------ MMA issuer (warp 1)

// Pass 1: A = window rows (M = 128 per row block), B = K tile (N = 128).
// Pass 2: A = K tile (M = 128 tokens), B = window rows (N = n_h per half).
template <int D, int PASS, int NBUF_LOG2>
__device__ __forceinline__ void issue(const TcArgs& a, const Smem& L, uint8_t* sm, const Bars& b, int stages,
                      int q_slots, const JobTable& jt, uint32_t ones_stride, int last_m64)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const uint32_t tmem = tc::ld_shared(b.tmem_slot());
    const uint32_t sbase = smem_u32(sm);
    constexpr int buf_mask = (1 << NBUF_LOG2) - 1;
    constexpr uint32_t buf_cols = (uint32_t)kTmemCols >> NBUF_LOG2;
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int cur_u = -1, cur_slot = 0, qwaits = 0, kt = 0, job = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        if (u != cur_u) {
            if (cur_u >= 0) tc::umma_commit(b.q_empty(cur_slot));  // previous unit's MMAs release its slot
            const int slot = qwaits % q_slots, use = qwaits / q_slots;
            if (!tc::mbar_wait(b.q_full(slot), use & 1, b.abort())) { ok = false; break; }
            tc::fence_after_sync();
            ++qwaits;
            cur_u = u;
            cur_slot = slot;
        }
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t, ++kt) {
            const int st = kt % stages, n = kt / stages;
            if (!tc::mbar_wait(b.k_full(st), n & 1, b.abort())) { ok = false; break; }
            tc::fence_after_sync();
            const uint32_t kaddr = sbase + L.k + st * L.k_stage;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (j >= jt.n_jobs) break;
                const int buf = job & buf_mask, nb = job >> NBUF_LOG2;
                ++job;
                if (!tc::mbar_wait(b.t_empty(buf), (nb & 1) ^ 1, b.abort())) { ok = false; break; }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + buf * buf_cols;
                // pass 1's last row block of 64 window rows: an M = 64 job,
                // which fills the first 16 lanes of each TMEM lane quarter
                const int m_rows = (PASS == 1 && last_m64 && j == jt.n_jobs - 1) ? 64 : 128;
                const uint32_t idesc = tc::idesc_bf16(m_rows, jt.n(j));
                const uint32_t qaddr = sbase + L.q + cur_slot * L.q_slot + jt.row0(j) * 128;
                if (PASS == 2)  // D = -lse2 / c per row (columns of D), then += K Q^T
                    tc::umma_bf16(d_tmem, tc::sdesc_sw128(sbase + L.ones, ones_stride),
                                  tc::sdesc_sw128(sbase + L.bias + cur_slot * L.bias_slot + 32 * j), idesc, 0);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const int kh = kk / 4;
                    const uint32_t koff = (kk % 4) * 32;
                    const uint64_t kd = tc::sdesc_sw128(kaddr + kh * kTileTok * 128 + koff);
                    const uint64_t qd = tc::sdesc_sw128(qaddr + kh * L.q_half + koff);
                    if (PASS == 1)
                        tc::umma_bf16(d_tmem, qd, kd, idesc, kk > 0);
                    else
                        tc::umma_bf16(d_tmem, kd, qd, idesc, 1);
                }
                tc::umma_commit(b.t_full(buf));
            }
            tc::umma_commit(b.k_empty(st));  // the K stage is free once these MMAs finish
        }
    }
    if (!ok) raise_abort(b, a.err);
    // every MMA issued must complete before TMEM is released
    tc::umma_commit(b.drain());
    tc::mbar_wait(b.drain(), 0, 0u);
}

// ------------------------------------------------- epilogue, pass 1 (stats)

// Maximum of NV logits by a tree of 3-input maxima.
template <int NV>
__device__ __forceinline__ float max_tree(const float* v)
{
    static_assert(NV == 32 || NV == 16, "32 or 16 logits");
    if constexpr (NV == 32) {
        float m9[11];
#pragma unroll
        for (int i = 0; i < 10; ++i) m9[i] = tc::max3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
        m9[10] = fmaxf(v[30], v[31]);
        const float mA = tc::max3(m9[0], m9[1], m9[2]);
        const float mB = tc::max3(m9[3], m9[4], m9[5]);
        const float mC = tc::max3(m9[6], m9[7], m9[8]);
        const float mD = fmaxf(m9[9], m9[10]);
        return fmaxf(tc::max3(mA, mB, mC), mD);
    } else {
        float m5[5];
#pragma unroll
        for (int i = 0; i < 5; ++i) m5[i] = tc::max3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
        return fmaxf(tc::max3(m5[0], m5[1], m5[2]), tc::max3(m5[3], m5[4], v[15]));
    }
}

// Folds NV more logits of one row, whose maximum is mx, into its running
// (max, sum of 2^(c x - max)), both in the log2 domain.  Masked logits are
// -inf.  (Exponentiating against the running maximum and redoing a job only
// when its sum overflows would save the maximum but costs a data-dependent
// branch per job, which measured slower than computing it.)
template <int NV, bool MASKED = true>
__device__ __forceinline__ void row_stats(const float* v, float mx, float c, unsigned long long c2,
                                          float& m_run, float& z_run)
{
    const float m_new = fmaxf(m_run, mx * c);
    if (MASKED && m_new == -INFINITY) return;
    const unsigned long long nm2 = tc::pack2(-m_new, -m_new);
    unsigned long long acc[2] = {0ull, 0ull};
#pragma unroll
    for (int j = 0; j < NV; j += 2) {
        const float2 tt = tc::unpack2(tc::fma2(tc::pack2(v[j], v[j + 1]), c2, nm2));
        acc[(j >> 1) & 1] = tc::add2(acc[(j >> 1) & 1], tc::pack2(fast_exp2(tt.x), fast_exp2(tt.y)));
    }
    const float2 s2 = tc::unpack2(tc::add2(acc[0], acc[1]));
    const float zs = s2.x + s2.y;
    // 2^0 = 1 when the maximum did not grow, 2^-inf = 0 for the first job
    z_run = z_run * fast_exp2(m_run - m_new) + zs;
    m_run = m_new;
}

// Thread = one window row (TMEM lane) x one 32-token quarter (its group) of
// every job; running (max, sum of 2^x) per row block, merged across the
// groups at the end of each chunk.  With last_m64 the last row block is an
// M = 64 job: its 64 rows sit in the first 16 lanes of each lane quarter,
// and a thread reads one of them and every other token of its 32 (16x64b
// shape), so the two threads holding a row combine their statistics before
// the merge.
template <int D, int J, bool H>
__device__ __forceinline__ void epilogue_stats(const TcArgs& a, const Smem& L, uint8_t* sm,
                                               const Bars& b, int q_rows, int last_m64_rt)
{
    // J > 0: every tile has J jobs (J - 1 full blocks and the half block when
    // H, else J full blocks), so a job's TMEM buffer and phase follow from the
    // tile count at compile-time offsets; J = 0: counted at run time
    const int last_m64 = J ? (H ? 1 : 0) : last_m64_rt;
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3;        // TMEM lanes this warp may access
    const int group = (warp - 2) >> 2;   // which 32 tokens of each job
    const uint32_t tmem = tc::ld_shared(b.tmem_slot());
    float2* xchg = reinterpret_cast<float2*>(sm + L.xchg);  // [group][rb][128]
    const int nrb = (q_rows + 127) / 128;
    const int nfull = J ? (H ? J - 1 : J) : (last_m64 ? nrb - 1 : nrb);  // 128-row blocks
    // window row of this thread in the half block, and its tokens 2 c + odd
    const int row_h = nfull * 128 + quarter * 16 + (lane >> 2) + 8 * (lane & 1);
    const int odd = (lane >> 1) & 1;
    const float c = kLog2e * rsqrtf((float)D);
    const unsigned long long c2 = tc::pack2(c, c);
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int job = 0, nch = 0, tcount = 0;
    bool ok = true;
    // the last position each of this thread's rows sees (rows of every block)
    int vis[4];
#pragma unroll
    for (int rb = 0; rb < 4; ++rb) vis[rb] = s.N - s.W + ((rb * 128 + quarter * 32 + lane) % s.W);
    const int vis_h = s.N - s.W + (row_h % s.W);
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        // running statistics per 128-row block, and of the half block,
        // restarted at every chunk: a chunk's partial depends on its own
        // logits only, whichever CTA and range of chunks processes it (every
        // launch shape gives the same bits)
        float m_run[4], z_run[4];
#pragma unroll
        for (int rb = 0; rb < 4; ++rb) {
            m_run[rb] = -INFINITY;
            z_run[rb] = 0.f;
        }
        float m_h = -INFINITY, z_h = 0.f;
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t) {
            const int tok0 = t * kTileTok + group * 32;
            const bool need_mask = tok0 + 31 > s.N - s.W;
            const int jt0 = tcount * J;  // this tile's first job (J > 0)
            ++tcount;
#pragma unroll
            for (int rb = 0; rb < 4; ++rb) {
                if (rb >= nfull) break;
                const int jj = J ? jt0 + rb : job++;
                const int buf = jj & 3, nb = jj >> 2;
                if (!tc::mbar_wait(b.t_full(buf), nb & 1, b.abort())) { ok = false; break; }
                tc::fence_after_sync();
                // the load also reduces the 32 logits to their maximum
                float v[32], mx;
                tc::tmem_ld32_max(tmem + ((uint32_t)(quarter * 32) << 16) + buf * 128 + group * 32, v,
                                  mx);
                tc::tmem_ld_wait_regs32_max(v, mx);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                if (need_mask) {
                    // tiles that reach into the window: mask, then the tree
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (tok0 + j > vis[rb]) v[j] = -INFINITY;
                    mx = max_tree<32>(v);
                    row_stats<32, true>(v, mx, c, c2, m_run[rb], z_run[rb]);
                } else {
                    row_stats<32, false>(v, mx, c, c2, m_run[rb], z_run[rb]);
                }
            }
            if (last_m64 && ok) {
                const int jj = J ? jt0 + (J - 1) : job++;
                const int buf = jj & 3, nb = jj >> 2;
                if (!tc::mbar_wait(b.t_full(buf), nb & 1, b.abort())) { ok = false; break; }
                tc::fence_after_sync();
                float v[16];
                tc::tmem_ld16x64b_x16(tmem + ((uint32_t)(quarter * 32) << 16) + buf * 128 + group * 32, v);
                tc::tmem_ld_wait_regs16(v);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                if (need_mask) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (tok0 + 2 * j + odd > vis_h) v[j] = -INFINITY;
                }
                row_stats<16>(v, max_tree<16>(v), c, c2, m_h, z_h);
            }
        }
        if (!ok) break;
        if (last_m64) {
            // the half block: the two threads of a row (lanes l and l ^ 2)
            // hold its even and odd tokens; combine them
            const float mo = __shfl_xor_sync(0xffffffffu, m_h, 2);
            const float zo = __shfl_xor_sync(0xffffffffu, z_h, 2);
            const float M = fmaxf(m_h, mo);
            if (M != -INFINITY) z_h = z_h * fast_exp2(m_h - M) + zo * fast_exp2(mo - M);
            m_h = M;
        }
        // merge the groups' statistics of each row and publish the chunk's
        // partial: group n mod 4 of this CTA's n-th chunk waits until the
        // other three groups of its lane quarter have left their (max, sum)
        // per row block in shared memory, merges them in group order and
        // frees the slot for the next chunk.  Every group, the merging one
        // included, first waits for the slot's previous read: a parity wait
        // is unambiguous only once the barrier's previous phase has
        // completed, and the merging group's x_full wait could otherwise pass
        // on the previous chunk's phase while a slower group is a chunk
        // behind.  (A lane holds the same row in every group.)
        const int merger = nch & 3;
        const uint32_t ph = (uint32_t)nch & 1u;
        ++nch;
        if (!tc::mbar_wait(b.x_empty(0, quarter), ph ^ 1u, b.abort())) {
            ok = false;
            break;
        }
        if (group != merger) {
#pragma unroll
            for (int rb = 0; rb < 4; ++rb) {
                if (rb >= nrb) break;
                const bool h = last_m64 && rb == nfull;
                xchg[(group * 4 + rb) * 128 + quarter * 32 + lane] =
                    h ? make_float2(m_h, z_h) : make_float2(m_run[rb], z_run[rb]);
            }
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(b.x_full(0, quarter));
        } else {
            if (!tc::mbar_wait(b.x_full(0, quarter), ph, b.abort())) {
                ok = false;
                break;
            }
            const float2* vx = xchg + quarter * 32 + lane;
#pragma unroll
            for (int rb = 0; rb < 4; ++rb) {
                if (rb >= nrb) break;
                const bool h = last_m64 && rb == nfull;
                float2 mz[kGroups];
#pragma unroll
                for (int gg = 0; gg < kGroups; ++gg)
                    mz[gg] = gg == group ? (h ? make_float2(m_h, z_h) : make_float2(m_run[rb], z_run[rb]))
                                         : vx[(gg * 4 + rb) * 128];
                float M = -INFINITY;
#pragma unroll
                for (int gg = 0; gg < kGroups; ++gg) M = fmaxf(M, mz[gg].x);
                float Z = 0.f;
                if (M != -INFINITY) {
#pragma unroll
                    for (int gg = 0; gg < kGroups; ++gg) {
                        const float zz = mz[gg].y * fast_exp2(mz[gg].x - M);
                        Z = gg == 0 ? zz : Z + zz;
                    }
                }
                const int r = h ? row_h : rb * 128 + quarter * 32 + lane;
                if ((!h || (lane & 2) == 0) && r < s.rows)
                    a.partial[((size_t)u * a.chunks + ci) * s.rows + r] = make_float2(M, Z);
            }
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(b.x_empty(0, quarter));
        }
    }
    if (!ok) raise_abort(b, a.err);
}

// ------------------------------------------------ epilogue, pass 2 (scores)

// Thread = one token (TMEM lane).  The accumulator of a job already holds
// logit - lse2 / c for each of its window rows (columns), so a column's share
// of B is 2^(c D) (= A_{q,i} / (G W)).  Each job's columns are cut into
// 32-column slices, one per group (a 224-column job into 64-column ranges),
// rotated from job to job so that the short last share moves between the
// groups.  Q sums the columns of last-position
// rows (scaled by W at the end, so that the G heads' rows average to Q).
struct ScoreCtx {
    unsigned long long c2;
    int N, W;
    uint32_t qmask;  // bit g: 16-row granule g ends on a last-position row
};

// WQ > 0: the window W (a multiple of 16) as a constant, so a granule's
// last-position test is a mask of its first row instead of a table lookup.
template <int NC, bool FASTQ, bool MASK, int WQ = 0>
__device__ __forceinline__ void score_slice(float* v, int r0, int tok, const ScoreCtx& k,
                                            unsigned long long* bacc, float& qacc)
{
    if (MASK) {
        // window row r sits at position N - W + (r mod W) and sees keys up to
        // it: this token is hidden from the rows with r mod W < tok - (N - W)
        const int lim = tok - (k.N - k.W);
        if (FASTQ) {
            // W % 16 == 0: r mod W runs up by one inside each 16-row granule
#pragma unroll
            for (int g = 0; g < NC / 16; ++g) {
                const int th = lim - (r0 + 16 * g) % k.W;
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    if (j < th) v[16 * g + j] = -INFINITY;
            }
        } else {
            int rm = r0 % k.W;
#pragma unroll
            for (int j = 0; j < NC; ++j) {
                if (rm < lim) v[j] = -INFINITY;
                rm = rm + 1 == k.W ? 0 : rm + 1;
            }
        }
    }
    int rm = FASTQ ? 0 : r0 % k.W;
    float q_end[NC / 16];  // FASTQ: the exponentials of the granules' last rows
#pragma unroll
    for (int j = 0; j < NC; j += 2) {
        const float2 t = tc::unpack2(tc::mul2(tc::pack2(v[j], v[j + 1]), k.c2));
        const float x0 = fast_exp2(t.x), x1 = fast_exp2(t.y);
        bacc[(j >> 1) & 1] = tc::add2(bacc[(j >> 1) & 1], tc::pack2(x0, x1));
        if (FASTQ) {
            if ((j & 15) == 14) q_end[j >> 4] = x1;
        } else {
            if (rm == k.W - 1) qacc += x0;
            rm = rm + 1 == k.W ? 0 : rm + 1;
            if (rm == k.W - 1) qacc += x1;
            rm = rm + 1 == k.W ? 0 : rm + 1;
        }
    }
    if (FASTQ) {
        // with W a multiple of 16 only a granule's last row can be a
        // last-position row: one mask test per granule, after the loop
#pragma unroll
        for (int g = 0; g < NC / 16; ++g) {
            const bool last_row = WQ ? (r0 + 16 * g + 16) % WQ == 0 : ((k.qmask >> ((r0 >> 4) + g)) & 1u);
            if (last_row) qacc += q_end[g];
        }
    }
}

// J > 0: every tile has J jobs and jt0 is this tile's first job, so a job's
// TMEM buffer, phase and slice rotation follow at compile-time offsets;
// J = 0: the jobs are counted at run time in `job`.  NPJ > 0: every job has
// NPJ 16-row granules, so its slices' sizes and first rows are constants.
// (Each instruction saved here is worth its share of the pass: the epilogue
// is bound by instruction issue.)
template <bool FASTQ, bool MASK, int NBUF_LOG2, int J, int NPJ, int WQ>
__device__ __forceinline__ bool score_tile(const JobTable& jt, int& job, int jt0, int rot0,
                                           int group, uint32_t tl, const Bars& b, const ScoreCtx& k,
                                           int tok, unsigned long long* bacc, float& qacc)
{
    const int lane = threadIdx.x & 31;
    constexpr uint32_t buf_cols = (uint32_t)kTmemCols >> NBUF_LOG2;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (j >= (J ? J : jt.n_jobs)) break;
        const int jj = J ? jt0 + j : job++;
        const int buf = jj & ((1 << NBUF_LOG2) - 1), nb = jj >> NBUF_LOG2;
        // the share rotation follows the tile's own index (rot0), not the
        // CTA's job count, so every launch shape sums a token's columns in
        // the same order (the same bits)
        const int sl = (group + rot0 + j) & (kGroups - 1);
        if (!tc::mbar_wait(b.t_full(buf), nb & 1, b.abort())) return false;
        tc::fence_after_sync();
        const int np = NPJ ? NPJ : jt.n(j) >> 4, ns = (np + 1) >> 1;
        // this group's 32-column slices of the job: sl, sl + 4, ...; the
        // buffer is released once the last of them is in registers
        const int mine = sl < ns ? (sl + kGroups < ns ? 2 : 1) : 0;
        if (mine == 0) {
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
        }
        if constexpr (NPJ == 14 && !MASK) {
            // 224 columns: the group of rotation sl takes columns [64 sl,
            // 64 sl + 64) (the last one [192, 224)) in one load pair and
            // releases the buffer once (fewer instructions per column)
            const uint32_t tb = tl + buf * buf_cols + 64 * sl;
            const int r0 = 16 * NPJ * j + 64 * sl;
            if (sl < 3) {
                float v[64];
                tc::tmem_ld32(tb, v);
                tc::tmem_ld32(tb + 32, v + 32);
                tc::tmem_ld_wait_regs32(v);
                tc::tmem_ld_wait_regs32(v + 32);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                score_slice<32, FASTQ, false, WQ>(v, r0, tok, k, bacc, qacc);
                score_slice<32, FASTQ, false, WQ>(v + 32, r0 + 32, tok, k, bacc, qacc);
            } else {
                float v[32];
                tc::tmem_ld32(tb, v);
                tc::tmem_ld_wait_regs32(v);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                score_slice<32, FASTQ, false, WQ>(v, r0, tok, k, bacc, qacc);
            }
        } else {
            for (int q = 0; q < mine; ++q) {
                const int sx = sl + kGroups * q;
                const uint32_t taddr = tl + buf * buf_cols + 32 * sx;
                const int r0 = (NPJ ? 16 * NPJ * j : jt.row0(j)) + 32 * sx;
                const bool two = (NPJ && NPJ % 2 == 0) ? true : 2 * sx + 1 < np;
                const bool last = q + 1 == mine;
                if (!MASK) {
                    float v[32];
                    if (two) {
                        tc::tmem_ld32(taddr, v);
                        tc::tmem_ld_wait_regs32(v);
                    } else {
                        tc::tmem_ld16(taddr, v);
                        tc::tmem_ld_wait_regs16(v);
                    }
                    if (last) {
                        tc::fence_before_sync();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                    }
                    if (two)
                        score_slice<32, FASTQ, false, WQ>(v, r0, tok, k, bacc, qacc);
                    else
                        score_slice<16, FASTQ, false, WQ>(v, r0, tok, k, bacc, qacc);
                } else {
                    // tiles that reach into the window (one or two per unit) go
                    // 16 columns at a time, keeping the masking's register demand low
                    float v[16];
                    for (int h = 0; h < (two ? 2 : 1); ++h) {
                        tc::tmem_ld16(taddr + 16 * h, v);
                        tc::tmem_ld_wait_regs16(v);
                        score_slice<16, FASTQ, true, WQ>(v, r0 + 16 * h, tok, k, bacc, qacc);
                    }
                    if (last) {
                        tc::fence_before_sync();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(b.t_empty(buf));
                    }
                }
            }
        }
    }
    return true;
}

template <int D, bool FASTQ, int NBUF_LOG2, int J, int NPJ, int WQ = 0>
__device__ __forceinline__ void epilogue_scores(const TcArgs& a, const Smem& L, uint8_t* sm,
                                                const Bars& b, const JobTable& jt)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3;
    const int group = (warp - 2) >> 2;
    const uint32_t tl = tc::ld_shared(b.tmem_slot()) + ((uint32_t)(quarter * 32) << 16);
    float2* xs = reinterpret_cast<float2*>(sm + L.xchg);  // [2][kGroups][128]
    ScoreCtx k;
    const float c = kLog2e * rsqrtf((float)D);
    k.c2 = tc::pack2(c, c);
    k.N = s.N;
    k.W = s.W;
    k.qmask = 0u;
    for (int g = 0; g < 32; ++g)
        if (16 * g + 15 < s.rows && (16 * g + 15) % s.W == s.W - 1) k.qmask |= 1u << g;
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int job = 0, ntile = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t) {
            const int tok = t * kTileTok + quarter * 32 + lane;
            const bool need_mask = t * kTileTok + kTileTok - 1 > s.N - s.W;
            unsigned long long bacc[2] = {0ull, 0ull};
            float qacc = 0.f;
            const int rot0 = t * (J ? J : jt.n_jobs);
            ok = need_mask
                     ? score_tile<FASTQ, true, NBUF_LOG2, J, NPJ, WQ>(jt, job, ntile * J, rot0, group,
                                                                    tl, b, k, tok, bacc, qacc)
                     : score_tile<FASTQ, false, NBUF_LOG2, J, NPJ, WQ>(jt, job, ntile * J, rot0, group,
                                                                     tl, b, k, tok, bacc, qacc);
            if (!ok) break;
            const float2 b2 = tc::unpack2(tc::add2(bacc[0], bacc[1]));
            const float bsum = b2.x + b2.y;
            const float qsum = qacc * (float)s.W;
            // the groups' partial sums of a token meet in shared memory (two
            // slots, used by this CTA's tiles in turn); group n mod 4 of the
            // CTA's n-th tile adds them in group order once the other three
            // have arrived on the slot's barrier, frees the slot and stores
            // the token's B, Q and E.  Every group, the merging one included,
            // first waits for the slot's previous read, so that the merging
            // group's parity wait on x_full cannot pass on the slot's previous
            // phase (with four TMEM buffers a group can run two tiles ahead
            // of another).
            const int par = ntile & 1;
            const uint32_t ph = (uint32_t)(ntile >> 1) & 1u;
            const int merger = ntile & 3;
            ++ntile;
            float2* slot = xs + (size_t)(par * kGroups) * 128 + quarter * 32 + lane;
            if (!tc::mbar_wait(b.x_empty(par, quarter), ph ^ 1u, b.abort())) {
                ok = false;
                break;
            }
            if (group != merger) {
                slot[group * 128] = make_float2(bsum, qsum);
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.x_full(par, quarter));
            } else {
                if (!tc::mbar_wait(b.x_full(par, quarter), ph, b.abort())) {
                    ok = false;
                    break;
                }
                float bt = 0.f, qt = 0.f;
#pragma unroll
                for (int gg = 0; gg < kGroups; ++gg) {
                    const float2 o = gg == group ? make_float2(bsum, qsum) : slot[gg * 128];
                    bt = gg == 0 ? o.x : bt + o.x;
                    qt = gg == 0 ? o.y : qt + o.y;
                }
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.x_empty(par, quarter));
                if (tok < s.N) {
                    const size_t idx = (size_t)u * s.N + tok;
                    a.B[idx] = bt;
                    a.Q[idx] = qt;
                    a.E[idx] = fmaxf(qt - bt, 0.f);
                }
            }
        }
    }
    if (!ok) raise_abort(b, a.err);
}

// ------------------------------------------------------------------ merge

// Per (unit, window row): log2 of the softmax normaliser over all chunks,
// plus log2(G W), so that pass 2's 2^(logit' - lse2) is A_{q,i} / (G W).
__global__ void window_combine_kernel(Shape s, int chunks, const float2* __restrict__ partial,
                                      float* __restrict__ lse2)
{
    const int u = blockIdx.x;
    const float log2_gw = log2f((float)s.rows);
    for (int r = threadIdx.x; r < s.rows; r += blockDim.x) {
        const float2* p = partial + (size_t)u * chunks * s.rows + r;
        float M = -INFINITY;
        for (int c = 0; c < chunks; ++c) M = fmaxf(M, p[(size_t)c * s.rows].x);
        float Z = 0.f;
        for (int c = 0; c < chunks; ++c) {
            const float2 v = p[(size_t)c * s.rows];
            if (v.y > 0.f) Z += v.y * exp2f(v.x - M);
        }
        lse2[(size_t)u * s.rows + r] = M + log2f(Z) + log2_gw;
    }
}

// Row normalisers supplied by the caller's prefill attention: per (request,
// layer) the natural-log LSE of each window row over the keys it sees,
// [Hq][W] = [Hkv][G W] -> lse2 = LSE log2(e) + log2(G W).
__global__ void lse_from_prefill_kernel(Shape s, LseTable t, float* __restrict__ lse2)
{
    const int u = blockIdx.x;
    const int pair = u / s.hkv, h = u - pair * s.hkv;
    const float log2_gw = log2f((float)s.rows);
    const float* src = t.lse[pair] + (size_t)h * s.rows;
    for (int r = threadIdx.x; r < s.rows; r += blockDim.x)
        lse2[(size_t)u * s.rows + r] = fmaf(src[r], kLog2e, log2_gw);
}

// --------------------------------------------------------------- kernels

template <int D, int PASS>
__global__ void __launch_bounds__(kThreads, 1) window_tc_kernel(TcArgs a, Plan pl)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const Smem L = smem_layout<D, PASS>(pl);
    const Bars b = bars_at(sm + L.bars, pl.stages);
    const int warp = threadIdx.x >> 5;
    const JobTable jt = make_jobs(pl.n_jobs, pl.granules);

    if (threadIdx.x == 0) {
        for (int i = 0; i < pl.stages; ++i) {
            tc::mbar_init(b.k_full(i), 1);
            tc::mbar_init(b.k_empty(i), 1);
        }
        for (int i = 0; i < 4; ++i) {
            tc::mbar_init(b.t_full(i), 1);
            tc::mbar_init(b.t_empty(i), kEpiThreads / 32);  // one arrival per epilogue warp
        }
        for (int slot = 0; slot < 2; ++slot) {
            tc::mbar_init(b.q_full(slot), PASS == 2 ? 2 : 1);  // pass 2: TMA bytes + the bias writes
            tc::mbar_init(b.q_empty(slot), 1);
        }
        tc::mbar_init(b.drain(), 1);
        for (int i = 0; i < 8; ++i) {
            tc::mbar_init(b.x_full(i >> 2, i & 3), kGroups - 1);
            tc::mbar_init(b.x_empty(i >> 2, i & 3), 1);
        }
        tc::st_shared_volatile(b.abort(), 0u);
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(b.tmem_slot(), kTmemCols);
        tc::tmem_relinquish();
    }
    if (PASS == 2 && threadIdx.x >= 64 && threadIdx.x < 64 + 128) {
        // constant operand: 1 in columns 0-2 of every token row (one atom of
        // 8 rows when ones_atom); the bias operand starts zeroed (the
        // producer fills columns 16 j .. 16 j + 2)
        const int row = threadIdx.x - 64;
        for (int rr = row; rr < pl.q_slots * pl.bias_rows; rr += 128) {
            uint4* bias = reinterpret_cast<uint4*>(sm + L.bias + rr * 128);
            for (int q = 0; q < 8; ++q) bias[q] = make_uint4(0u, 0u, 0u, 0u);
        }
        if (!pl.ones_atom || row < 8) {
            uint4* ones = reinterpret_cast<uint4*>(sm + L.ones + row * 128);
            for (int q = 0; q < 8; ++q) ones[q] = make_uint4(0u, 0u, 0u, 0u);
            uint8_t* r = sm + L.ones + sw128_offset(row, 0);
            *reinterpret_cast<uint32_t*>(r) = 0x3F803F80u;  // bf16 1.0, 1.0
            *reinterpret_cast<uint32_t*>(r + 4) = 0x00003F80u;
        }
        tc::fence_proxy_async_smem();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();

    if (warp == 0) {
        produce<D, PASS>(a, L, sm, b, pl.stages, pl.q_rows, pl.q_slots, jt);
    } else if (warp == 1) {
        if (tc::elect_one()) {
            const uint32_t ones_stride = pl.ones_atom ? 0u : 1024u;
            if (pl.nbuf_log2 == 1)
                issue<D, PASS, 1>(a, L, sm, b, pl.stages, pl.q_slots, jt, ones_stride, pl.last_m64);
            else
                issue<D, PASS, 2>(a, L, sm, b, pl.stages, pl.q_slots, jt, ones_stride, pl.last_m64);
        }
    } else {
        if (PASS == 1)
        {
            const int nrb = (pl.q_rows + 127) / 128;
            if (nrb == 4 && pl.last_m64)
                epilogue_stats<D, 4, true>(a, L, sm, b, pl.q_rows, pl.last_m64);
            else if (nrb == 2 && !pl.last_m64)
                epilogue_stats<D, 2, false>(a, L, sm, b, pl.q_rows, pl.last_m64);
            else
                epilogue_stats<D, 0, false>(a, L, sm, b, pl.q_rows, pl.last_m64);
        }
        else if (a.s.W % 16 == 0 && pl.nbuf_log2 == 1) {
            if (pl.n_jobs == 2 && pl.granules == 28 && a.s.W == 64)
                epilogue_scores<D, true, 1, 2, 14, 64>(a, L, sm, b, jt);
            else if (pl.n_jobs == 2 && pl.granules == 28)
                epilogue_scores<D, true, 1, 2, 14>(a, L, sm, b, jt);
            else if (pl.n_jobs == 2)
                epilogue_scores<D, true, 1, 2, 0>(a, L, sm, b, jt);
            else if (pl.n_jobs == 1 && pl.granules == 14 && a.s.W == 32)
                epilogue_scores<D, true, 1, 1, 14, 32>(a, L, sm, b, jt);
            else if (pl.n_jobs == 1 && pl.granules == 14)
                epilogue_scores<D, true, 1, 1, 14>(a, L, sm, b, jt);
            else if (pl.n_jobs == 1)
                epilogue_scores<D, true, 1, 1, 0>(a, L, sm, b, jt);
            else
                epilogue_scores<D, true, 1, 0, 0>(a, L, sm, b, jt);
        } else if (a.s.W % 16 == 0)
            epilogue_scores<D, true, 2, 0, 0>(a, L, sm, b, jt);
        else  // W % 16 != 0: always four accumulators (see launch_impl)
            epilogue_scores<D, false, 2, 0, 0>(a, L, sm, b, jt);
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(tc::ld_shared(b.tmem_slot()), kTmemCols);
    }
}

int num_sms()
{
    static int cache[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 1;
    if (cache[dev] == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = n > 0 ? n : 1;
    }
    return cache[dev];
}

template <int D, int PASS>
cudaError_t launch_impl(const TcArgs& a, cudaStream_t st)
{
    const int rows = a.s.rows;
    const size_t budget = 227 * 1024 - 1024;
    // window rows in shared memory: whole 64-row TMA boxes.  Pass 1 runs
    // whole 128-row MMA blocks over them in four 128-column accumulators; the
    // last block's rows beyond q_rows read the next shared-memory region and
    // their statistics are dropped (they are not window rows).  Pass 2 cuts
    // the rows into jobs of up to 256 rows (two 256-column accumulators, the
    // more efficient MMA shape) when shared memory allows, else up to 128.
    Plan pl;
    pl.q_rows = (rows + kQBox - 1) / kQBox * kQBox;
    pl.last_m64 = (PASS == 1 && pl.q_rows % 128 == 64) ? 1 : 0;
    const int granules = (rows + 15) / 16;
    Smem L;
    bool fits = false;
    // (a window that is not a multiple of 16 rows always takes 128-row jobs)
    for (int attempt = a.s.W % 16 == 0 ? 0 : 1; attempt < 2 && !fits; ++attempt) {
        const int per_job = PASS == 1 ? 8 : (attempt == 0 ? 16 : 8);  // granules
        pl.n_jobs = PASS == 1 ? (pl.q_rows + 127) / 128 : (granules + per_job - 1) / per_job;
        pl.granules = PASS == 1 ? 8 * pl.n_jobs : granules;
        pl.nbuf_log2 = per_job == 16 ? 1 : 2;
        pl.bias_rows = PASS == 2 ? 16 * ((pl.granules + pl.n_jobs - 1) / pl.n_jobs) : 0;
        // two slots of window rows when they fit beside at least three K
        // stages, else one
        for (pl.ones_atom = 0; pl.ones_atom < 2 && !fits; ++pl.ones_atom) {
            for (int qs = 2; qs >= 1 && !fits; --qs) {
                pl.q_slots = qs;
                for (pl.stages = 4; pl.stages > 2; --pl.stages)
                    if (smem_layout<D, PASS>(pl).total <= budget) break;
                L = smem_layout<D, PASS>(pl);
                fits = L.total <= budget && (qs == 1 || pl.stages >= 3);
            }
            if (fits) break;
        }
    }
    if (!fits) return cudaErrorInvalidValue;
    // at least half of the SM's shared memory: one CTA (and one 512-column
    // TMEM allocation) per SM
    size_t bytes = L.total + 1024;
    if (bytes < 116 * 1024) bytes = 116 * 1024;
    cudaError_t e = cudaFuncSetAttribute(window_tc_kernel<D, PASS>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    const int grid = a.total_chunks < num_sms() ? a.total_chunks : num_sms();
    window_tc_kernel<D, PASS><<<grid, kThreads, bytes, st>>>(a, pl);
    return cudaGetLastError();
}

}  // namespace

int window_tc_max_rows() { return 512; }

cudaError_t launch_lse_from_prefill(const Shape& s, const LseTable& t, float* lse2, cudaStream_t st)
{
    const int threads = s.rows < 512 ? ((s.rows + 31) / 32) * 32 : 512;
    lse_from_prefill_kernel<<<s.units, threads, 0, st>>>(s, t, lse2);
    return cudaGetLastError();
}

cudaError_t launch_window_combine(const Shape& s, int chunks, const float2* partial,
                                  float* lse2, cudaStream_t st)
{
    const int threads = s.rows < 512 ? ((s.rows + 31) / 32) * 32 : 512;
    window_combine_kernel<<<s.units, threads, 0, st>>>(s, chunks, partial, lse2);
    return cudaGetLastError();
}


cudaError_t launch_window_stats_tc(const TcArgs& a, cudaStream_t st)
{
    if (a.s.d == 128) return launch_impl<128, 1>(a, st);
    if (a.s.d == 64) return launch_impl<64, 1>(a, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_window_scores_tc(const TcArgs& a, cudaStream_t st)
{
    if (a.s.d == 128) return launch_impl<128, 2>(a, st);
    if (a.s.d == 64) return launch_impl<64, 2>(a, st);
    return cudaErrorInvalidValue;
}

// ------------------------------------------------------------ tensor maps

namespace {
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeFn g_encode = nullptr;
}  // namespace

bool encode_rows_map(CUtensorMap* out, const void* base, int d, long long rows, int box_rows)
{
    if (!g_encode) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn)
            return false;
        g_encode = reinterpret_cast<EncodeFn>(fn);
    }
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return g_encode(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace bacon
