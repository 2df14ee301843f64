// Window scores (Eqs. 1, 2, 4) on the 5th-generation tensor cores.
//
// Same two-pass structure as the softmax needs (see window.cu), built for
// sm_103a:
//   * K tiles (128 tokens x d) and the kv-head's G*W window rows are brought
//     into shared memory by TMA in the 128-byte-swizzled K-major layout that
//     tcgen05.mma reads directly;
//   * one thread issues tcgen05.mma (bf16 x bf16 -> fp32) into TMEM; the
//     accumulators never visit registers until the epilogue reads them;
//   * sixteen epilogue warps (four groups, each with one warp per TMEM lane
//     quarter) share every job's columns and turn logits into softmax
//     statistics (pass 1) or per-token sums (pass 2) while the MMA of the
//     next job runs into another TMEM buffer; exp2 runs on the SFU.
// Pass 1 (stats):  D[row][token], 128 rows x 128 tokens per job, 4 TMEM
//                  buffers; a thread owns one window row and 32 tokens.
// Pass 2 (scores): D[token][row], 128 tokens x up to 128 rows per job, 4
//                  TMEM buffers (so the next tile's MMA overlaps this tile's
//                  epilogue); a thread owns one token and every fourth
//                  16-row piece of the tile.
// Each CTA is persistent and takes a contiguous range of 1024-token chunks
// of the flattened (unit, chunk) space, so a CTA reloads the window rows only
// when its range crosses into the next (request, layer, kv-head).
// Every wait is bounded: on timeout the CTA raises an abort flag, records
// kErrTimeout in the error word, drains its own copies and MMAs, frees TMEM
// and returns.
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
    uint32_t q, k, tables, xchg, bars;
    uint32_t q_half;      // bytes of one 64-column half of the window rows
    uint32_t k_stage;     // bytes of one K tile
    uint32_t total;
};

template <int D, int PASS>
__host__ __device__ inline Smem smem_layout(int q_rows, int stages)
{
    Smem s;
    constexpr int H = D / 64;
    s.q_half = (uint32_t)q_rows * 128u;
    s.k_stage = (uint32_t)H * kTileTok * 128u;
    s.q = 0;
    s.k = s.q + H * s.q_half;
    s.tables = s.k + (uint32_t)stages * s.k_stage;
    // pass 2 only: per-row nl, qw and last visible key
    s.xchg = s.tables + (PASS == 2 ? (uint32_t)q_rows * 12u : 0u);
    s.xchg = (s.xchg + 15u) & ~15u;
    // partials of groups 1.. (pass 1: per row block; pass 2: two tiles) + flags
    s.bars = s.xchg + (kGroups - 1) * (PASS == 1 ? 4u : 2u) * 128u * 8u + 64u;
    s.bars = (s.bars + 7u) & ~7u;
    s.total = s.bars + 256u;  // barriers, TMEM base, abort flag
    return s;
}

struct Bars {
    uint64_t* k_full;   // [stages]
    uint64_t* k_empty;  // [stages]
    uint64_t* t_full;   // [4]
    uint64_t* t_empty;  // [4]
    uint64_t* q_full;
    uint64_t* q_empty;
    uint64_t* drain;
    uint64_t* ep_all;   // all epilogue warps
    uint64_t* ep_pair;  // [4] the two epilogue warps of a TMEM lane quarter
    uint32_t* tmem_base;
    volatile int* abort;
};

__device__ inline Bars bars_at(uint8_t* base, int stages)
{
    Bars b;
    uint64_t* p = reinterpret_cast<uint64_t*>(base);
    b.k_full = p;
    b.k_empty = p + stages;
    b.t_full = p + 2 * stages;
    b.t_empty = p + 2 * stages + 4;
    b.q_full = p + 2 * stages + 8;
    b.q_empty = p + 2 * stages + 9;
    b.drain = p + 2 * stages + 10;
    b.ep_all = p + 2 * stages + 11;
    b.ep_pair = p + 2 * stages + 12;
    b.tmem_base = reinterpret_cast<uint32_t*>(p + 2 * stages + 16);
    b.abort = reinterpret_cast<volatile int*>(p + 2 * stages + 17);
    return b;
}

// Barrier among epilogue warps built on an mbarrier (one arrival per warp),
// so that it shares the bounded, abort-aware wait of the pipeline.
__device__ inline bool warp_barrier(uint64_t* bar, int& phase, volatile int* abort)
{
    __syncwarp();
    if ((threadIdx.x & 31) == 0) tc::mbar_arrive(bar);
    const bool ok = tc::mbar_wait(bar, phase & 1, abort);
    ++phase;
    return ok;
}

__device__ inline void raise_abort(const Bars& b, int* err)
{
    *b.abort = 1;
    if (err) atomicExch(err, tc::kErrTimeout);
}

// Range of global chunks [c0, c1) owned by this CTA.
__device__ inline void chunk_range(int total, int* c0, int* c1)
{
    *c0 = (int)(((long long)blockIdx.x * total) / gridDim.x);
    *c1 = (int)(((long long)(blockIdx.x + 1) * total) / gridDim.x);
}

// Jobs of one tile.  Pass 1: n_jobs row blocks of 128 rows.  Pass 2: the
// window rows, rounded up to 16-row granules, split into n_jobs groups of at
// most 128 rows as evenly as granules allow.  The job loops are unrolled over
// the four possible jobs so the sizes stay in registers.
struct JobTable {
    int n_jobs;
    int n[4];
    int row0[4];
};

__device__ __forceinline__ JobTable make_jobs(int n_jobs, int granules)
{
    JobTable jt;
    jt.n_jobs = n_jobs;
    int r = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int nj = granules == 0
                           ? 128
                           : 16 * (granules / n_jobs + (j < granules % n_jobs ? 1 : 0));
        jt.n[j] = j < n_jobs ? nj : 0;
        jt.row0[j] = r;
        r += jt.n[j];
    }
    return jt;
}

// --------------------------------------------------- producer (TMA, warp 0)

template <int D>
__device__ __forceinline__ void produce(const TcArgs& a, const Smem& L, uint8_t* sm, const Bars& b, int stages,
                        int q_rows)
{
    constexpr int H = D / 64;
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int cur_u = -1, qloads = 0, kt = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        const int pair = u / s.hkv, h = u - pair * s.hkv;
        if (u != cur_u) {
            if (!tc::mbar_wait(b.q_empty, (qloads & 1) ^ 1, b.abort)) { ok = false; break; }
            tc::mbar_arrive_expect_tx(b.q_full, H * L.q_half);
            for (int kh = 0; kh < H; ++kh)
                for (int rb = 0; rb < q_rows / kQBox; ++rb)
                    tc::tma_load_2d(sm + L.q + kh * L.q_half + rb * kQBox * 128, a.qmaps + pair,
                                    kh * 64, h * s.rows + rb * kQBox, b.q_full);
            ++qloads;
            cur_u = u;
        }
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1; ++t, ++kt) {
            const int st = kt % stages, n = kt / stages;
            if (!tc::mbar_wait(b.k_empty + st, (n & 1) ^ 1, b.abort)) { ok = false; break; }
            tc::mbar_arrive_expect_tx(b.k_full + st, L.k_stage);
            for (int kh = 0; kh < H; ++kh)
                tc::tma_load_2d(sm + L.k + st * L.k_stage + kh * kTileTok * 128, a.kmaps + pair,
                                kh * 64, h * s.N + t * kTileTok, b.k_full + st);
        }
    }
    if (!ok) raise_abort(b, a.err);
    // drain: the last load of every stage (and of Q) must have landed before
    // this CTA's shared memory can be released
    volatile int never = 0;
    for (int st = 0; st < stages && st < kt; ++st) {
        const int last = kt - 1 - ((kt - 1 - st) % stages);
        tc::mbar_wait(b.k_full + st, (last / stages) & 1, &never);
    }
    if (qloads > 0) tc::mbar_wait(b.q_full, (qloads - 1) & 1, &never);
}

// ------------------------------------------------------ MMA issuer (warp 1)

// Pass 1: A = window rows (M = 128 per row block), B = K tile (N = 128).
// Pass 2: A = K tile (M = 128 tokens), B = window rows (N = n_h per half).
template <int D, int PASS>
__device__ __forceinline__ void issue(const TcArgs& a, const Smem& L, uint8_t* sm, const Bars& b, int stages,
                      int q_rows, const JobTable& jt)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const uint32_t tmem = *b.tmem_base;
    const uint32_t sbase = smem_u32(sm);
    constexpr int NBUF = 4;
    constexpr int BUF_COLS = 128;
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int cur_u = -1, qwaits = 0, kt = 0, job = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        if (u != cur_u) {
            if (cur_u >= 0) tc::umma_commit(b.q_empty);  // previous unit's MMAs release Q
            if (!tc::mbar_wait(b.q_full, qwaits & 1, b.abort)) { ok = false; break; }
            tc::fence_after_sync();
            ++qwaits;
            cur_u = u;
        }
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t, ++kt) {
            const int st = kt % stages, n = kt / stages;
            if (!tc::mbar_wait(b.k_full + st, n & 1, b.abort)) { ok = false; break; }
            tc::fence_after_sync();
            const uint32_t kaddr = sbase + L.k + st * L.k_stage;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (j >= jt.n_jobs) break;
                const int buf = job % NBUF, nb = job / NBUF;
                ++job;
                if (!tc::mbar_wait(b.t_empty + buf, (nb & 1) ^ 1, b.abort)) { ok = false; break; }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + buf * BUF_COLS;
                const uint32_t idesc = tc::idesc_bf16(128, jt.n[j]);
                const uint32_t qaddr = sbase + L.q + jt.row0[j] * 128;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const int kh = kk / 4;
                    const uint32_t koff = (kk % 4) * 32;
                    const uint64_t kd = tc::sdesc_sw128(kaddr + kh * kTileTok * 128 + koff);
                    const uint64_t qd = tc::sdesc_sw128(qaddr + kh * L.q_half + koff);
                    if (PASS == 1)
                        tc::umma_bf16(d_tmem, qd, kd, idesc, kk > 0);
                    else
                        tc::umma_bf16(d_tmem, kd, qd, idesc, kk > 0);
                }
                tc::umma_commit(b.t_full + buf);
            }
            tc::umma_commit(b.k_empty + st);  // the K stage is free once these MMAs finish
        }
    }
    if (!ok) raise_abort(b, a.err);
    // every MMA issued must complete before TMEM is released
    tc::umma_commit(b.drain);
    volatile int never = 0;
    tc::mbar_wait(b.drain, 0, &never);
    (void)q_rows;
}

// ------------------------------------------------- epilogue, pass 1 (stats)

// Thread = one window row (TMEM lane) x one 32-token quarter (its group) of
// every job; running (max, sum of 2^x) per row block, merged across the
// groups at the end of each chunk.
template <int D>
__device__ __forceinline__ void epilogue_stats(const TcArgs& a, const Smem& L, uint8_t* sm,
                                               const Bars& b, int q_rows)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3;        // TMEM lanes this warp may access
    const int group = (warp - 2) >> 2;   // which 32 tokens of each job
    const uint32_t tmem = *b.tmem_base;
    float2* xchg = reinterpret_cast<float2*>(sm + L.xchg);  // [group - 1][rb][128]
    const int nrb = q_rows / 128;
    const float c = kLog2e * rsqrtf((float)D);
    const unsigned long long c2 = tc::pack2(c, c);
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int job = 0, ep_phase = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        float m_run[4], z_run[4];
        int vis[4];
#pragma unroll
        for (int rb = 0; rb < 4; ++rb) {
            m_run[rb] = -INFINITY;
            z_run[rb] = 0.f;
            const int r = rb * 128 + quarter * 32 + lane;
            vis[rb] = s.N - s.W + (r % s.W);
        }
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t) {
            const int tok0 = t * kTileTok + group * 32;
            const bool need_mask = tok0 + 31 > s.N - s.W;
#pragma unroll
            for (int rb = 0; rb < 4; ++rb) {
                if (rb >= nrb) break;
                const int buf = job & 3, nb = job >> 2;
                ++job;
                if (!tc::mbar_wait(b.t_full + buf, nb & 1, b.abort)) { ok = false; break; }
                tc::fence_after_sync();
                float v[32];
                tc::tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + buf * 128 + group * 32, v);
                tc::tmem_ld_wait_regs32(v);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(b.t_empty + buf);
                if (need_mask) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (tok0 + j > vis[rb]) v[j] = -INFINITY;
                }
                float mx[4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    mx[i] = tc::max3(tc::max3(v[8 * i], v[8 * i + 1], v[8 * i + 2]),
                                     tc::max3(v[8 * i + 3], v[8 * i + 4], v[8 * i + 5]),
                                     fmaxf(v[8 * i + 6], v[8 * i + 7]));
                const float m_new = fmaxf(m_run[rb], fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * c);
                if (m_new != -INFINITY) {
                    const unsigned long long nm2 = tc::pack2(-m_new, -m_new);
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int j = 0; j < 32; j += 2) {
                        const float2 tt = tc::unpack2(tc::fma2(tc::pack2(v[j], v[j + 1]), c2, nm2));
                        acc[(j >> 1) & 3] += fast_exp2(tt.x) + fast_exp2(tt.y);
                    }
                    z_run[rb] = z_run[rb] * fast_exp2(m_run[rb] - m_new) + ((acc[0] + acc[1]) + (acc[2] + acc[3]));
                    m_run[rb] = m_new;
                }
            }
        }
        if (!ok) break;
        // merge the groups' statistics of each row, then publish the chunk's partial
        if (group > 0)
            for (int rb = 0; rb < nrb; ++rb)
                xchg[((group - 1) * 4 + rb) * 128 + quarter * 32 + lane] = make_float2(m_run[rb], z_run[rb]);
        if (!warp_barrier(b.ep_all, ep_phase, b.abort)) { ok = false; break; }
        if (group == 0) {
            for (int rb = 0; rb < nrb; ++rb) {
                const int r = rb * 128 + quarter * 32 + lane;
                float M = m_run[rb];
                for (int gg = 0; gg < kGroups - 1; ++gg)
                    M = fmaxf(M, xchg[(gg * 4 + rb) * 128 + quarter * 32 + lane].x);
                float Z = 0.f;
                if (M != -INFINITY) {
                    Z = z_run[rb] * fast_exp2(m_run[rb] - M);
                    for (int gg = 0; gg < kGroups - 1; ++gg) {
                        const float2 o = xchg[(gg * 4 + rb) * 128 + quarter * 32 + lane];
                        Z += o.y * fast_exp2(o.x - M);
                    }
                }
                if (r < s.rows)
                    a.partial[((size_t)u * a.chunks + ci) * s.rows + r] = make_float2(M, Z);
            }
        }
        if (!warp_barrier(b.ep_all, ep_phase, b.abort)) { ok = false; break; }
    }
    if (!ok) raise_abort(b, a.err);
}

// ------------------------------------------------ epilogue, pass 2 (scores)

// Thread = one token (TMEM lane); the 32-column chunks of a tile's jobs are
// dealt alternately to the two warps of a lane quarter.  Per-row terms in
// shared memory: nl = -(log2 of the row's softmax normaliser times G W);
// qw = W on the rows of the last window position (their sum is Q), else 0;
// the last key position each row may see; and, per 16-row group, whether
// its last row is a last-position row (with W a multiple of 16 that is the
// only place such a row can sit: FASTQ).
struct ScoreTabs {
    const float* nl;  // [q_rows] nl, then [q_rows] qw, then [q_rows] vis
    int q_rows;
    const uint8_t* qflag;
    __device__ __forceinline__ const float* qw() const { return nl + q_rows; }
    __device__ __forceinline__ const int* vis() const
    {
        return reinterpret_cast<const int*>(nl + 2 * q_rows);
    }
};

template <int NV, bool FASTQ, bool MASK>
__device__ __forceinline__ void score_chunk(const float* v, int r, const ScoreTabs& tb,
                                            unsigned long long c2, int tok, float* bacc,
                                            float* qacc, float& qlast)
{
#pragma unroll
    for (int jj = 0; jj < NV; jj += 4) {
        const float4 nl = *reinterpret_cast<const float4*>(tb.nl + r + jj);
        const float2 t0 = tc::unpack2(tc::fma2(tc::pack2(v[jj], v[jj + 1]), c2, tc::pack2(nl.x, nl.y)));
        const float2 t1 = tc::unpack2(tc::fma2(tc::pack2(v[jj + 2], v[jj + 3]), c2, tc::pack2(nl.z, nl.w)));
        float x0 = fast_exp2(t0.x), x1 = fast_exp2(t0.y);
        float x2 = fast_exp2(t1.x), x3 = fast_exp2(t1.y);
        if (MASK) {
            const int4 vis = *reinterpret_cast<const int4*>(tb.vis() + r + jj);
            if (tok > vis.x) x0 = 0.f;
            if (tok > vis.y) x1 = 0.f;
            if (tok > vis.z) x2 = 0.f;
            if (tok > vis.w) x3 = 0.f;
        }
        bacc[0] += x0;
        bacc[1] += x1;
        bacc[2] += x2;
        bacc[3] += x3;
        if (!FASTQ) {
            const float4 qw = *reinterpret_cast<const float4*>(tb.qw() + r + jj);
            qacc[0] = fmaf(x0, qw.x, qacc[0]);
            qacc[1] = fmaf(x1, qw.y, qacc[1]);
            qacc[0] = fmaf(x2, qw.z, qacc[0]);
            qacc[1] = fmaf(x3, qw.w, qacc[1]);
        } else if ((jj & 15) == 12) {
            if (tb.qflag[(r + jj) >> 4]) qlast += x3;  // the group's last column
        }
    }
}

template <bool FASTQ, bool MASK>
__device__ __forceinline__ bool score_tile(const JobTable& jt, int& job, int group, int quarter,
                                           uint32_t tmem,
                                           const Bars& b, const ScoreTabs& tb,
                                           unsigned long long c2, int tok, float* bacc,
                                           float* qacc, float& qlast)
{
    const int lane = threadIdx.x & 31;
    int kglob = 0;  // 16-column piece index of the tile where this job starts
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (j >= jt.n_jobs) break;
        const int buf = job & 3, nb = job >> 2;
        ++job;
        if (!tc::mbar_wait(b.t_full + buf, nb & 1, b.abort)) return false;
        tc::fence_after_sync();
        const int np = jt.n[j] / 16, r0 = jt.row0[j];
        const uint32_t taddr = tmem + ((uint32_t)(quarter * 32) << 16) + buf * 128;
        // pieces i = group, group + 4, ... of the tile that fall in this job
        for (int i = (group - kglob) & (kGroups - 1); i < np; i += kGroups) {
            float v[16];
            tc::tmem_ld16(taddr + 16 * i, v);
            tc::tmem_ld_wait_regs16(v);
            score_chunk<16, FASTQ, MASK>(v, r0 + 16 * i, tb, c2, tok, bacc, qacc, qlast);
        }
        kglob += np;
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(b.t_empty + buf);
    }
    return true;
}

template <int D, bool FASTQ>
__device__ __forceinline__ void epilogue_scores(const TcArgs& a, const Smem& L, uint8_t* sm, const Bars& b,
                                int q_rows, const JobTable& jt)
{
    const Shape& s = a.s;
    const int ntiles = (s.N + kTileTok - 1) / kTileTok;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3;
    const int group = (warp - 2) >> 2;
    const int et = threadIdx.x - 64;  // among the epilogue threads
    const uint32_t tmem = *b.tmem_base;
    float* nl_s = reinterpret_cast<float*>(sm + L.tables);  // [q_rows]
    float* qw_s = nl_s + q_rows;                            // [q_rows]
    int* vis_s = reinterpret_cast<int*>(qw_s + q_rows);     // [q_rows]
    uint8_t* qflag_s = reinterpret_cast<uint8_t*>(sm + L.xchg) + 2 * (kGroups - 1) * 128 * 8;  // [q_rows / 16]
    float2* xs = reinterpret_cast<float2*>(sm + L.xchg);    // [2][kGroups - 1][128]
    const ScoreTabs tb{nl_s, q_rows, qflag_s};
    const float c = kLog2e * rsqrtf((float)D);
    const unsigned long long c2 = tc::pack2(c, c);
    int c0, c1;
    chunk_range(a.total_chunks, &c0, &c1);
    int cur_u = -1, job = 0, ep_phase = 0, pair_phase = 0;
    bool ok = true;
    for (int g = c0; g < c1 && ok; ++g) {
        const int u = g / a.chunks, ci = g - u * a.chunks;
        if (u != cur_u) {
            // all epilogue warps are done with the previous unit's tables
            if (!warp_barrier(b.ep_all, ep_phase, b.abort)) { ok = false; break; }
            for (int r = et; r < q_rows; r += kEpiThreads) {
                const bool real = r < s.rows;
                const bool last = real && (r % s.W) == s.W - 1;
                nl_s[r] = real ? -a.lse2[(size_t)u * s.rows + r] : -INFINITY;
                qw_s[r] = last ? (float)s.W : 0.f;
                vis_s[r] = s.N - s.W + (r % s.W);
                if ((r & 15) == 15) qflag_s[r >> 4] = last ? 1 : 0;
            }
            if (!warp_barrier(b.ep_all, ep_phase, b.abort)) { ok = false; break; }
            cur_u = u;
        }
        const int t1 = min(ntiles, (ci + 1) * kTilesPerChunk);
        for (int t = ci * kTilesPerChunk; t < t1 && ok; ++t) {
            const int tok = t * kTileTok + quarter * 32 + lane;
            const bool need_mask = t * kTileTok + kTileTok - 1 > s.N - s.W;
            float bacc[4] = {0.f, 0.f, 0.f, 0.f};
            float qacc[2] = {0.f, 0.f};
            float qlast = 0.f;
            ok = need_mask ? score_tile<FASTQ, true>(jt, job, group, quarter, tmem, b, tb, c2, tok,
                                                     bacc, qacc, qlast)
                           : score_tile<FASTQ, false>(jt, job, group, quarter, tmem, b, tb, c2, tok,
                                                      bacc, qacc, qlast);
            if (!ok) break;
            float bsum = (bacc[0] + bacc[1]) + (bacc[2] + bacc[3]);
            float qsum = FASTQ ? qlast * (float)s.W : qacc[0] + qacc[1];
            // the groups' partial sums of a token meet in shared memory
            // (double-buffered by tile)
            float2* slots = xs + (t & 1) * (kGroups - 1) * 128 + quarter * 32 + lane;
            if (group > 0) slots[(group - 1) * 128] = make_float2(bsum, qsum);
            if (!warp_barrier(b.ep_pair + quarter, pair_phase, b.abort)) { ok = false; break; }
            if (group == 0 && tok < s.N) {
                for (int gg = 0; gg < kGroups - 1; ++gg) {
                    const float2 o = slots[gg * 128];
                    bsum += o.x;
                    qsum += o.y;
                }
                const size_t idx = (size_t)u * s.N + tok;
                a.B[idx] = bsum;
                a.Q[idx] = qsum;
                a.E[idx] = fmaxf(qsum - bsum, 0.f);
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
__global__ void __launch_bounds__(kThreads, 1) window_tc_kernel(TcArgs a, int q_rows, int stages,
                                                               int n_jobs, int granules)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const Smem L = smem_layout<D, PASS>(q_rows, stages);
    const Bars b = bars_at(sm + L.bars, stages);
    const int warp = threadIdx.x >> 5;
    const JobTable jt = make_jobs(n_jobs, granules);

    if (threadIdx.x == 0) {
        for (int i = 0; i < stages; ++i) {
            tc::mbar_init(b.k_full + i, 1);
            tc::mbar_init(b.k_empty + i, 1);
        }
        for (int i = 0; i < 4; ++i) {
            tc::mbar_init(b.t_full + i, 1);
            tc::mbar_init(b.t_empty + i, kEpiThreads / 32);  // one arrival per epilogue warp
        }
        tc::mbar_init(b.q_full, 1);
        tc::mbar_init(b.q_empty, 1);
        tc::mbar_init(b.drain, 1);
        tc::mbar_init(b.ep_all, kEpiThreads / 32);
        for (int i = 0; i < 4; ++i) tc::mbar_init(b.ep_pair + i, kGroups);
        *b.abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(b.tmem_base, kTmemCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();

    if (warp == 0) {
        if (tc::elect_one()) produce<D>(a, L, sm, b, stages, q_rows);
    } else if (warp == 1) {
        if (tc::elect_one()) issue<D, PASS>(a, L, sm, b, stages, q_rows, jt);
    } else {
        if (PASS == 1)
            epilogue_stats<D>(a, L, sm, b, q_rows);
        else if (a.s.W % 16 == 0)
            epilogue_scores<D, true>(a, L, sm, b, q_rows, jt);
        else
            epilogue_scores<D, false>(a, L, sm, b, q_rows, jt);
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::fence_after_sync();
        tc::tmem_dealloc(*b.tmem_base, kTmemCols);
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
    // pass 1: whole 128-row MMA blocks; pass 2: whole 64-row TMA boxes
    const int q_rows = PASS == 1 ? (rows + 127) / 128 * 128 : (rows + kQBox - 1) / kQBox * kQBox;
    const int granules = PASS == 1 ? 0 : (rows + 15) / 16;
    const int n_jobs = PASS == 1 ? q_rows / 128 : (granules + 7) / 8;
    int stages = 4;
    const size_t budget = 227 * 1024 - 1024;
    while (stages > 2 && smem_layout<D, PASS>(q_rows, stages).total > budget) --stages;
    const Smem L = smem_layout<D, PASS>(q_rows, stages);
    if (L.total > budget) return cudaErrorInvalidValue;
    // at least half of the SM's shared memory: one CTA (and one 512-column
    // TMEM allocation) per SM
    size_t bytes = L.total + 1024;
    if (bytes < 116 * 1024) bytes = 116 * 1024;
    cudaError_t e = cudaFuncSetAttribute(window_tc_kernel<D, PASS>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    const int grid = a.total_chunks < num_sms() ? a.total_chunks : num_sms();
    window_tc_kernel<D, PASS><<<grid, kThreads, bytes, st>>>(a, q_rows, stages, n_jobs, granules);
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
