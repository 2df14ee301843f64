// C ABI of the BACON library: argument checks, context and state ownership,
// and the launch sequence of the compression step.
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cmath>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "bacon.h"
#include "common.cuh"
#include "window_tc.h"

using namespace bacon;

namespace {

thread_local std::string g_last_error;

bacon_status fail(bacon_status st, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

bacon_status cuda_fail(cudaError_t e, const char* what)
{
    return fail(BACON_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define BACON_CUDA(call, what)                         \
    do {                                               \
        cudaError_t e_ = (call);                       \
        if (e_ != cudaSuccess) return cuda_fail(e_, what); \
    } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kChunkTokens = 1024;  // pass-1 token chunk (multiple of the 128-token tile)
constexpr int kMaxSeq = 24576;      // calibration keeps 2 x N fp32 in shared memory
static_assert(kMaxVariants == BACON_MAX_VARIANTS, "variant table size");

// Makes the context's device current for the duration of a call.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard()
    {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

template <typename T>
cudaError_t dalloc(T** p, size_t count)
{
    *p = nullptr;
    if (count == 0) return cudaSuccess;
    return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T));
}

}  // namespace

struct bacon_ctx {
    int device = 0;
    int layers = 0, hkv = 0, hq = 0, group = 0, d = 0, W = 0, pool = 1, budget = 0;
    int rows = 0;
    bacon_params p{};
    int max_chunks = 0;
    size_t unit_cap = 0;  // max_requests * layers * hkv
    float* B = nullptr;
    float* Q = nullptr;
    float* E = nullptr;
    float* S = nullptr;
    float* V = nullptr;
    float* Bp = nullptr;
    float* lam = nullptr;
    float* lse2 = nullptr;
    float2* partial = nullptr;
    int* err = nullptr;
    int last_units = 0, last_N = 0;
    // staging buffers of bacon_compress_host
    void* hq_buf = nullptr;
    void* hk_buf = nullptr;
    void* hv_buf = nullptr;
    void* hko_buf = nullptr;
    void* hvo_buf = nullptr;
    int32_t* hidx_buf = nullptr;
    size_t hq_cap = 0, hk_cap = 0, hv_cap = 0, hko_cap = 0, hvo_cap = 0, hidx_cap = 0;
    // TMA descriptors of the last whole-step call: [kMaxPairs] K maps, then
    // [kMaxPairs] window-query maps (device copy + pinned host staging)
    CUtensorMap* d_maps = nullptr;
    CUtensorMap* h_maps = nullptr;
    cudaEvent_t maps_ev = nullptr;
    std::vector<const void*> map_key;
    int map_key_N = -1;
    // host-buffer path: copy streams and per-request events
    cudaStream_t h2d = nullptr, d2h = nullptr;
    std::vector<cudaEvent_t> ev_in, ev_done;
    // per-kernel timing (bacon_profile_enable)
    int prof_on = 0;
    // test-only fault injection, read from the environment at bacon_init
    // (BACON_FAULT=missing_arrival): the next two-pass window step runs pass
    // 1 with one K-tile load withheld, so its bounded waits run out
    int fault_pending = 0;
    std::vector<cudaEvent_t> ev_free;
    std::vector<std::vector<cudaEvent_t>> ev_pending;  // 6 events per call
    std::vector<uint32_t> ev_skipped;                  // per call: stages that launched nothing
};

struct bacon_state {
    bacon_ctx* ctx = nullptr;
    int next_layer = 0;
    int N = 0;
    int scored = 0;
    int ring = 1;
    float* Ering = nullptr;  // [ring][hkv][max_seq_len]
    float* B = nullptr;
    float* Q = nullptr;
    float* S = nullptr;
    float* lam = nullptr;
    float* lse2 = nullptr;
    float2* partial = nullptr;
    CUtensorMap* d_maps = nullptr;  // [0] K map, [1] window-query map
    CUtensorMap* h_maps = nullptr;
    cudaEvent_t maps_ev = nullptr;
    std::vector<const void*> map_key;
    int map_key_N = -1;
};

namespace {

Calib calib_of(const bacon_ctx* c)
{
    Calib k;
    k.r = c->p.r;
    k.m = c->p.m;
    k.rho = c->p.rho;
    k.gamma = c->p.gamma;
    k.eps = c->p.eps;
    k.use_E = c->p.use_E;
    k.use_L = c->p.use_L;
    k.use_T = c->p.use_T;
    k.keep_window = c->p.keep_window;
    k.pool = c->pool;
    return k;
}

Shape shape_of(const bacon_ctx* c, int layers, int requests, int N)
{
    Shape s;
    s.layers = layers;
    s.hkv = c->hkv;
    s.group = c->group;
    s.d = c->d;
    s.W = c->W;
    s.N = N;
    s.units = requests * layers * c->hkv;
    s.rows = c->rows;
    return s;
}

bacon_status check_seq(const bacon_ctx* c, int N, int budget)
{
    if (N < c->W) return fail(BACON_EINVAL, "seq_len %d is shorter than the window %d", N, c->W);
    if (N > c->p.max_seq_len)
        return fail(BACON_EINVAL, "seq_len %d exceeds max_seq_len %d", N, c->p.max_seq_len);
    if (budget < 1) return fail(BACON_EINVAL, "budget must be positive");
    if (c->p.keep_window && budget < c->W)
        return fail(BACON_EINVAL, "budget %d is smaller than the window %d", budget, c->W);
    return BACON_OK;
}

// Encode the TMA descriptors of the (request, layer) pairs in slots
// [map0, map0 + pairs) and copy them to `d_maps` on the stream (K maps at
// [0, stride), query maps at [stride, 2 stride)); skipped when those slots
// already hold the same pointers for this N.
bacon_status upload_maps(const bacon_ctx* c, CUtensorMap* d_maps, CUtensorMap* h_maps,
                         cudaEvent_t ev, std::vector<const void*>& key, int& key_N, int stride,
                         int map0, int pairs, const void* const* q, const void* const* k, int N,
                         cudaStream_t st)
{
    if (key_N != N || (int)key.size() != 2 * stride) {
        key.assign(2 * stride, nullptr);  // every slot must be encoded again
        key_N = N;
    }
    bool same = true;
    for (int i = 0; same && i < pairs; ++i)
        same = key[2 * (map0 + i)] == k[i] && key[2 * (map0 + i) + 1] == q[i];
    if (same) return BACON_OK;
    BACON_CUDA(cudaEventSynchronize(ev), "descriptor staging wait");
    for (int i = 0; i < pairs; ++i) {
        if (!encode_rows_map(h_maps + map0 + i, k[i], c->d, (long long)c->hkv * N, kTcKBoxRows) ||
            !encode_rows_map(h_maps + stride + map0 + i, q[i], c->d, (long long)c->hq * c->W,
                             kTcQBoxRows))
            return fail(BACON_ECUDA, "cuTensorMapEncodeTiled failed for pair %d", map0 + i);
    }
    BACON_CUDA(cudaMemcpyAsync(d_maps + map0, h_maps + map0, sizeof(CUtensorMap) * pairs,
                               cudaMemcpyHostToDevice, st),
               "descriptor upload");
    BACON_CUDA(cudaMemcpyAsync(d_maps + stride + map0, h_maps + stride + map0,
                               sizeof(CUtensorMap) * pairs, cudaMemcpyHostToDevice, st),
               "descriptor upload");
    BACON_CUDA(cudaEventRecord(ev, st), "descriptor event");
    for (int i = 0; i < pairs; ++i) {
        key[2 * (map0 + i)] = k[i];
        key[2 * (map0 + i) + 1] = q[i];
    }
    return BACON_OK;
}

TcArgs tc_args(const Shape& s, const CUtensorMap* kmaps, const CUtensorMap* qmaps,
               float2* partial, const float* lse2, float* B, float* Q, float* E, int* err)
{
    TcArgs a;
    a.kmaps = kmaps;
    a.qmaps = qmaps;
    a.s = s;
    a.chunks = (s.N + kTcChunkTokens - 1) / kTcChunkTokens;
    a.total_chunks = s.units * a.chunks;
    a.partial = partial;
    a.lse2 = lse2;
    a.B = B;
    a.Q = Q;
    a.E = E;
    a.err = err;
    return a;
}

void free_ctx_buffers(bacon_ctx* c)
{
    for (cudaEvent_t e : c->ev_in) cudaEventDestroy(e);
    for (cudaEvent_t e : c->ev_done) cudaEventDestroy(e);
    c->ev_in.clear();
    c->ev_done.clear();
    if (c->h2d) cudaStreamDestroy(c->h2d);
    if (c->d2h) cudaStreamDestroy(c->d2h);
    c->h2d = c->d2h = nullptr;
    if (c->maps_ev) cudaEventDestroy(c->maps_ev);
    if (c->h_maps) cudaFreeHost(c->h_maps);
    if (c->d_maps) cudaFree(c->d_maps);
    c->maps_ev = nullptr;
    c->h_maps = nullptr;
    c->d_maps = nullptr;
    for (auto& v : c->ev_pending)
        for (cudaEvent_t e : v)
            if (e) cudaEventDestroy(e);
    for (cudaEvent_t e : c->ev_free)
        if (e) cudaEventDestroy(e);
    c->ev_pending.clear();
    c->ev_skipped.clear();
    c->ev_free.clear();
    void* bufs[] = {c->B,      c->Q,      c->E,      c->S,      c->V,      c->Bp,
                    c->lam,    c->lse2,   c->partial, c->err,   c->hq_buf, c->hk_buf,
                    c->hv_buf, c->hko_buf, c->hvo_buf, c->hidx_buf};
    for (void* b : bufs)
        if (b) cudaFree(b);
}

// Events bracketing the five launches of one call (profiling only).
struct StageEvents {
    bacon_ctx* c;
    cudaStream_t st;
    std::vector<cudaEvent_t> ev;
    StageEvents(bacon_ctx* c_, cudaStream_t st_) : c(c_), st(st_)
    {
        if (!c->prof_on) return;
        for (int i = 0; i < BACON_PROFILE_STAGES + 1; ++i) {
            cudaEvent_t e = nullptr;
            if (!c->ev_free.empty()) {
                e = c->ev_free.back();
                c->ev_free.pop_back();
            } else if (cudaEventCreate(&e) != cudaSuccess) {
                e = nullptr;
            }
            ev.push_back(e);
        }
    }
    uint32_t skipped = 0;
    bool range_open = false;
    // stage boundary i: CUDA-event timing (bacon_profile_enable) and an NVTX
    // range per stage ("bacon/window_stats", ...) around its launches, for
    // profilers (no cost without one attached)
    void mark(int i)
    {
        if (c->prof_on && ev[i]) cudaEventRecord(ev[i], st);
        static const char* const names[BACON_PROFILE_STAGES] = {
            "bacon/window_stats", "bacon/window_combine", "bacon/window_scores",
            "bacon/calibrate_select", "bacon/gather"};
        if (range_open) nvtxRangePop();
        range_open = i < BACON_PROFILE_STAGES;
        if (range_open) nvtxRangePushA(names[i]);
    }
    void skip(int i) { skipped |= 1u << i; }  // stage i launched nothing in this call
    void commit()
    {
        if (c->prof_on) {
            c->ev_pending.push_back(ev);
            c->ev_skipped.push_back(skipped);
        }
        ev.clear();
    }
    ~StageEvents()
    {
        if (range_open) nvtxRangePop();
        for (cudaEvent_t e : ev)  // a call that failed before commit()
            if (e) c->ev_free.push_back(e);
    }
};

// Window passes (Eqs. 1-4) of every unit of a call into the scratch slice
// that starts at unit `unit0`: B, Q and E.  With prefill_lse the window
// rows' normalisers come from the caller and pass 1 is skipped.
bacon_status window_passes(bacon_ctx* c, const Shape& s, const void* const* q,
                           const void* const* k, size_t unit0, const float* const* prefill_lse,
                           StageEvents& prof, cudaStream_t st, int map0 = 0)
{
    const int pairs = s.units / s.hkv, N = s.N;
    const int chunks = (N + kTcChunkTokens - 1) / kTcChunkTokens;
    float* lse2 = c->lse2 + unit0 * c->rows;
    float2* partial = c->partial + unit0 * chunks * c->rows;
    bacon_status rc = upload_maps(c, c->d_maps, c->h_maps, c->maps_ev, c->map_key, c->map_key_N,
                                  kMaxPairs, map0, pairs, q, k, N, st);
    if (rc != BACON_OK) return rc;
    TcArgs ta = tc_args(s, c->d_maps + map0, c->d_maps + kMaxPairs + map0, partial, lse2,
                        c->B + unit0 * N, c->Q + unit0 * N, c->E + unit0 * N, c->err);
    prof.mark(0);
    if (!prefill_lse && window_onepass_fits(s)) {
        // the unit's logits stay in tensor memory: one kernel, one pass over K
        // (timed as the scores stage)
        prof.mark(1);
        prof.mark(2);
        prof.skip(0);
        prof.skip(1);
        BACON_CUDA(launch_window_onepass(ta, st), "window_onepass launch");
        prof.mark(3);
        return BACON_OK;
    }
    if (prefill_lse) {
        prof.mark(1);
        prof.skip(0);
        LseTable t;
        for (int i = 0; i < pairs; ++i) t.lse[i] = prefill_lse[i];
        BACON_CUDA(launch_lse_from_prefill(s, t, lse2, st), "normaliser conversion launch");
    } else {
        if (c->fault_pending) {
            TcArgs tf = ta;
            tf.fault = 1;
            c->fault_pending = 0;
            BACON_CUDA(launch_window_stats_tc(tf, st), "window_stats launch");
        } else {
            BACON_CUDA(launch_window_stats_tc(ta, st), "window_stats launch");
        }
        prof.mark(1);
        BACON_CUDA(launch_window_combine(s, ta.chunks, partial, lse2, st), "window_combine launch");
    }
    prof.mark(2);
    BACON_CUDA(launch_window_scores_tc(ta, st), "window_scores launch");
    prof.mark(3);
    return BACON_OK;
}

// The whole step.  layer_budget[l] is the budget of layer l (window
// included); idx[pair] receives the pair's [Hkv][min(budget, N)] positions.
// With adaptive = true (uniform budget), the heads of each layer share the
// budget (AdaKV-style, g = guaranteed candidates per head first): idx[pair]
// and the K/V outputs are flat per pair, heads in order, with per-head kept
// counts in `counts`.
bacon_status compress_device(bacon_ctx* c, int R, const void* const* q, const void* const* k,
                             const void* const* v, int N, const int* layer_budget,
                             void* const* ko, void* const* vo, int32_t* const* idx,
                             cudaStream_t st, bool adaptive = false, int guaranteed = 0,
                             int32_t* counts = nullptr, size_t unit0 = 0,
                             const float* const* prefill_lse = nullptr, int map0 = 0)
{
    const int pairs = R * c->layers;
    const Shape s = shape_of(c, c->layers, R, N);
    float* B = c->B + unit0 * N;
    float* E = c->E + unit0 * N;
    float* S = c->S + unit0 * N;
    float* lam = c->lam + unit0;

    GatherTable gt;
    CalibArgs a;
    for (int i = 0; i < pairs; ++i) {
        const int budget = layer_budget[i % c->layers];
        gt.k[i] = static_cast<const uint16_t*>(k[i]);
        gt.v[i] = static_cast<const uint16_t*>(v[i]);
        gt.ko[i] = static_cast<uint16_t*>(ko[i]);
        gt.vo[i] = static_cast<uint16_t*>(vo[i]);
        gt.idx[i] = idx[i];
        gt.kept[i] = budget < N ? budget : N;
        a.idx[i] = idx[i];
        a.budget[i] = budget;
        a.calib_budget[i] = budget;
    }
    StageEvents prof(c, st);
    bacon_status rc = window_passes(c, s, q, k, unit0, prefill_lse, prof, st, map0);
    if (rc != BACON_OK) return rc;

    a.B = B;
    a.Ering = E;
    a.ring = c->layers;
    a.ring_req_stride = (long long)c->layers * c->hkv * N;
    a.layer0 = 0;
    a.S = S;
    a.V = c->p.keep_scores ? c->V + unit0 * N : nullptr;
    a.Bp = c->p.keep_scores ? c->Bp + unit0 * N : nullptr;
    a.lambda = lam;
    a.compute_scores = 1;
    a.do_select = adaptive ? 0 : 1;
    a.write_S = (c->p.keep_scores || adaptive) ? 1 : 0;
    a.err = c->err;
    BACON_CUDA(launch_calibrate_select(s, calib_of(c), a, st), "calibrate_select launch");
    if (adaptive) {
        AdaptArgs ad;
        ad.S = S;
        ad.budget = layer_budget[0];
        ad.guaranteed = guaranteed;
        for (int i = 0; i < pairs; ++i) {
            ad.idx[i] = idx[i];
            gt.kept[i] = c->hkv * (layer_budget[0] < N ? layer_budget[0] : N);
        }
        ad.counts = counts;
        ad.err = c->err;
        BACON_CUDA(launch_adaptive_select(s, c->p.keep_window, ad, st), "adaptive select launch");
    }
    prof.mark(4);
    if (adaptive)
        BACON_CUDA(launch_gather_flat(gt, s, counts, c->err, st), "gather launch");
    else
        BACON_CUDA(launch_gather(gt, s, c->err, st), "gather launch");
    prof.mark(5);
    prof.commit();
    c->last_units = (int)unit0 + s.units;
    c->last_N = N;
    return BACON_OK;
}

// Ablation / sensitivity sweep: one set of window passes, then calibration
// and selection of every unit under each variant.  idx receives int32
// [variants][pairs][Hkv][kept]; lambda_out (may be null) fp32
// [variants][units].
bacon_status sweep_device(bacon_ctx* c, int R, const void* const* q, const void* const* k, int N,
                          int budget, int variants, const bacon_variant* var, int32_t* idx,
                          float* lambda_out, cudaStream_t st)
{
    const int pairs = R * c->layers;
    const Shape s = shape_of(c, c->layers, R, N);
    const int kept = budget < N ? budget : N;
    CalibArgs a;
    for (int i = 0; i < pairs; ++i) {
        a.idx[i] = idx + (size_t)i * c->hkv * kept;
        a.budget[i] = budget;
        a.calib_budget[i] = budget;
    }
    CalibTable t;
    for (int j = 0; j < variants; ++j) {
        Calib& cj = t.c[j];
        cj = calib_of(c);
        cj.r = var[j].r;
        cj.m = var[j].m;
        cj.rho = var[j].rho;
        cj.gamma = var[j].gamma;
        cj.use_E = var[j].use_E;
        cj.use_L = var[j].use_L;
        cj.use_T = var[j].use_T;
    }
    StageEvents prof(c, st);
    bacon_status rc = window_passes(c, s, q, k, 0, nullptr, prof, st);
    if (rc != BACON_OK) return rc;
    a.B = c->B;
    a.Ering = c->E;
    a.ring = c->layers;
    a.ring_req_stride = (long long)c->layers * c->hkv * N;
    a.layer0 = 0;
    a.S = nullptr;
    a.V = nullptr;
    a.Bp = nullptr;
    a.lambda = lambda_out;
    a.idx_variant_stride = (long long)pairs * c->hkv * kept;
    a.compute_scores = 1;
    a.do_select = 1;
    a.write_S = 0;
    a.err = c->err;
    BACON_CUDA(launch_calibrate_sweep(s, t, variants, a, st), "calibrate_sweep launch");
    prof.mark(4);
    prof.mark(5);
    prof.commit();
    c->last_units = 0;  // S, V, B~ and lambda of the scratch are not this call's
    return BACON_OK;
}

// Device address of page-locked host memory the current device can read
// (registered or allocated through CUDA, 16-byte aligned), else null.
const void* host_device_pointer(const void* p)
{
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (at.type != cudaMemoryTypeHost || !at.devicePointer || !aligned16(at.devicePointer))
        return nullptr;
    return at.devicePointer;
}

bacon_status check_pointer_arrays(const bacon_ctx* c, int pairs, const void* const* q,
                                  const void* const* k, const void* const* v, void* const* ko,
                                  void* const* vo)
{
    if (!q || !k || !v || !ko || !vo) return fail(BACON_EINVAL, "null pointer array");
    for (int i = 0; i < pairs; ++i) {
        const void* ps[] = {q[i], k[i], v[i], ko[i], vo[i]};
        for (const void* p : ps) {
            if (!p) return fail(BACON_EINVAL, "null tensor pointer at pair %d", i);
            if (!aligned16(p)) return fail(BACON_EINVAL, "tensor pointer at pair %d is not 16-byte aligned", i);
        }
    }
    (void)c;
    return BACON_OK;
}

template <typename T>
bacon_status grow(T** buf, size_t* cap, size_t bytes, const char* what)
{
    if (*cap >= bytes) return BACON_OK;
    if (*buf) cudaFree(*buf);
    *buf = nullptr;
    *cap = 0;
    if (cudaMalloc(reinterpret_cast<void**>(buf), bytes) != cudaSuccess) {
        cudaGetLastError();
        return fail(BACON_ENOMEM, "cannot allocate %zu bytes for %s", bytes, what);
    }
    *cap = bytes;
    return BACON_OK;
}

}  // namespace

extern "C" {

void bacon_default_params(bacon_params* p)
{
    if (!p) return;
    p->r = 5;
    p->m = 4;
    p->rho = 2;
    p->gamma = 1.0f;
    p->eps = 1e-8f;
    p->use_E = 1;
    p->use_L = 1;
    p->use_T = 1;
    p->keep_window = 1;
    p->max_seq_len = 16384;
    p->max_requests = 4;
    p->keep_scores = 0;
}

const char* bacon_last_error(void) { return g_last_error.c_str(); }

bacon_status bacon_init(bacon_ctx** out, int layers, int kv_heads, int q_heads, int head_dim,
                        int window, int pool, int budget, const bacon_params* p)
{
    g_last_error.clear();
    if (!out) return fail(BACON_EINVAL, "out is NULL");
    *out = nullptr;
    bacon_params prm;
    if (p)
        prm = *p;
    else
        bacon_default_params(&prm);
    if (layers < 1 || kv_heads < 1 || q_heads < 1) return fail(BACON_EINVAL, "layers and heads must be positive");
    if (q_heads % kv_heads) return fail(BACON_EINVAL, "q_heads %d is not a multiple of kv_heads %d", q_heads, kv_heads);
    if (head_dim != 64 && head_dim != 128) return fail(BACON_EINVAL, "head_dim %d unsupported (64 or 128)", head_dim);
    if (window < 1) return fail(BACON_EINVAL, "window must be positive");
    if (pool < 1 || pool % 2 == 0) return fail(BACON_EINVAL, "pool width %d must be odd and positive", pool);
    if (prm.r < 0 || prm.m < 0 || prm.rho < 0) return fail(BACON_EINVAL, "r, m, rho must be >= 0");
    if (!(prm.gamma >= 0.f) || !(prm.eps >= 0.f)) return fail(BACON_EINVAL, "gamma and eps must be >= 0");
    if (prm.max_requests < 1) return fail(BACON_EINVAL, "max_requests must be positive");
    if ((long long)prm.max_requests * layers > kMaxPairs)
        return fail(BACON_EINVAL, "max_requests * layers = %lld exceeds %d",
                    (long long)prm.max_requests * layers, kMaxPairs);
    if (prm.max_seq_len < window || prm.max_seq_len > kMaxSeq)
        return fail(BACON_EINVAL, "max_seq_len %d outside [window, %d]", prm.max_seq_len, kMaxSeq);
    const int group = q_heads / kv_heads;
    const int rows = group * window;
    if (rows > window_tc_max_rows())
        return fail(BACON_EUNSUPPORTED, "group * window = %d exceeds %d", rows, window_tc_max_rows());
    if (budget < 1 || (prm.keep_window && budget < window))
        return fail(BACON_EINVAL, "budget %d invalid for window %d", budget, window);

    bacon_ctx* c = new (std::nothrow) bacon_ctx();
    if (!c) return fail(BACON_ENOMEM, "host allocation failed");
    cudaGetDevice(&c->device);
    c->layers = layers;
    c->hkv = kv_heads;
    c->hq = q_heads;
    c->group = group;
    c->d = head_dim;
    c->W = window;
    c->pool = pool;
    c->budget = budget;
    c->rows = rows;
    c->p = prm;
    c->max_chunks = (prm.max_seq_len + kChunkTokens - 1) / kChunkTokens;
    c->unit_cap = (size_t)prm.max_requests * layers * kv_heads;
    const size_t tok = c->unit_cap * (size_t)prm.max_seq_len;
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = dalloc(&c->B, tok);
    if (e == cudaSuccess) e = dalloc(&c->Q, tok);
    if (e == cudaSuccess) e = dalloc(&c->E, tok);
    if (e == cudaSuccess) e = dalloc(&c->S, tok);
    if (e == cudaSuccess) e = dalloc(&c->V, prm.keep_scores ? tok : 0);
    if (e == cudaSuccess) e = dalloc(&c->Bp, prm.keep_scores ? tok : 0);
    if (e == cudaSuccess) e = dalloc(&c->lam, c->unit_cap);
    if (e == cudaSuccess) e = dalloc(&c->lse2, c->unit_cap * rows);
    if (e == cudaSuccess) e = dalloc(&c->partial, c->unit_cap * c->max_chunks * rows);
    if (e == cudaSuccess) e = dalloc(&c->err, 1);
    if (e == cudaSuccess) e = cudaMemset(c->err, 0, sizeof(int));
    if (e == cudaSuccess) e = dalloc(&c->d_maps, 2 * (size_t)kMaxPairs);
    if (e == cudaSuccess)
        e = cudaHostAlloc(reinterpret_cast<void**>(&c->h_maps), 2 * kMaxPairs * sizeof(CUtensorMap),
                          cudaHostAllocDefault);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->maps_ev, cudaEventDisableTiming);
    if (e != cudaSuccess) {
        cudaGetLastError();
        free_ctx_buffers(c);
        delete c;
        return fail(BACON_ENOMEM, "device allocation failed: %s", cudaGetErrorString(e));
    }
    const char* fault = std::getenv("BACON_FAULT");  // tests only
    if (fault && std::strcmp(fault, "missing_arrival") == 0) c->fault_pending = 1;
    *out = c;
    return BACON_OK;
}

void bacon_destroy(bacon_ctx* ctx)
{
    if (!ctx) return;
    DeviceGuard dg(ctx->device);
    cudaDeviceSynchronize();
    free_ctx_buffers(ctx);
    delete ctx;
}

bacon_status bacon_state_create(bacon_ctx* ctx, bacon_state** out)
{
    g_last_error.clear();
    if (!ctx || !out) return fail(BACON_EINVAL, "null argument");
    DeviceGuard dg(ctx->device);
    bacon_state* st = new (std::nothrow) bacon_state();
    if (!st) return fail(BACON_ENOMEM, "host allocation failed");
    st->ctx = ctx;
    st->ring = ctx->p.m + 1;
    const size_t tok = (size_t)ctx->hkv * ctx->p.max_seq_len;
    const int chunks = ctx->max_chunks;
    cudaError_t e = dalloc(&st->Ering, tok * st->ring);
    if (e == cudaSuccess) e = dalloc(&st->B, tok);
    if (e == cudaSuccess) e = dalloc(&st->Q, tok);
    if (e == cudaSuccess) e = dalloc(&st->S, tok);
    if (e == cudaSuccess) e = dalloc(&st->lam, ctx->hkv);
    if (e == cudaSuccess) e = dalloc(&st->lse2, (size_t)ctx->hkv * ctx->rows);
    if (e == cudaSuccess) e = dalloc(&st->partial, (size_t)ctx->hkv * chunks * ctx->rows);
    if (e == cudaSuccess) e = dalloc(&st->d_maps, 2);
    if (e == cudaSuccess)
        e = cudaHostAlloc(reinterpret_cast<void**>(&st->h_maps), 2 * sizeof(CUtensorMap),
                          cudaHostAllocDefault);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&st->maps_ev, cudaEventDisableTiming);
    if (e != cudaSuccess) {
        cudaGetLastError();
        bacon_state_destroy(st);
        return fail(BACON_ENOMEM, "device allocation failed: %s", cudaGetErrorString(e));
    }
    *out = st;
    return BACON_OK;
}

bacon_status bacon_state_reset(bacon_state* st)
{
    if (!st) return fail(BACON_EINVAL, "null state");
    st->next_layer = 0;
    st->N = 0;
    st->scored = 0;
    return BACON_OK;
}

void bacon_state_destroy(bacon_state* st)
{
    if (!st) return;
    void* bufs[] = {st->Ering, st->B, st->Q, st->S, st->lam, st->lse2, st->partial, st->d_maps};
    for (void* b : bufs)
        if (b) cudaFree(b);
    if (st->h_maps) cudaFreeHost(st->h_maps);
    if (st->maps_ev) cudaEventDestroy(st->maps_ev);
    delete st;
}

bacon_status bacon_score_layer(bacon_ctx* ctx, bacon_state* st, int layer, const void* q_win,
                               const void* k, int seq_len, float* scores_out,
                               bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx || !st || st->ctx != ctx) return fail(BACON_EINVAL, "context/state mismatch");
    if (!q_win || !k || !aligned16(q_win) || !aligned16(k))
        return fail(BACON_EINVAL, "q_win and k must be non-null, 16-byte aligned device pointers");
    if (layer < 0 || layer >= ctx->layers) return fail(BACON_EINVAL, "layer %d out of range", layer);
    if (layer != st->next_layer)
        return fail(BACON_ESTATE, "layer %d scored out of order (expected %d)", layer, st->next_layer);
    bacon_status rc = check_seq(ctx, seq_len, ctx->budget);
    if (rc != BACON_OK) return rc;
    if (layer > 0 && seq_len != st->N)
        return fail(BACON_ESTATE, "seq_len changed within a request (%d vs %d)", seq_len, st->N);
    DeviceGuard dg(ctx->device);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);

    const Shape s = shape_of(ctx, 1, 1, seq_len);
    float* Eslot = st->Ering + (size_t)(layer % st->ring) * ctx->hkv * seq_len;
    rc = upload_maps(ctx, st->d_maps, st->h_maps, st->maps_ev, st->map_key, st->map_key_N, 1, 0, 1,
                     &q_win, &k, seq_len, cs);
    if (rc != BACON_OK) return rc;
    const TcArgs ta = tc_args(s, st->d_maps, st->d_maps + 1, st->partial, st->lse2, st->B, st->Q,
                              Eslot, ctx->err);
    BACON_CUDA(launch_window_stats_tc(ta, cs), "window_stats launch");
    BACON_CUDA(launch_window_combine(s, ta.chunks, st->partial, st->lse2, cs), "window_combine launch");
    BACON_CUDA(launch_window_scores_tc(ta, cs), "window_scores launch");

    CalibArgs a;
    a.B = st->B;
    a.Ering = st->Ering;
    a.ring = st->ring;
    a.ring_req_stride = 0;
    a.layer0 = layer;
    a.S = st->S;
    a.V = nullptr;
    a.Bp = nullptr;
    a.lambda = st->lam;
    a.idx[0] = nullptr;
    a.budget[0] = ctx->budget;
    a.calib_budget[0] = ctx->budget;
    a.compute_scores = 1;
    a.do_select = 0;
    a.write_S = 1;
    a.err = ctx->err;
    BACON_CUDA(launch_calibrate_select(s, calib_of(ctx), a, cs), "calibrate launch");
    if (scores_out)
        BACON_CUDA(cudaMemcpyAsync(scores_out, st->S, sizeof(float) * ctx->hkv * seq_len,
                                   cudaMemcpyDeviceToDevice, cs),
                   "score copy");
    st->N = seq_len;
    st->next_layer = layer + 1;
    st->scored = 1;
    return BACON_OK;
}

bacon_status bacon_select(bacon_ctx* ctx, bacon_state* st, int budget, int32_t* idx_out,
                          bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx || !st || st->ctx != ctx) return fail(BACON_EINVAL, "context/state mismatch");
    if (!st->scored) return fail(BACON_ESTATE, "no layer has been scored with this state");
    if (!idx_out || !aligned16(idx_out)) return fail(BACON_EINVAL, "idx_out must be a 16-byte aligned device pointer");
    bacon_status rc = check_seq(ctx, st->N, budget);
    if (rc != BACON_OK) return rc;
    DeviceGuard dg(ctx->device);
    const Shape s = shape_of(ctx, 1, 1, st->N);
    CalibArgs a;
    a.B = st->B;
    a.Ering = st->Ering;
    a.ring = st->ring;
    a.ring_req_stride = 0;
    a.layer0 = st->next_layer - 1;
    a.S = st->S;
    a.V = nullptr;
    a.Bp = nullptr;
    a.lambda = st->lam;
    a.idx[0] = idx_out;
    a.budget[0] = budget;
    a.calib_budget[0] = ctx->budget;
    a.compute_scores = 0;
    a.do_select = 1;
    a.write_S = 0;
    a.err = ctx->err;
    BACON_CUDA(launch_calibrate_select(s, calib_of(ctx), a, static_cast<cudaStream_t>(stream)),
               "select launch");
    return BACON_OK;
}

bacon_status bacon_compact(bacon_ctx* ctx, const void* k, const void* v, const int32_t* idx,
                           int seq_len, int count, void* k_out, void* v_out, bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    const void* ps[] = {k, v, idx, k_out, v_out};
    for (const void* p : ps)
        if (!p || !aligned16(p)) return fail(BACON_EINVAL, "tensor pointers must be non-null and 16-byte aligned");
    if (seq_len < 1 || seq_len > ctx->p.max_seq_len) return fail(BACON_EINVAL, "seq_len %d out of range", seq_len);
    if (count < 0 || count > seq_len) return fail(BACON_EINVAL, "count %d out of range", count);
    DeviceGuard dg(ctx->device);
    const Shape s = shape_of(ctx, 1, 1, seq_len);
    GatherTable gt;
    gt.k[0] = static_cast<const uint16_t*>(k);
    gt.v[0] = static_cast<const uint16_t*>(v);
    gt.ko[0] = static_cast<uint16_t*>(k_out);
    gt.vo[0] = static_cast<uint16_t*>(v_out);
    gt.idx[0] = idx;
    gt.kept[0] = count;
    BACON_CUDA(launch_gather(gt, s, ctx->err, static_cast<cudaStream_t>(stream)), "gather launch");
    return BACON_OK;
}

bacon_status bacon_compress_all_layers(bacon_ctx* ctx, int requests, const void* const* q_win,
                                       const void* const* k, const void* const* v, int seq_len,
                                       int budget, void* const* k_out, void* const* v_out,
                                       int32_t* idx_out, bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    bacon_status rc = check_seq(ctx, seq_len, budget);
    if (rc != BACON_OK) return rc;
    rc = check_pointer_arrays(ctx, requests * ctx->layers, q_win, k, v, k_out, v_out);
    if (rc != BACON_OK) return rc;
    if (!idx_out || !aligned16(idx_out)) return fail(BACON_EINVAL, "idx_out must be a 16-byte aligned device pointer");
    DeviceGuard dg(ctx->device);
    const int kept = budget < seq_len ? budget : seq_len;
    std::vector<int> budgets(ctx->layers, budget);
    int32_t* idx_pairs[kMaxPairs];
    for (int i = 0; i < requests * ctx->layers; ++i) idx_pairs[i] = idx_out + (size_t)i * ctx->hkv * kept;
    return compress_device(ctx, requests, q_win, k, v, seq_len, budgets.data(), k_out, v_out,
                           idx_pairs, static_cast<cudaStream_t>(stream));
}

bacon_status bacon_compress_layer_budgets(bacon_ctx* ctx, int requests, const void* const* q_win,
                                          const void* const* k, const void* const* v,
                                          int seq_len, const int* layer_budgets,
                                          void* const* k_out, void* const* v_out,
                                          int32_t* const* idx_out, bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    if (!layer_budgets || !idx_out) return fail(BACON_EINVAL, "null budget or index array");
    for (int l = 0; l < ctx->layers; ++l) {
        bacon_status rc = check_seq(ctx, seq_len, layer_budgets[l]);
        if (rc != BACON_OK) return rc;
    }
    bacon_status rc = check_pointer_arrays(ctx, requests * ctx->layers, q_win, k, v, k_out, v_out);
    if (rc != BACON_OK) return rc;
    for (int i = 0; i < requests * ctx->layers; ++i)
        if (!idx_out[i] || !aligned16(idx_out[i]))
            return fail(BACON_EINVAL, "index pointer of pair %d must be a 16-byte aligned device pointer", i);
    DeviceGuard dg(ctx->device);
    return compress_device(ctx, requests, q_win, k, v, seq_len, layer_budgets, k_out, v_out,
                           idx_out, static_cast<cudaStream_t>(stream));
}

bacon_status bacon_compress_with_lse(bacon_ctx* ctx, int requests, const void* const* q_win,
                                     const void* const* k, const void* const* v,
                                     const float* const* lse, int seq_len, int budget,
                                     void* const* k_out, void* const* v_out, int32_t* idx_out,
                                     bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    bacon_status rc = check_seq(ctx, seq_len, budget);
    if (rc != BACON_OK) return rc;
    rc = check_pointer_arrays(ctx, requests * ctx->layers, q_win, k, v, k_out, v_out);
    if (rc != BACON_OK) return rc;
    if (!lse) return fail(BACON_EINVAL, "null normaliser array");
    for (int i = 0; i < requests * ctx->layers; ++i)
        if (!lse[i] || (reinterpret_cast<uintptr_t>(lse[i]) & 3u))
            return fail(BACON_EINVAL, "normaliser pointer of pair %d must be a 4-byte aligned device pointer", i);
    if (!idx_out || !aligned16(idx_out)) return fail(BACON_EINVAL, "idx_out must be a 16-byte aligned device pointer");
    DeviceGuard dg(ctx->device);
    const int kept = budget < seq_len ? budget : seq_len;
    std::vector<int> budgets(ctx->layers, budget);
    int32_t* idx_pairs[kMaxPairs];
    for (int i = 0; i < requests * ctx->layers; ++i) idx_pairs[i] = idx_out + (size_t)i * ctx->hkv * kept;
    return compress_device(ctx, requests, q_win, k, v, seq_len, budgets.data(), k_out, v_out,
                           idx_pairs, static_cast<cudaStream_t>(stream), false, 0, nullptr, 0, lse);
}

bacon_status bacon_compress_adaptive(bacon_ctx* ctx, int requests, const void* const* q_win,
                                     const void* const* k, const void* const* v, int seq_len,
                                     int budget, float alpha, void* const* k_out,
                                     void* const* v_out, int32_t* const* idx_out,
                                     int32_t* counts_out, bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    if (!(alpha >= 0.f && alpha <= 1.f)) return fail(BACON_EINVAL, "alpha %g outside [0, 1]", (double)alpha);
    bacon_status rc = check_seq(ctx, seq_len, budget);
    if (rc != BACON_OK) return rc;
    rc = check_pointer_arrays(ctx, requests * ctx->layers, q_win, k, v, k_out, v_out);
    if (rc != BACON_OK) return rc;
    if (!idx_out || !counts_out || !aligned16(counts_out)) return fail(BACON_EINVAL, "null index or count array");
    for (int i = 0; i < requests * ctx->layers; ++i)
        if (!idx_out[i] || !aligned16(idx_out[i]))
            return fail(BACON_EINVAL, "index pointer of pair %d must be a 16-byte aligned device pointer", i);
    const int win = ctx->p.keep_window ? ctx->W : 0;
    if (adaptive_smem(ctx->hkv, seq_len - win) > 200 * 1024)
        return fail(BACON_EUNSUPPORTED, "kv_heads x candidates = %d exceeds the adaptive selection's %d",
                    ctx->hkv * (seq_len - win), 200 * 1024);
    const int kept = budget < seq_len ? budget : seq_len;
    const int guaranteed = (int)floor((double)alpha * (double)(kept - win));
    DeviceGuard dg(ctx->device);
    std::vector<int> budgets(ctx->layers, budget);
    return compress_device(ctx, requests, q_win, k, v, seq_len, budgets.data(), k_out, v_out,
                           idx_out, static_cast<cudaStream_t>(stream), true, guaranteed,
                           counts_out);
}

bacon_status bacon_sweep(bacon_ctx* ctx, int requests, const void* const* q_win,
                         const void* const* k, int seq_len, int budget, int n_variants,
                         const bacon_variant* variants, int32_t* idx_out, float* lambda_out,
                         bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    if (n_variants < 1 || n_variants > BACON_MAX_VARIANTS)
        return fail(BACON_EINVAL, "n_variants %d outside [1, %d]", n_variants, BACON_MAX_VARIANTS);
    if (!variants) return fail(BACON_EINVAL, "null variant array");
    for (int j = 0; j < n_variants; ++j) {
        const bacon_variant& x = variants[j];
        if (x.r < 0 || x.m < 0 || x.rho < 0)
            return fail(BACON_EINVAL, "variant %d: r, m, rho must be >= 0", j);
        if (!(x.gamma >= 0.f) || !(x.gamma < INFINITY))
            return fail(BACON_EINVAL, "variant %d: gamma must be finite and >= 0", j);
    }
    bacon_status rc = check_seq(ctx, seq_len, budget);
    if (rc != BACON_OK) return rc;
    const int pairs = requests * ctx->layers;
    if (!q_win || !k) return fail(BACON_EINVAL, "null pointer array");
    for (int i = 0; i < pairs; ++i)
        if (!q_win[i] || !k[i] || !aligned16(q_win[i]) || !aligned16(k[i]))
            return fail(BACON_EINVAL, "tensor pointer at pair %d is null or not 16-byte aligned", i);
    if (!idx_out || !aligned16(idx_out)) return fail(BACON_EINVAL, "idx_out must be a 16-byte aligned device pointer");
    if (lambda_out && (reinterpret_cast<uintptr_t>(lambda_out) & 3u))
        return fail(BACON_EINVAL, "lambda_out must be 4-byte aligned");
    DeviceGuard dg(ctx->device);
    return sweep_device(ctx, requests, q_win, k, seq_len, budget, n_variants, variants, idx_out,
                        lambda_out, static_cast<cudaStream_t>(stream));
}

void bacon_pyramid_budgets(int layers, int window, int budget, int beta, int* out)
{
    if (!out || layers < 1) return;
    const int K = budget - window;
    if (layers == 1 || beta < 1 || K <= 0) {
        for (int l = 0; l < layers; ++l) out[l] = budget;
        return;
    }
    const int lo = K / beta, hi = 2 * K - lo;
    for (int l = 0; l < layers; ++l)
        out[l] = window + lo + (int)((long long)(layers - 1 - l) * (hi - lo) / (layers - 1));
}

bacon_status bacon_compress_host(bacon_ctx* ctx, int requests, const void* q_win, const void* k,
                                 const void* v, int seq_len, int budget, void* k_out, void* v_out,
                                 int32_t* idx_out, bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx) return fail(BACON_EINVAL, "null context");
    if (!q_win || !k || !v || !k_out || !v_out || !idx_out) return fail(BACON_EINVAL, "null host buffer");
    if (requests < 1 || requests > ctx->p.max_requests)
        return fail(BACON_EINVAL, "requests %d outside [1, %d]", requests, ctx->p.max_requests);
    bacon_status rc = check_seq(ctx, seq_len, budget);
    if (rc != BACON_OK) return rc;
    DeviceGuard dg(ctx->device);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    const int pairs = requests * ctx->layers;
    const int kept = budget < seq_len ? budget : seq_len;
    const size_t q_pair = (size_t)ctx->hq * ctx->W * ctx->d;       // elements per (request, layer)
    const size_t kv_pair = (size_t)ctx->hkv * seq_len * ctx->d;
    const size_t o_pair = (size_t)ctx->hkv * kept * ctx->d;
    const size_t idx_count = (size_t)pairs * ctx->hkv * kept;
    if ((rc = grow(&ctx->hq_buf, &ctx->hq_cap, q_pair * pairs * 2, "queries")) != BACON_OK) return rc;
    // Values are only read where a row is kept (about budget / seq_len of
    // them): when the caller's value buffer is page-locked host memory the
    // device can address, the gather reads those rows in place instead of
    // uploading the whole tensor.
    const void* v_dev = host_device_pointer(v);
    if ((rc = grow(&ctx->hk_buf, &ctx->hk_cap, kv_pair * pairs * 2, "keys")) != BACON_OK) return rc;
    if (!v_dev &&
        (rc = grow(&ctx->hv_buf, &ctx->hv_cap, kv_pair * pairs * 2, "values")) != BACON_OK)
        return rc;
    if ((rc = grow(&ctx->hko_buf, &ctx->hko_cap, o_pair * pairs * 2, "compacted keys")) != BACON_OK)
        return rc;
    if ((rc = grow(&ctx->hvo_buf, &ctx->hvo_cap, o_pair * pairs * 2, "compacted values")) != BACON_OK)
        return rc;
    if ((rc = grow(&ctx->hidx_buf, &ctx->hidx_cap, idx_count * 4, "indices")) != BACON_OK) return rc;

    if (!ctx->h2d) {
        BACON_CUDA(cudaStreamCreateWithFlags(&ctx->h2d, cudaStreamNonBlocking), "copy stream");
        BACON_CUDA(cudaStreamCreateWithFlags(&ctx->d2h, cudaStreamNonBlocking), "copy stream");
    }
    while ((int)ctx->ev_in.size() < requests) {
        cudaEvent_t a = nullptr, b = nullptr;
        BACON_CUDA(cudaEventCreateWithFlags(&a, cudaEventDisableTiming), "event");
        BACON_CUDA(cudaEventCreateWithFlags(&b, cudaEventDisableTiming), "event");
        ctx->ev_in.push_back(a);
        ctx->ev_done.push_back(b);
    }
    // Requests are pipelined: every upload is queued on one copy stream, a
    // request is compressed on the caller's stream as soon as its inputs have
    // landed, and its outputs go back on a second copy stream while the next
    // request computes.
    const int L = ctx->layers;
    const char* qh = static_cast<const char*>(q_win);
    const char* kh = static_cast<const char*>(k);
    const char* vh = static_cast<const char*>(v);
    const void* qs[kMaxPairs];
    const void* ks[kMaxPairs];
    const void* vs[kMaxPairs];
    void* kos[kMaxPairs];
    void* vos[kMaxPairs];
    for (int i = 0; i < pairs; ++i) {
        qs[i] = static_cast<const uint16_t*>(ctx->hq_buf) + q_pair * i;
        ks[i] = static_cast<const uint16_t*>(ctx->hk_buf) + kv_pair * i;
        vs[i] = static_cast<const uint16_t*>(v_dev ? v_dev : ctx->hv_buf) + kv_pair * i;
        kos[i] = static_cast<uint16_t*>(ctx->hko_buf) + o_pair * i;
        vos[i] = static_cast<uint16_t*>(ctx->hvo_buf) + o_pair * i;
    }
    // The TMA descriptors of every request's staging buffers go to the
    // device first (cached across calls while the buffers stay the same): a
    // descriptor copy queued on the compute stream after the uploads would
    // wait behind all of them in the copy engine and hold back the first
    // request's kernels until the last upload had landed.
    {
        rc = upload_maps(ctx, ctx->d_maps, ctx->h_maps, ctx->maps_ev, ctx->map_key, ctx->map_key_N,
                         kMaxPairs, 0, pairs, qs, ks, seq_len, cs);
        if (rc != BACON_OK) return rc;
    }
    BACON_CUDA(cudaEventRecord(ctx->ev_done[0], cs), "event");  // uploads start after earlier work
    BACON_CUDA(cudaStreamWaitEvent(ctx->h2d, ctx->ev_done[0], 0), "event wait");
    for (int r = 0; r < requests; ++r) {
        const size_t qb = q_pair * L * 2, kb = kv_pair * L * 2;
        BACON_CUDA(cudaMemcpyAsync(static_cast<char*>(ctx->hq_buf) + r * qb, qh + r * qb, qb,
                                   cudaMemcpyHostToDevice, ctx->h2d), "query upload");
        BACON_CUDA(cudaMemcpyAsync(static_cast<char*>(ctx->hk_buf) + r * kb, kh + r * kb, kb,
                                   cudaMemcpyHostToDevice, ctx->h2d), "key upload");
        if (!v_dev)
            BACON_CUDA(cudaMemcpyAsync(static_cast<char*>(ctx->hv_buf) + r * kb, vh + r * kb, kb,
                                       cudaMemcpyHostToDevice, ctx->h2d), "value upload");
        BACON_CUDA(cudaEventRecord(ctx->ev_in[r], ctx->h2d), "event");
    }

    std::vector<int> budgets(L, budget);
    int32_t* idx_pairs[kMaxPairs];
    for (int i = 0; i < pairs; ++i) idx_pairs[i] = ctx->hidx_buf + (size_t)i * ctx->hkv * kept;
    for (int r = 0; r < requests; ++r) {
        BACON_CUDA(cudaStreamWaitEvent(cs, ctx->ev_in[r], 0), "event wait");
        rc = compress_device(ctx, 1, qs + r * L, ks + r * L, vs + r * L, seq_len, budgets.data(),
                             kos + r * L, vos + r * L, idx_pairs + r * L, cs, false, 0, nullptr,
                             (size_t)r * L * ctx->hkv, nullptr, r * L);
        if (rc != BACON_OK) return rc;
        BACON_CUDA(cudaEventRecord(ctx->ev_done[r], cs), "event");
        BACON_CUDA(cudaStreamWaitEvent(ctx->d2h, ctx->ev_done[r], 0), "event wait");
        const size_t ob = o_pair * L * 2, ib = (size_t)L * ctx->hkv * kept * 4;
        BACON_CUDA(cudaMemcpyAsync(static_cast<char*>(k_out) + r * ob,
                                   static_cast<char*>(ctx->hko_buf) + r * ob, ob,
                                   cudaMemcpyDeviceToHost, ctx->d2h), "key download");
        BACON_CUDA(cudaMemcpyAsync(static_cast<char*>(v_out) + r * ob,
                                   static_cast<char*>(ctx->hvo_buf) + r * ob, ob,
                                   cudaMemcpyDeviceToHost, ctx->d2h), "value download");
        BACON_CUDA(cudaMemcpyAsync(reinterpret_cast<char*>(idx_out) + r * ib,
                                   reinterpret_cast<char*>(ctx->hidx_buf) + r * ib, ib,
                                   cudaMemcpyDeviceToHost, ctx->d2h), "index download");
    }
    (void)idx_count;
    BACON_CUDA(cudaStreamSynchronize(ctx->d2h), "host-path synchronisation");
    BACON_CUDA(cudaStreamSynchronize(cs), "host-path synchronisation");
    return bacon_sync(ctx, stream);
}

bacon_status bacon_get_scores(bacon_ctx* ctx, bacon_score_kind kind, float* out, size_t count,
                              bacon_stream stream)
{
    g_last_error.clear();
    if (!ctx || !out) return fail(BACON_EINVAL, "null argument");
    if (ctx->last_units == 0) return fail(BACON_ESTATE, "no whole-step call has run yet");
    const size_t per_tok = (size_t)ctx->last_units * ctx->last_N;
    const float* src = nullptr;
    size_t n = per_tok;
    switch (kind) {
        case BACON_SCORE_B: src = ctx->B; break;
        case BACON_SCORE_Q: src = ctx->Q; break;
        case BACON_SCORE_E: src = ctx->E; break;
        case BACON_SCORE_V: src = ctx->V; break;
        case BACON_SCORE_BPOOL: src = ctx->Bp; break;
        case BACON_SCORE_S: src = ctx->S; break;
        case BACON_SCORE_LAMBDA:
            src = ctx->lam;
            n = ctx->last_units;
            break;
        default: return fail(BACON_EINVAL, "unknown score kind %d", (int)kind);
    }
    if (!src) return fail(BACON_ESTATE, "score kind %d is kept only with keep_scores = 1", (int)kind);
    if (count < n) return fail(BACON_EINVAL, "output holds %zu floats, %zu needed", count, n);
    DeviceGuard dg(ctx->device);
    BACON_CUDA(cudaMemcpyAsync(out, src, n * sizeof(float), cudaMemcpyDeviceToDevice,
                               static_cast<cudaStream_t>(stream)),
               "score copy");
    return BACON_OK;
}

bacon_status bacon_profile_enable(bacon_ctx* ctx, int enable)
{
    if (!ctx) return fail(BACON_EINVAL, "null context");
    ctx->prof_on = enable ? 1 : 0;
    return BACON_OK;
}

bacon_status bacon_profile_read(bacon_ctx* ctx, double* ms, int* launches, int n)
{
    if (!ctx || !ms || !launches) return fail(BACON_EINVAL, "null argument");
    if (n < 0 || n > BACON_PROFILE_STAGES) return fail(BACON_EINVAL, "n must be in [0, %d]", BACON_PROFILE_STAGES);
    DeviceGuard dg(ctx->device);
    for (int i = 0; i < n; ++i) {
        ms[i] = 0.0;
        launches[i] = 0;
    }
    bacon_status rc = BACON_OK;
    for (size_t c = 0; c < ctx->ev_pending.size(); ++c) {
        auto& v = ctx->ev_pending[c];
        const uint32_t skipped = c < ctx->ev_skipped.size() ? ctx->ev_skipped[c] : 0u;
        if (v.back() && cudaEventSynchronize(v.back()) != cudaSuccess) rc = fail(BACON_ECUDA, "event wait failed");
        for (int i = 0; i < n && rc == BACON_OK; ++i) {
            float t = 0.f;
            if ((skipped >> i) & 1u) continue;
            if (v[i] && v[i + 1] && cudaEventElapsedTime(&t, v[i], v[i + 1]) == cudaSuccess) {
                ms[i] += t;
                launches[i] += 1;
            }
        }
        for (cudaEvent_t e : v)
            if (e) ctx->ev_free.push_back(e);
    }
    ctx->ev_pending.clear();
    ctx->ev_skipped.clear();
    return rc;
}

bacon_status bacon_sync(bacon_ctx* ctx, bacon_stream stream)
{
    if (!ctx) return fail(BACON_EINVAL, "null context");
    DeviceGuard dg(ctx->device);
    BACON_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream synchronisation");
    int flag = 0;
    BACON_CUDA(cudaMemcpy(&flag, ctx->err, sizeof(int), cudaMemcpyDeviceToHost), "error flag read");
    if (flag) {
        // the word is cleared before the latched error is reported, so that
        // the context's next call starts clean
        BACON_CUDA(cudaMemset(ctx->err, 0, sizeof(int)), "error flag reset");
        if (flag == 1) return fail(BACON_EINVAL, "a gather index was outside [0, seq_len)");
        if (flag == 3) return fail(BACON_ETIMEOUT, "a window-score kernel timed out waiting on its pipeline");
        if (flag == 2)
            return fail(BACON_ECUDA, "internal check failed: a selection emitted a different count "
                                     "than its budget");
        return fail(BACON_ECUDA, "unknown device error code %d", flag);
    }
    return BACON_OK;
}

}  // extern "C"
