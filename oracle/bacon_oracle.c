/*
 * BACON CPU oracle -- TEST INFRASTRUCTURE ONLY (see bacon_oracle.h).
 *
 * Each function below is one equation of Section 4 written out literally in
 * double precision, with no blocking, fusion or reordering beyond what the
 * equation states.  Library routines used as steps: exp, sqrt, qsort.
 */
#include "bacon_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

void bo_default_params(bo_params* p)
{
    p->r = 5;           /* Section 4.3, "r = 5 by default"            */
    p->m = 4;           /* Section 4.3, "m = 4 by default"            */
    p->rho = 2;         /* Section 4.4, "rho = 2 by default"          */
    p->gamma = 1.0;     /* Section 4.4 gives no value; reading: 1     */
    p->eps = 1e-8;      /* Section 4.4 "small constant"; reading: 1e-8 */
    p->use_E = 1;
    p->use_L = 1;
    p->use_T = 1;
    p->pool_kernel = 7; /* SnapKV-style max pool of the backbone score */
    p->keep_window = 1;
}

void bo_bf16_to_double(const uint16_t* x, long n, double* out)
{
    for (long i = 0; i < n; ++i) {
        uint32_t bits = (uint32_t)x[i] << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        out[i] = (double)f;
    }
}

/* Section 4.1, Eq. 1 (observation-window score) and Section 4.2, Eq. 2
 * (last-query score).  The causal attention row of the query at position p
 * is softmax_i(q . k_i / sqrt(d)) over keys i <= p (scale: Appendix A). */
void bo_window_scores(const double* qwin, const double* k, int G, int W,
                      int N, int d, double* B, double* Q)
{
    const double scale = 1.0 / sqrt((double)d);
    double* row = (double*)malloc(sizeof(double) * (size_t)N);
    for (int i = 0; i < N; ++i) {
        B[i] = 0.0;
        Q[i] = 0.0;
    }
    for (int g = 0; g < G; ++g) {
        for (int w = 0; w < W; ++w) {
            const double* q = qwin + ((size_t)g * W + w) * d;
            const int p = N - W + w; /* position of this window query */
            double mx = -INFINITY;
            for (int i = 0; i <= p; ++i) {
                double s = 0.0;
                for (int c = 0; c < d; ++c) s += q[c] * k[(size_t)i * d + c];
                row[i] = s * scale;
                if (row[i] > mx) mx = row[i];
            }
            double z = 0.0;
            for (int i = 0; i <= p; ++i) {
                row[i] = exp(row[i] - mx);
                z += row[i];
            }
            for (int i = 0; i <= p; ++i) {
                const double a = row[i] / z; /* A_{q,i} */
                B[i] += a;
                if (w == W - 1) Q[i] += a; /* q = D, the last position */
            }
        }
    }
    for (int i = 0; i < N; ++i) {
        B[i] /= (double)G * (double)W; /* 1/|W|, and the mean over the group */
        Q[i] /= (double)G;
    }
    free(row);
}

/* Section 4.2, Eq. 4: E_i = [Q_i - B_i]_+ */
void bo_residual(const double* Q, const double* B, int N, double* E)
{
    for (int i = 0; i < N; ++i) {
        const double x = Q[i] - B[i];
        E[i] = x > 0.0 ? x : 0.0;
    }
}

/* Section 4.3, Eqs. 5-7: N_r(i) = {u : |u - i| <= r, u inside the
 * sequence}; (P_r)_{i,u} = 1/|N_r(i)| on N_r(i); L = P_r e. */
void bo_coherence(const double* E, int N, int r, double* L)
{
    for (int i = 0; i < N; ++i) {
        double sum = 0.0;
        int count = 0;
        for (int u = i - r; u <= i + r; ++u) {
            if (u < 0 || u >= N) continue;
            sum += E[u];
            ++count;
        }
        L[i] = sum / (double)count;
    }
}

/* Section 4.3, Eqs. 8-9: T_i = mean over j in P_m(l) of E^{j}_i, and 0 when
 * P_m(l) is empty. */
void bo_persistence(const double* const* E_prev, int n_prev, int N,
                    double* T)
{
    for (int i = 0; i < N; ++i) {
        if (n_prev == 0) {
            T[i] = 0.0;
            continue;
        }
        double sum = 0.0;
        for (int j = 0; j < n_prev; ++j) sum += E_prev[j][i];
        T[i] = sum / (double)n_prev;
    }
}

/* Section 4.3, Eq. 10: V = E + L + T (terms switchable for the ablation). */
void bo_evidence(const double* E, const double* L, const double* T, int N,
                 int use_E, int use_L, int use_T, double* V)
{
    for (int i = 0; i < N; ++i) {
        double v = 0.0;
        if (use_E) v += E[i];
        if (use_L) v += L[i];
        if (use_T) v += T[i];
        V[i] = v;
    }
}

void bo_maxpool(const double* x, int n, int kernel, double* y)
{
    const int half = kernel / 2;
    for (int i = 0; i < n; ++i) {
        double best = -INFINITY;
        for (int u = i - half; u <= i + half; ++u) {
            if (u < 0 || u >= n) continue;
            if (x[u] > best) best = x[u];
        }
        y[i] = best;
    }
}

typedef struct {
    double v;
    int32_t i;
} bo_item;

/* larger value first; equal values -> lower index first */
static int bo_item_cmp(const void* a, const void* b)
{
    const bo_item* x = (const bo_item*)a;
    const bo_item* y = (const bo_item*)b;
    if (x->v > y->v) return -1;
    if (x->v < y->v) return 1;
    return (x->i > y->i) - (x->i < y->i);
}

static int bo_int_cmp(const void* a, const void* b)
{
    const int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
    return (x > y) - (x < y);
}

/* TopK (Eqs. 13 and 17): a full sort of all n items under the total order
 * (value desc, index asc), then the first k. */
void bo_rank_topk(const double* x, int n, int k, int32_t* out)
{
    bo_item* items = (bo_item*)malloc(sizeof(bo_item) * (size_t)(n > 0 ? n : 1));
    for (int i = 0; i < n; ++i) {
        items[i].v = x[i];
        items[i].i = i;
    }
    qsort(items, (size_t)n, sizeof(bo_item), bo_item_cmp);
    for (int j = 0; j < k && j < n; ++j) out[j] = items[j].i;
    free(items);
}

/* population standard deviation of x over the positions sel[0..M) */
static double bo_std_over(const double* x, const int32_t* sel, int M)
{
    double mean = 0.0;
    for (int j = 0; j < M; ++j) mean += x[sel[j]];
    mean /= (double)M;
    double var = 0.0;
    for (int j = 0; j < M; ++j) {
        const double dlt = x[sel[j]] - mean;
        var += dlt * dlt;
    }
    return sqrt(var / (double)M);
}

/* Section 4.4, Eqs. 12-15: M = min(rho K, |I|); set = TopK of the backbone
 * score over the candidates; lambda = gamma Std(B) / (Std(V) + eps). */
double bo_lambda(const double* Bt, const double* V, int n_cand, int keep,
                 int rho, double gamma, double eps, int* M_out)
{
    long Ml = (long)rho * (long)keep;
    int M = Ml < n_cand ? (int)Ml : n_cand;
    if (M_out) *M_out = M;
    if (M <= 0) return 0.0; /* nothing is kept: no scale to match */
    int32_t* sel = (int32_t*)malloc(sizeof(int32_t) * (size_t)M);
    bo_rank_topk(Bt, n_cand, M, sel);
    const double sb = bo_std_over(Bt, sel, M);
    const double sv = bo_std_over(V, sel, M);
    free(sel);
    return gamma * sb / (sv + eps);
}

static int bo_check(int G, int W, int N, int d, const bo_params* p,
                    int budget)
{
    if (G < 1 || W < 1 || N < 1 || d < 1 || W > N) return -1;
    if (p->r < 0 || p->m < 0 || p->rho < 0) return -1;
    if (p->pool_kernel < 1 || (p->pool_kernel % 2) == 0) return -1;
    if (budget < 0) return -1;
    if (p->keep_window && budget < W) return -1;
    return 0;
}

/* number of candidates and of candidates kept for (N, W, budget) */
static void bo_sizes(int N, int W, int budget, const bo_params* p,
                     int* n_cand, int* keep)
{
    const int win = p->keep_window ? W : 0;
    const int kept_total = budget < N ? budget : N;
    *n_cand = N - win;
    *keep = kept_total - win;
}

int bo_score_unit(const double* qwin, const double* k, int G, int W, int N,
                  int d, const double* const* E_prev, int n_prev,
                  const bo_params* p, int budget,
                  double* B, double* Q, double* E, double* L, double* T,
                  double* V, double* Bt, double* S, double* lambda)
{
    if (bo_check(G, W, N, d, p, budget) != 0 || E == NULL) return -1;
    const size_t bytes = sizeof(double) * (size_t)N;
    double* b = (double*)malloc(bytes);
    double* q = (double*)malloc(bytes);
    double* l = (double*)malloc(bytes);
    double* t = (double*)malloc(bytes);
    double* v = (double*)malloc(bytes);
    double* bt = (double*)malloc(bytes);
    double* s = (double*)malloc(bytes);

    bo_window_scores(qwin, k, G, W, N, d, b, q); /* Eqs. 1-2 */
    bo_residual(q, b, N, E);                      /* Eq. 4 */
    bo_coherence(E, N, p->r, l);                  /* Eqs. 5-7 */
    bo_persistence(E_prev, n_prev, N, t);         /* Eqs. 8-9 */
    bo_evidence(E, l, t, N, p->use_E, p->use_L, p->use_T, v); /* Eq. 10 */

    int n_cand, keep;
    bo_sizes(N, W, budget, p, &n_cand, &keep);
    for (int i = 0; i < N; ++i) {
        bt[i] = 0.0;
        s[i] = 0.0;
    }
    bo_maxpool(b, n_cand, p->pool_kernel, bt);    /* pooled backbone */
    const double lam = bo_lambda(bt, v, n_cand, keep, p->rho, p->gamma,
                                 p->eps, NULL);   /* Eqs. 12-15 */
    for (int i = 0; i < n_cand; ++i) s[i] = bt[i] + lam * v[i]; /* Eq. 16 */

    if (B) memcpy(B, b, bytes);
    if (Q) memcpy(Q, q, bytes);
    if (L) memcpy(L, l, bytes);
    if (T) memcpy(T, t, bytes);
    if (V) memcpy(V, v, bytes);
    if (Bt) memcpy(Bt, bt, bytes);
    if (S) memcpy(S, s, bytes);
    if (lambda) *lambda = lam;
    free(b);
    free(q);
    free(l);
    free(t);
    free(v);
    free(bt);
    free(s);
    return 0;
}

/* Section 4.4, Eq. 17 and the cache construction that follows it. */
int bo_select(const double* S, int N, int W, int budget, const bo_params* p,
              int32_t* idx, double* gap)
{
    if (N < 1 || W < 1 || W > N || budget < 0) return -1;
    if (p->keep_window && budget < W) return -1;
    int n_cand, keep;
    bo_sizes(N, W, budget, p, &n_cand, &keep);
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)(n_cand > 0 ? n_cand : 1));
    bo_rank_topk(S, n_cand, n_cand, order);
    if (gap) {
        if (keep <= 0 || keep >= n_cand)
            *gap = INFINITY;
        else
            *gap = S[order[keep - 1]] - S[order[keep]];
    }
    for (int j = 0; j < keep; ++j) idx[j] = order[j];
    qsort(idx, (size_t)keep, sizeof(int32_t), bo_int_cmp);
    int count = keep;
    if (p->keep_window)
        for (int i = N - W; i < N; ++i) idx[count++] = i;
    free(order);
    return count;
}

void bo_gather(const uint16_t* x, int N, int d, const int32_t* idx,
               int count, uint16_t* out)
{
    (void)N;
    for (int j = 0; j < count; ++j)
        memcpy(out + (size_t)j * d, x + (size_t)idx[j] * d,
               sizeof(uint16_t) * (size_t)d);
}

/* Layer budgets of a linear pyramid from K_max at the first layer to K_min
 * at the last, each rounded down so that the total never exceeds the
 * uniform candidate budget K per layer. */
void bo_pyramid_budgets(int layers, int window, int budget, int beta, int* out)
{
    const int K = budget - window;
    if (layers <= 1) {
        if (layers == 1) out[0] = budget;
        return;
    }
    const int K_min = K / beta;
    const int K_max = 2 * K - K_min;
    for (int l = 0; l < layers; ++l) {
        const long long rise = (long long)(layers - 1 - l) * (K_max - K_min) / (layers - 1);
        out[l] = K_min + (int)rise + window;
    }
}

/* (score desc, head asc, position asc) over the flattened (head, position)
 * pairs; the flattened index h * n + i carries both tie-breaks. */
int bo_select_adaptive(const double* S, int H, int N, int W, int budget, double alpha,
                       const bo_params* p, int32_t* idx, int32_t* counts)
{
    if (H < 1 || N < 1 || W < 1 || W > N || budget < 0 || alpha < 0.0 || alpha > 1.0) return -1;
    if (p->keep_window && budget < W) return -1;
    int n_cand, keep;
    bo_sizes(N, W, budget, p, &n_cand, &keep);
    const int g = (int)floor(alpha * (double)keep);
    char* taken = (char*)calloc((size_t)H * (size_t)(n_cand > 0 ? n_cand : 1), 1);
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)(n_cand > 0 ? n_cand : 1));
    /* each head's guaranteed share */
    for (int h = 0; h < H; ++h) {
        bo_rank_topk(S + (size_t)h * N, n_cand, n_cand, order);
        for (int j = 0; j < g && j < n_cand; ++j) taken[(size_t)h * n_cand + order[j]] = 1;
    }
    /* the rest, jointly over all heads */
    const long total = (long)H * n_cand;
    double* rest = (double*)malloc(sizeof(double) * (size_t)(total > 0 ? total : 1));
    for (int h = 0; h < H; ++h)
        for (int i = 0; i < n_cand; ++i)
            rest[(size_t)h * n_cand + i] = taken[(size_t)h * n_cand + i] ? -INFINITY
                                                                        : S[(size_t)h * N + i];
    long R = (long)H * keep - (long)H * (g < n_cand ? g : n_cand);
    int32_t* jorder = (int32_t*)malloc(sizeof(int32_t) * (size_t)(total > 0 ? total : 1));
    bo_rank_topk(rest, (int)total, (int)total, jorder);
    for (long j = 0; j < R && j < total; ++j) taken[jorder[j]] = 1;
    for (int h = 0; h < H; ++h) {
        int c = 0;
        for (int i = 0; i < n_cand; ++i)
            if (taken[(size_t)h * n_cand + i]) idx[(size_t)h * N + c++] = i;
        if (p->keep_window)
            for (int i = N - W; i < N; ++i) idx[(size_t)h * N + c++] = i;
        counts[h] = c;
    }
    free(taken);
    free(order);
    free(rest);
    free(jorder);
    return 0;
}
