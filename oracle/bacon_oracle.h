/*
 * BACON CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, double-precision restatement of the BACON token-scoring
 * method (Boundary Attention CalibratiON, Sections 4.1-4.4, Eqs. 1-17) used
 * to check the CUDA library.  Only the test-suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it.  It shares no code, header or
 * constant with the CUDA library and the CUDA library never calls it.
 *
 * Conventions
 *   - positions are 0-based (the paper counts from 1; the sets are the same);
 *   - the observation window W is the last W prompt positions N-W .. N-1,
 *     the last query position D is N-1;
 *   - a kv-head h serves G = Hq/Hkv query heads; their window attention rows
 *     are averaged into the head's score (the paper does not address GQA;
 *     this is the reading both the oracle and the CUDA path follow);
 *   - every floating-point quantity is double; bf16 inputs are widened
 *     exactly.
 */
#ifndef BACON_ORACLE_H
#define BACON_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int r;            /* coherence radius, Eq. 5 (default 5)             */
    int m;            /* persistence depth, Eq. 8 (default 4)            */
    int rho;          /* scale-matching expansion, Eq. 12 (default 2)    */
    double gamma;     /* calibration strength, Eq. 14 (default 1)        */
    double eps;       /* stabiliser, Eq. 15 (default 1e-8)               */
    int use_E, use_L, use_T;   /* terms of Eq. 10 (ablation switches)    */
    int pool_kernel;  /* odd width of the 1-D max pool on B (7); 1 = none */
    int keep_window;  /* 1: window always kept, candidates = [0, N-W)     */
} bo_params;

void bo_default_params(bo_params* p);

/* exact bf16 -> double widening of n values */
void bo_bf16_to_double(const uint16_t* x, long n, double* out);

/* Eq. 1 and Eq. 2.  qwin [G][W][d] are the window queries of the G query
 * heads of one kv-head, query w sitting at position N-W+w; k [N][d].
 * B[i] = mean over (g, w) of softmax row (g, w) at key i (causal);
 * Q[i] = mean over g of the row of the last position N-1. */
void bo_window_scores(const double* qwin, const double* k, int G, int W,
                      int N, int d, double* B, double* Q);

/* Eq. 4: E = max(Q - B, 0) */
void bo_residual(const double* Q, const double* B, int N, double* E);

/* Eqs. 5-7: L = P_r e, truncated radius-r box mean */
void bo_coherence(const double* E, int N, int r, double* L);

/* Eqs. 8-9: T = mean of the given preceding-layer residuals (0 if none).
 * E_prev[j] are the residuals of the layers in P_m(l). */
void bo_persistence(const double* const* E_prev, int n_prev, int N,
                    double* T);

/* Eq. 10 with the ablation switches */
void bo_evidence(const double* E, const double* L, const double* T, int N,
                 int use_E, int use_L, int use_T, double* V);

/* 1-D max pool of width `kernel` (odd), stride 1, centred, positions
 * outside [0, n) ignored. */
void bo_maxpool(const double* x, int n, int kernel, double* y);

/* Order used by every TopK here: larger value first, ties -> lower index. */
/* Writes the k best positions of x[0..n) in rank order (best first). */
void bo_rank_topk(const double* x, int n, int k, int32_t* out);

/* Eqs. 12-15.  Bt and V over the candidate set [0, n_cand); keep = K_{l,h}.
 * Returns lambda; *M_out = |scale-matching set|. */
double bo_lambda(const double* Bt, const double* V, int n_cand, int keep,
                 int rho, double gamma, double eps, int* M_out);

/* Whole scoring path for one (layer, kv-head).  E_prev holds the residuals
 * of the layers in P_m(l) (n_prev of them).  Outputs (length N unless
 * stated): B, Q, E, L, T, V; Bt and S over the candidates (length N, with
 * non-candidates set to 0); *lambda.  Any output pointer may be NULL except E.
 * budget is the total number of kept tokens (window included when
 * keep_window). Returns 0, or -1 on an invalid argument. */
int bo_score_unit(const double* qwin, const double* k, int G, int W, int N,
                  int d, const double* const* E_prev, int n_prev,
                  const bo_params* p, int budget,
                  double* B, double* Q, double* E, double* L, double* T,
                  double* V, double* Bt, double* S, double* lambda);

/* Eq. 17 plus cache layout: kept positions in ascending order.  Writes
 * min(budget, N) indices.  gap (may be NULL) receives S_(k) - S_(k+1) at
 * the candidate boundary (or +inf when nothing is cut). */
int bo_select(const double* S, int N, int W, int budget, const bo_params* p,
              int32_t* idx, double* gap);

/* PyramidKV-style layer budgets (a base-compressor schedule BACON plugs into,
 * Sec. 5 / App. B): with K = budget - W candidates kept per layer on
 * average, K_min = floor(K / beta), K_max = 2 K - K_min, layer l keeps
 * K_min + floor((layers - 1 - l) (K_max - K_min) / (layers - 1)) candidates
 * (K for a single layer), plus the W window tokens.  out[l] = that budget;
 * the layers together keep at most layers x K candidates. */
void bo_pyramid_budgets(int layers, int window, int budget, int beta, int* out);

/* AdaKV-style adaptive per-head budgets for one (request, layer), the base
 * compressor of Sec. 5 / App. B that spreads a layer's budget over its heads.
 * S [H][N] holds each head's final score (Eq. 16) over its candidates.  With
 * K = budget - W per head on average, every head first keeps its own top
 * g = floor(alpha K) candidates; the remaining H K - H g slots go to the best
 * remaining candidates of all heads together (larger score first, ties to
 * the lower head, then the lower position).  Head h's kept positions, in
 * ascending order followed by the window, are written to idx + h * N;
 * counts[h] receives their number.  Returns 0, or -1 on bad arguments. */
int bo_select_adaptive(const double* S, int H, int N, int W, int budget, double alpha,
                       const bo_params* p, int32_t* idx, int32_t* counts);

/* Compacted cache: out[j] = x[idx[j]] row-wise, d values per row, bitwise. */
void bo_gather(const uint16_t* x, int N, int d, const int32_t* idx,
               int count, uint16_t* out);

#ifdef __cplusplus
}
#endif
#endif
