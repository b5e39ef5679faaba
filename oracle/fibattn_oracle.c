/*
 * fibattn_oracle.c -- plain, slow, fp64 CPU oracle for depth-staggered
 * scaled-Fibonacci sparse attention (arXiv 2606.28560, Section 2 "Method").
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent definition that the
 * CUDA path is checked against.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load it.  It shares no code, header,
 * table or constant with the CUDA library and includes none of its files.
 *
 * What it computes (per batch b, head h, query position i):
 *   - Attended set (Section 2, "Attended set"): the dense causal window at
 *     distances t = 0..W (self always present), plus K rungs at continuous
 *     distances d_k = alpha * f_k.
 *   - Each rung is read by linear interpolation between the floor and
 *     floor-plus-one positions: with s0 = floor(d_k) and w = d_k - s0 the rung
 *     key is (1-w) * k~[i-s0] + w * k~[i-s0-1], and likewise for the value
 *     (Section 2, "Attended set").
 *   - RoPE is applied at true positions BEFORE the gather: q~_i = R(i) q_i,
 *     k~_j = R(j) k_j (Section 2, "Attended set"; RoPE base 1e4 from Section 3
 *     "Model and training").  Values are not rotated.
 *   - Softmax over the attended slots with scale 1/sqrt(D) (the paper does
 *     not write the softmax out; standard scaled dot-product attention is the
 *     reading taken), then the probability-weighted sum of the value slots.
 *   - alpha = 0.5 + sigmoid(theta) (Section 2, "The per-layer scalar"), so
 *     dtheta = dalpha * (alpha - 0.5) * (1.5 - alpha).
 *
 * Readings where the paper is silent (each is listed in the design notes):
 *   - dedup: a rung with d_k <= W duplicates window distances; with dedup=1
 *     it is dropped so the attended set is the set union of Section 2.
 *   - a rung with d_k > i reaches before position 0 and is masked.  At
 *     d_k == i (integer) the floor row is row 0 and the weight-0 far row -1
 *     is taken as a zero row.
 *   - floor is taken of the distance: the far row i-s0-1 carries weight w.
 *     At an integer d_k the derivative dkey/dd_k = k~[i-s0-1] - k~[i-s0]
 *     (one-sided, from above).
 *   - d_k is rounded once to fp32 by the caller-side prep (fibo_offsets_fp32);
 *     the core routines take the distances as given, in fp64.
 *   - RoPE pairs dimension m with m + D/2 ("rotate-half"), frequency
 *     base^(-2m/D), positions 0..T-1.
 *   - GQA: head h reads key/value head h / (H / Hkv).
 *
 * Layouts: q, out, dout, dq are [B][H][T][D]; k, v, dk, dv are [B][Hkv][T][D];
 * lse is [B][H][T]; all row-major, fp64.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* One attended slot of one query: up to two rows j0, j1 with weights c0, c1
 * (window slot: j1 = -1, c1 = 0); rung index (or -1 for a window slot). */
typedef struct { int j0, j1; double c0, c1; int rung; } slot_t;

/* ---- offset prep (Section 2: d_k = alpha * f_k, rounded once to fp32) ---- */
void fibo_offsets_fp32(double alpha, const double* f, int K, double* d_out)
{
    for (int k = 0; k < K; ++k) {
        float a = (float)alpha, fk = (float)f[k];
        /* the product of two fp32 values is exact in fp64; one rounding to
         * fp32 then equals an fp32 multiply */
        d_out[k] = (double)(float)((double)a * (double)fk);
    }
}

/* ---- RoPE at a true position (rotate-half pairing) ---- */
static void rope_rotate(const double* x, double* y, int D, int pos, double base, int inverse)
{
    int half = D / 2;
    for (int m = 0; m < half; ++m) {
        double freq = pow(base, -2.0 * (double)m / (double)D);
        double ang = (double)pos * freq;
        double c = cos(ang), s = sin(ang);
        double a = x[m], b = x[m + half];
        if (!inverse) {            /* y = R(pos) x */
            y[m] = a * c - b * s;
            y[m + half] = b * c + a * s;
        } else {                   /* y = R(pos)^T x */
            y[m] = a * c + b * s;
            y[m + half] = b * c - a * s;
        }
    }
}

/* ---- attended set of query i (Section 2, "Attended set") ---- */
static int build_slots(int i, int W, const double* d, int K, int dedup, slot_t* sl)
{
    int n = 0;
    for (int t = 0; t <= W; ++t) {              /* dense causal window */
        int j = i - t;
        if (j < 0) break;
        sl[n].j0 = j; sl[n].j1 = -1; sl[n].c0 = 1.0; sl[n].c1 = 0.0; sl[n].rung = -1; ++n;
    }
    for (int k = 0; k < K; ++k) {               /* scaled rungs */
        if (dedup && !(d[k] > (double)W)) continue;    /* inside the window */
        if (d[k] > (double)i) continue;                /* before position 0 */
        double s0 = floor(d[k]);
        double w = d[k] - s0;
        int j0 = i - (int)s0;
        sl[n].j0 = j0; sl[n].j1 = j0 - 1;       /* j1 may be -1 (then w == 0) */
        sl[n].c0 = 1.0 - w; sl[n].c1 = w; sl[n].rung = k; ++n;
    }
    return n;
}

/* interpolated row of a slot: out = c0 * X[j0] + c1 * X[j1] (row -1 is zero) */
static void slot_row(const slot_t* s, const double* X, int D, double* out)
{
    for (int e = 0; e < D; ++e) {
        double v = s->c0 * X[(size_t)s->j0 * D + e];
        if (s->j1 >= 0) v += s->c1 * X[(size_t)s->j1 * D + e];
        out[e] = v;
    }
}

/* difference row X[j1] - X[j0] (row -1 is zero): d(slot row)/d(d_k) */
static void slot_diff(const slot_t* s, const double* X, int D, double* out)
{
    for (int e = 0; e < D; ++e) {
        double far = s->j1 >= 0 ? X[(size_t)s->j1 * D + e] : 0.0;
        out[e] = far - X[(size_t)s->j0 * D + e];
    }
}

static double dot(const double* a, const double* b, int D)
{
    double s = 0.0;
    for (int e = 0; e < D; ++e) s += a[e] * b[e];
    return s;
}

/* Forward of one (b, h): rotated keys kt [T][D] precomputed by the caller. */
static void fwd_head(const double* Q, const double* KT, const double* V, double* O, double* LSE,
                     int T, int D, int W, const double* d, int K, double scale,
                     double base, int dedup, slot_t* sl, double* wk)
{
    double* qt = wk; double* key = wk + D; double* val = wk + 2 * D; double* sc = wk + 3 * D;
    for (int i = 0; i < T; ++i) {
        rope_rotate(Q + (size_t)i * D, qt, D, i, base, 0);
        int n = build_slots(i, W, d, K, dedup, sl);
        double mx = -INFINITY;
        for (int s = 0; s < n; ++s) {
            slot_row(&sl[s], KT, D, key);
            sc[s] = scale * dot(qt, key, D);
            if (sc[s] > mx) mx = sc[s];
        }
        double l = 0.0;
        for (int s = 0; s < n; ++s) l += exp(sc[s] - mx);
        double* o = O + (size_t)i * D;
        for (int e = 0; e < D; ++e) o[e] = 0.0;
        for (int s = 0; s < n; ++s) {
            double p = exp(sc[s] - mx) / l;
            slot_row(&sl[s], V, D, val);
            for (int e = 0; e < D; ++e) o[e] += p * val[e];
        }
        if (LSE) LSE[i] = mx + log(l);
    }
}

static void rotate_rows(const double* X, double* XT, int T, int D, double base, int inverse)
{
    for (int j = 0; j < T; ++j) rope_rotate(X + (size_t)j * D, XT + (size_t)j * D, D, j, base, inverse);
}

/* Forward pass.  Returns 0 on success, nonzero on bad arguments. */
int fibo_forward(const double* q, const double* k, const double* v, double* out, double* lse,
                 int B, int H, int Hkv, int T, int D, int W,
                 const double* d, int K, double scale, double rope_base, int dedup, int nthreads)
{
    if (B < 0 || H <= 0 || Hkv <= 0 || H % Hkv || T < 0 || D <= 0 || D % 2 || W < 0 || K < 0) return 1;
    int G = H / Hkv;
    int npairs = B * H;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int p = 0; p < npairs; ++p) {
        int b = p / H, h = p % H, hk = h / G;
        const double* Q = q + ((size_t)b * H + h) * T * D;
        const double* Kp = k + ((size_t)b * Hkv + hk) * T * D;
        const double* Vp = v + ((size_t)b * Hkv + hk) * T * D;
        double* KT = (double*)malloc(sizeof(double) * (size_t)T * D + 1);
        slot_t* sl = (slot_t*)malloc(sizeof(slot_t) * (size_t)(W + 1 + K) + 1);
        double* wk = (double*)malloc(sizeof(double) * (size_t)(3 * D + W + 1 + K) + 1);
        rotate_rows(Kp, KT, T, D, rope_base, 0);
        fwd_head(Q, KT, Vp, out + ((size_t)b * H + h) * T * D, lse ? lse + ((size_t)b * H + h) * T : NULL,
                 T, D, W, d, K, scale, rope_base, dedup, sl, wk);
        free(KT); free(sl); free(wk);
    }
    (void)nthreads;
    return 0;
}

/* Backward pass: the chain rule of the forward definition, in fp64.
 * Recomputes the forward internally from q, k, v.  Writes dq, dk, dv
 * (w.r.t. the pre-RoPE inputs), dd[K] = dL/dd_k.  dk and dv are overwritten. */
int fibo_backward(const double* q, const double* k, const double* v, const double* dout,
                  double* dq, double* dk, double* dv, double* dd,
                  int B, int H, int Hkv, int T, int D, int W,
                  const double* d, int K, double scale, double rope_base, int dedup, int nthreads)
{
    if (B < 0 || H <= 0 || Hkv <= 0 || H % Hkv || T < 0 || D <= 0 || D % 2 || W < 0 || K < 0) return 1;
    int G = H / Hkv;
    int nkv = B * Hkv;
    memset(dk, 0, sizeof(double) * (size_t)B * Hkv * T * D);
    memset(dv, 0, sizeof(double) * (size_t)B * Hkv * T * D);
    double* ddp = (double*)calloc((size_t)nkv * (K > 0 ? K : 1), sizeof(double));
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int p = 0; p < nkv; ++p) {             /* one kv head and its G query heads */
        int b = p / Hkv, hk = p % Hkv;
        const double* Kp = k + ((size_t)b * Hkv + hk) * T * D;
        const double* Vp = v + ((size_t)b * Hkv + hk) * T * D;
        double* dKp = dk + ((size_t)b * Hkv + hk) * T * D;
        double* dVp = dv + ((size_t)b * Hkv + hk) * T * D;
        size_t TD = (size_t)T * D;
        double* KT = (double*)malloc(sizeof(double) * TD + 1);
        double* dKT = (double*)calloc(TD + 1, sizeof(double));   /* grad w.r.t. rotated keys */
        int S = W + 1 + K;
        slot_t* sl = (slot_t*)malloc(sizeof(slot_t) * (size_t)S + 1);
        double* qt = (double*)malloc(sizeof(double) * (size_t)D * 5 + 1);
        double* key = qt + D; double* val = qt + 2 * D; double* dqt = qt + 3 * D; double* diff = qt + 4 * D;
        double* sc = (double*)malloc(sizeof(double) * (size_t)S * 3 + 1);
        double* pr = sc + S; double* dp = sc + 2 * S;
        rotate_rows(Kp, KT, T, D, rope_base, 0);
        for (int g = 0; g < G; ++g) {
            int h = hk * G + g;
            const double* Q = q + ((size_t)b * H + h) * TD;
            const double* dO = dout + ((size_t)b * H + h) * TD;
            double* dQ = dq + ((size_t)b * H + h) * TD;
            for (int i = 0; i < T; ++i) {
                const double* go = dO + (size_t)i * D;
                rope_rotate(Q + (size_t)i * D, qt, D, i, rope_base, 0);
                int n = build_slots(i, W, d, K, dedup, sl);
                /* forward recompute: scores and probabilities */
                double mx = -INFINITY;
                for (int s = 0; s < n; ++s) {
                    slot_row(&sl[s], KT, D, key);
                    sc[s] = scale * dot(qt, key, D);
                    if (sc[s] > mx) mx = sc[s];
                }
                double l = 0.0;
                for (int s = 0; s < n; ++s) l += exp(sc[s] - mx);
                for (int s = 0; s < n; ++s) pr[s] = exp(sc[s] - mx) / l;
                /* dL/dp_s = dO_i . val_s ; Delta = sum_s p_s dp_s (= dO_i . o_i) */
                double delta = 0.0;
                for (int s = 0; s < n; ++s) {
                    slot_row(&sl[s], Vp, D, val);
                    dp[s] = dot(go, val, D);
                    delta += pr[s] * dp[s];
                }
                for (int e = 0; e < D; ++e) dqt[e] = 0.0;
                for (int s = 0; s < n; ++s) {
                    double ds = pr[s] * (dp[s] - delta);     /* dL/dscore_s */
                    slot_row(&sl[s], KT, D, key);
                    for (int e = 0; e < D; ++e) dqt[e] += scale * ds * key[e];
                    /* key side: dL/dkey_s = scale * ds * q~_i, split onto rows */
                    for (int e = 0; e < D; ++e) {
                        double gk = scale * ds * qt[e];
                        dKT[(size_t)sl[s].j0 * D + e] += sl[s].c0 * gk;
                        if (sl[s].j1 >= 0) dKT[(size_t)sl[s].j1 * D + e] += sl[s].c1 * gk;
                    }
                    /* value side: dL/dval_s = p_s * dO_i */
                    for (int e = 0; e < D; ++e) {
                        double gv = pr[s] * go[e];
                        dVp[(size_t)sl[s].j0 * D + e] += sl[s].c0 * gv;
                        if (sl[s].j1 >= 0) dVp[(size_t)sl[s].j1 * D + e] += sl[s].c1 * gv;
                    }
                    /* rung distance: dkey/dd_k = k~[j1] - k~[j0], dval/dd_k = v[j1] - v[j0] */
                    if (sl[s].rung >= 0) {
                        double acc = 0.0;
                        slot_diff(&sl[s], KT, D, diff);
                        acc += scale * ds * dot(qt, diff, D);
                        slot_diff(&sl[s], Vp, D, diff);
                        acc += pr[s] * dot(go, diff, D);
                        ddp[(size_t)p * K + sl[s].rung] += acc;
                    }
                }
                rope_rotate(dqt, dQ + (size_t)i * D, D, i, rope_base, 1);
            }
        }
        /* back through the key rotation: dk_j = R(j)^T dk~_j */
        rotate_rows(dKT, dKp, T, D, rope_base, 1);
        free(KT); free(dKT); free(sl); free(qt); free(sc);
    }
    for (int kk = 0; kk < K; ++kk) {            /* fixed-order sum over kv heads */
        double s = 0.0;
        for (int p = 0; p < nkv; ++p) s += ddp[(size_t)p * K + kk];
        dd[kk] = s;
    }
    free(ddp);
    (void)nthreads;
    return 0;
}

/* Chain rule to the per-layer scalar: d_k = alpha f_k, alpha = 0.5 + sigmoid(theta). */
void fibo_dtheta(double alpha, const double* f, const double* dd, int K, double* dalpha, double* dtheta)
{
    double da = 0.0;
    for (int k = 0; k < K; ++k) da += f[k] * dd[k];
    *dalpha = da;
    *dtheta = da * (alpha - 0.5) * (1.5 - alpha);
}

/* Debug view of one query: attended slots, their rows/weights and softmax
 * probabilities.  Returns the slot count (<= W+1+K).  rows0/rows1/c0/c1/prob/
 * rung are arrays of W+1+K entries. */
int fibo_query_slots(const double* q, const double* k, int T, int D, int W, int i,
                     const double* d, int K, double scale, double rope_base, int dedup,
                     int* rows0, int* rows1, double* c0, double* c1, double* prob, int* rung)
{
    if (i < 0 || i >= T) return -1;
    int S = W + 1 + K;
    slot_t* sl = (slot_t*)malloc(sizeof(slot_t) * (size_t)S + 1);
    double* KT = (double*)malloc(sizeof(double) * (size_t)T * D + 1);
    double* qt = (double*)malloc(sizeof(double) * (size_t)D * 2 + 1);
    double* key = qt + D;
    double* sc = (double*)malloc(sizeof(double) * (size_t)S + 1);
    rotate_rows(k, KT, T, D, rope_base, 0);
    rope_rotate(q + (size_t)i * D, qt, D, i, rope_base, 0);
    int n = build_slots(i, W, d, K, dedup, sl);
    double mx = -INFINITY;
    for (int s = 0; s < n; ++s) {
        slot_row(&sl[s], KT, D, key);
        sc[s] = scale * dot(qt, key, D);
        if (sc[s] > mx) mx = sc[s];
    }
    double l = 0.0;
    for (int s = 0; s < n; ++s) l += exp(sc[s] - mx);
    for (int s = 0; s < n; ++s) {
        rows0[s] = sl[s].j0; rows1[s] = sl[s].j1; c0[s] = sl[s].c0; c1[s] = sl[s].c1;
        prob[s] = exp(sc[s] - mx) / l; rung[s] = sl[s].rung;
    }
    free(sl); free(KT); free(qt); free(sc);
    return n;
}
