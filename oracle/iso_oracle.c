/*
 * iso_oracle.c -- CPU oracle for the ISO delta-merge hot path.
 *
 * TEST INFRASTRUCTURE ONLY: a plain, slow, single-threaded restatement of the
 * paper's definitions, used to check the CUDA library.  Only tests/,
 * __graft_entry__.smoke() and bench.py's CPU-baseline leg may call it.  It
 * shares no code with the CUDA library.  Compile with -ffp-contract=off so that
 * every float operation below is one IEEE operation.
 *
 * Precision.  Values are computed in binary64.  The decisions that the GPU
 * takes in binary32 -- the magnitude key that TopKMask ranks, the sign of the
 * TIES election sum, and RAM's activity test |tau| > eps_act -- are taken here
 * in binary32 in the same order, so
 * that both sides decide identically.
 *
 * Parity status: every function here is pinned by tests (hand-worked cases,
 * brute force against a library sort / solve, closed forms and invariants).
 */
#include "iso_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* IEEE encodings                                                            */
/* ------------------------------------------------------------------------ */

static uint32_t f32_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }
static float bits_f32(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

/* bfloat16 is the upper half of a binary32: widening is exact. */
float orc_bf16_to_f32(uint16_t b) { return bits_f32((uint32_t)b << 16); }

/* Round a binary32 to bfloat16, nearest with ties to even (IEEE 754
 * roundTiesToEven).  The integer form is the standard rounding-bias method
 * for truncating formats (as in TensorFlow's float-to-bfloat16 rounding):
 * add half an ulp of the result minus one, plus the kept least-significant
 * bit, so an exact half rounds up only when that bit is odd; then truncate. */
uint16_t orc_f32_to_bf16(float f) {
    uint32_t u = f32_bits(f);
    if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x0040u); /* quiet NaN */
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

void orc_f32_to_bf16_array(const float* x, int64_t n, uint16_t* out) {
    for (int64_t p = 0; p < n; ++p) out[p] = orc_f32_to_bf16(x[p]);
}

/* round-half-even of a non-negative binary64 that is an exact multiple of 1/2
 * or finer: y = floor + frac, frac compared with 1/2 exactly. */
static double round_half_even(double y) {
    double fl = floor(y);
    double fr = y - fl; /* exact: y and fl share the exponent range */
    if (fr > 0.5) return fl + 1.0;
    if (fr < 0.5) return fl;
    return (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
}

/* Round a binary64 to bfloat16 in ONE step (no double rounding through
 * binary32).  bfloat16 has 8 significant bits, exponents down to 2^-126 for
 * normals and a subnormal spacing of 2^-133. */
uint16_t orc_f64_to_bf16(double x) {
    if (isnan(x)) return 0x7FC0u;
    uint16_t sign = signbit(x) ? 0x8000u : 0u;
    double a = fabs(x);
    if (a == 0.0) return sign;
    if (isinf(a)) return (uint16_t)(sign | 0x7F80u);
    int e;
    (void)frexp(a, &e);                    /* a = m 2^e, m in [1/2, 1) */
    int q_exp = e - 8;                     /* spacing of 8-bit significands */
    if (q_exp < -133) q_exp = -133;        /* subnormal spacing */
    double q = round_half_even(ldexp(a, -q_exp));
    double r = ldexp(q, q_exp);            /* exact */
    /* largest finite bfloat16 is (2 - 2^-7) 2^127 */
    if (r > ldexp(255.0, 120)) return (uint16_t)(sign | 0x7F80u);
    float rf = (float)r;                   /* exact: r is a bfloat16 value */
    return (uint16_t)(sign | (f32_bits(rf) >> 16));
}

void orc_f64_to_bf16_array(const double* x, int64_t n, uint16_t* out) {
    for (int64_t p = 0; p < n; ++p) out[p] = orc_f64_to_bf16(x[p]);
}

/* ------------------------------------------------------------------------ */
/* Task vectors (App. F: tau_i = theta_i - theta_0)                          */
/* ------------------------------------------------------------------------ */

static float load_f32(const void* x, int32_t dtype, int64_t p) {
    if (dtype == ORC_BF16) return orc_bf16_to_f32(((const uint16_t*)x)[p]);
    return ((const float*)x)[p];
}

void orc_load(const void* x, int32_t dtype, int64_t n, float* v32, double* v64) {
    for (int64_t p = 0; p < n; ++p) {
        float v = load_f32(x, dtype, p);
        if (v32) v32[p] = v;
        if (v64) v64[p] = (double)v;
    }
}

void orc_delta(const void* theta_i, int32_t dtype_i, const void* theta_0, int32_t dtype_0,
               int64_t n, float* tau32, double* tau64) {
    for (int64_t p = 0; p < n; ++p) {
        float a = load_f32(theta_i, dtype_i, p);
        float b = load_f32(theta_0, dtype_0, p);
        if (tau32) tau32[p] = a - b;                   /* one binary32 subtraction */
        if (tau64) tau64[p] = (double)a - (double)b;   /* binary64 */
    }
}

/* ------------------------------------------------------------------------ */
/* TopKMask (App. F, TIES trim): m = 1 on the largest rho-fraction of |tau|   */
/* ------------------------------------------------------------------------ */

/* The magnitude key: the binary32 pattern of |tau| with the sign cleared.
 * For non-negative finite floats the pattern order is the value order, and
 * -0 and +0 share key 0. */
static uint32_t mag_key(float t) { return f32_bits(t) & 0x7FFFFFFFu; }

int64_t orc_topk_k(double rho, int64_t n) {
    double kk = floor(rho * (double)n + 0.5);
    if (kk < 0.0) kk = 0.0;
    if (kk > (double)n) kk = (double)n;
    return (int64_t)kk;
}

static void fill_stats(orc_unit_stats* st, uint32_t t, int64_t k, int64_t above,
                       int64_t ties, int64_t taken) {
    if (!st) return;
    st->thresh_key = t;
    st->pad = 0;
    st->k = k;
    st->count_above = above;
    st->ties_at_thresh = ties;
    st->ties_taken = taken;
}

typedef struct { uint32_t key; int64_t pos; } key_pos;

static int cmp_key_desc_pos_asc(const void* a, const void* b) {
    const key_pos* x = (const key_pos*)a;
    const key_pos* y = (const key_pos*)b;
    if (x->key != y->key) return (x->key > y->key) ? -1 : 1;
    if (x->pos != y->pos) return (x->pos < y->pos) ? -1 : 1;
    return 0;
}

/* Method 1: order all entries by (|tau| descending, position ascending) and
 * keep the first k. */
void orc_topk_sort(const float* tau32, int64_t n, int64_t k, uint8_t* mask, orc_unit_stats* st) {
    memset(mask, 0, (size_t)n);
    if (k <= 0 || n <= 0) { fill_stats(st, 0xFFFFFFFFu, 0, 0, 0, 0); return; }
    key_pos* a = (key_pos*)malloc((size_t)n * sizeof(key_pos));
    for (int64_t p = 0; p < n; ++p) { a[p].key = mag_key(tau32[p]); a[p].pos = p; }
    qsort(a, (size_t)n, sizeof(key_pos), cmp_key_desc_pos_asc);
    for (int64_t r = 0; r < k; ++r) mask[a[r].pos] = 1;
    uint32_t t = a[k - 1].key;
    int64_t above = 0, ties = 0, taken = 0;
    for (int64_t r = 0; r < n; ++r) {
        if (a[r].key > t) above++;
        else if (a[r].key == t) { ties++; if (r < k) taken++; }
    }
    fill_stats(st, t, k, above, ties, taken);
    free(a);
}

/* k-th largest key (1-based k) by quickselect with a three-way partition, so
 * that long runs of equal keys cost linear time. */
static uint32_t kth_largest(uint32_t* a, int64_t n, int64_t k) {
    int64_t lo = 0, hi = n; /* search a[lo, hi) */
    for (;;) {
        uint32_t x = a[lo], y = a[lo + (hi - lo) / 2], z = a[hi - 1];
        uint32_t piv = (x < y) ? ((y < z) ? y : ((x < z) ? z : x))
                               : ((x < z) ? x : ((y < z) ? z : y)); /* median of 3 */
        /* partition a[lo,hi) into [> piv][== piv][< piv] */
        int64_t gt = lo, i = lo, lt = hi;
        while (i < lt) {
            if (a[i] > piv) { uint32_t s = a[gt]; a[gt] = a[i]; a[i] = s; gt++; i++; }
            else if (a[i] < piv) { lt--; uint32_t s = a[lt]; a[lt] = a[i]; a[i] = s; }
            else i++;
        }
        int64_t n_gt = gt - lo, n_eq = lt - gt;
        if (k <= n_gt) hi = gt;
        else if (k <= n_gt + n_eq) return piv;
        else { k -= n_gt + n_eq; lo = lt; }
    }
}

/* Method 2: t = k-th largest key; keep every key above t and the first
 * k - #(key > t) entries with key == t in position order. */
void orc_topk_select(const float* tau32, int64_t n, int64_t k, uint8_t* mask, orc_unit_stats* st) {
    memset(mask, 0, (size_t)n);
    if (k <= 0 || n <= 0) { fill_stats(st, 0xFFFFFFFFu, 0, 0, 0, 0); return; }
    uint32_t* keys = (uint32_t*)malloc((size_t)n * sizeof(uint32_t));
    for (int64_t p = 0; p < n; ++p) keys[p] = mag_key(tau32[p]);
    uint32_t t = kth_largest(keys, n, k);
    int64_t above = 0, ties = 0;
    for (int64_t p = 0; p < n; ++p) {
        uint32_t kp = mag_key(tau32[p]);
        if (kp > t) above++;
        else if (kp == t) ties++;
    }
    int64_t need = k - above, taken = 0;
    for (int64_t p = 0; p < n; ++p) {
        uint32_t kp = mag_key(tau32[p]);
        if (kp > t) mask[p] = 1;
        else if (kp == t && taken < need) { mask[p] = 1; taken++; }
    }
    fill_stats(st, t, k, above, ties, taken);
    free(keys);
}

/* ------------------------------------------------------------------------ */
/* Retention coefficients (Sec. 4.2 retention system; App. E; Algorithm 1)   */
/* ------------------------------------------------------------------------ */

/* Solve A x = b (m x m, row-major, overwritten) by Gaussian elimination with
 * partial pivoting. */
static void gauss_solve(int m, double* A, double* b, double* x) {
    for (int c = 0; c < m; ++c) {
        int piv = c;
        for (int r = c + 1; r < m; ++r)
            if (fabs(A[r * m + c]) > fabs(A[piv * m + c])) piv = r;
        if (piv != c) {
            for (int j = 0; j < m; ++j) { double s = A[c * m + j]; A[c * m + j] = A[piv * m + j]; A[piv * m + j] = s; }
            double s = b[c]; b[c] = b[piv]; b[piv] = s;
        }
        for (int r = c + 1; r < m; ++r) {
            double f = A[r * m + c] / A[c * m + c];
            for (int j = c; j < m; ++j) A[r * m + j] -= f * A[c * m + j];
            b[r] -= f * b[c];
        }
    }
    for (int r = m - 1; r >= 0; --r) {
        double s = b[r];
        for (int j = r + 1; j < m; ++j) s -= A[r * m + j] * x[j];
        x[r] = s / A[r * m + r];
    }
}

void orc_retention(int32_t K, const double* gram, double ridge, double c_min, double c_max,
                   double* coef) {
    /* I = { i : ||g_i||^2 > 0 }; experts outside I get coefficient 0 */
    int idx[64];
    int m = 0;
    for (int i = 0; i < K; ++i) {
        coef[i] = 0.0;
        if (gram[i * K + i] > 0.0) idx[m++] = i;
    }
    if (m == 0) return;
    double* A = (double*)malloc((size_t)m * m * sizeof(double));
    double* b = (double*)malloc((size_t)m * sizeof(double));
    double* x = (double*)malloc((size_t)m * sizeof(double));
    for (int r = 0; r < m; ++r) {
        for (int c = 0; c < m; ++c) A[r * m + c] = gram[idx[r] * K + idx[c]];
        A[r * m + r] += ridge;              /* (Gamma + lambda_ridge I) */
        b[r] = gram[idx[r] * K + idx[r]];   /* b = diag(Gamma): unit self-retention */
    }
    gauss_solve(m, A, b, x);
    for (int r = 0; r < m; ++r) {
        double c = x[r];
        if (c < c_min) c = c_min;           /* clip(c_bar; c_min, c_max) */
        if (c > c_max) c = c_max;
        coef[idx[r]] = c;
    }
    free(A); free(b); free(x);
}

/* ------------------------------------------------------------------------ */
/* Merge operators                                                           */
/* ------------------------------------------------------------------------ */

static int sign_f(float v) { return (v > 0.0f) - (v < 0.0f); }

/* mask == NULL: the tensor is not trimmed, every entry is kept */
static int kept(const uint8_t* const* mask, int i, int64_t p) { return mask ? mask[i][p] : 1; }

/* theta = theta_0 + update; an update of exactly zero leaves theta_0 as is
 * (this keeps the sign of a -0 base weight). */
static double add_update(double theta0, double upd) { return (upd == 0.0) ? theta0 : theta0 + upd; }

void orc_merge_tensor(int32_t op, int32_t K, int64_t n, int32_t is_1d,
                      const double* theta0,
                      const float* const* tau32, const double* const* tau64,
                      const uint8_t* const* mask,
                      double lambda, double ridge, double c_min, double c_max,
                      double* out, double* gram, double* coef) {
    if (op == ORC_TA) {
        /* Task Arithmetic (App. F): tau_TA = lambda sum_i tau_i */
        for (int64_t p = 0; p < n; ++p) {
            double s = 0.0;
            for (int i = 0; i < K; ++i) s += tau64[i][p];
            out[p] = add_update(theta0[p], lambda * s);
        }
        return;
    }
    if (op == ORC_TIES) {
        /* TIES (App. F): trim, elect sign, disjoint mean */
        for (int64_t p = 0; p < n; ++p) {
            float s32 = 0.0f;                     /* election sum in binary32, i = 1..K */
            for (int i = 0; i < K; ++i) {
                float tt = kept(mask, i, p) ? tau32[i][p] : 0.0f;
                s32 = s32 + tt;
            }
            int gamma = sign_f(s32);
            double acc = 0.0;
            int cnt = 0;
            for (int i = 0; i < K; ++i) {
                if (!kept(mask, i, p)) continue;
                float tt = tau32[i][p];
                if (tt != 0.0f && sign_f(tt) == gamma) { acc += tau64[i][p]; cnt++; }
            }
            double merged = cnt ? acc / (double)cnt : 0.0;
            out[p] = add_update(theta0[p], lambda * merged);
        }
        return;
    }
    /* ISO */
    if (is_1d) {
        /* 1-D parameters: task-vector average (App. E, Algorithm 1) */
        for (int64_t p = 0; p < n; ++p) {
            double s = 0.0;
            for (int i = 0; i < K; ++i) s += tau64[i][p];
            out[p] = add_update(theta0[p], s / (double)K);
        }
        return;
    }
    /* 2-D: g_i = trimmed task vector; Gamma_ij = <g_i, g_j>; retention solve */
    double G[64 * 64];
    double c[64];
    for (int i = 0; i < K; ++i)
        for (int j = 0; j < K; ++j) G[i * K + j] = 0.0;
    for (int i = 0; i < K; ++i) {
        for (int j = i; j < K; ++j) {
            double s = 0.0;
            for (int64_t p = 0; p < n; ++p) {
                double gi = kept(mask, i, p) ? tau64[i][p] : 0.0;
                double gj = kept(mask, j, p) ? tau64[j][p] : 0.0;
                s += gi * gj;
            }
            G[i * K + j] = s;
            G[j * K + i] = s;
        }
    }
    orc_retention(K, G, ridge, c_min, c_max, c);
    if (gram) for (int q = 0; q < K * K; ++q) gram[q] = G[q];
    if (coef) for (int i = 0; i < K; ++i) coef[i] = c[i];
    for (int64_t p = 0; p < n; ++p) {
        double s = 0.0;
        for (int i = 0; i < K; ++i)
            if (kept(mask, i, p)) s += c[i] * tau64[i][p];
        out[p] = add_update(theta0[p], s);
    }
}

/* ------------------------------------------------------------------------ */
/* RAM (App. F): inactive coordinates are dropped, a coordinate that one
 * expert updates keeps that expert's value, a coordinate that several update
 * takes the mean over those experts only. */

void orc_merge_ram(int32_t K, int64_t n, const double* theta0,
                   const float* const* tau32, const double* const* tau64,
                   double eps_act, double lambda, double* out) {
    for (int64_t p = 0; p < n; ++p) {
        /* A_p and c^p */
        int active[64];
        int c = 0;
        for (int i = 0; i < K; ++i) {
            if (fabs((double)tau32[i][p]) > eps_act) active[c++] = i;
        }
        double tau_ram;
        if (c == 0) {
            tau_ram = 0.0;
        } else if (c == 1) {
            tau_ram = tau64[active[0]][p];
        } else {
            double s = 0.0;
            for (int a = 0; a < c; ++a) s += tau64[active[a]][p];
            tau_ram = s / (double)c;
        }
        out[p] = add_update(theta0[p], lambda * tau_ram);
    }
}
