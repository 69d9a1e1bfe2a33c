/*
 * iso_oracle.h -- CPU oracle for the ISO delta-merge hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, single-threaded C
 * restatement of the definitions in "ISO: An RLVR-Native Optimization Stack"
 * (App. F: task vectors, TopKMask, Task Arithmetic, TIES, RAM; Sec. 4.2, App. E
 * and Algorithm 1: the retention combiner and the 1-D average).  Only tests/,
 * __graft_entry__.smoke() and bench.py's CPU-baseline leg may call it.  It
 * shares no code, header, table or helper with the CUDA library.
 *
 * Element encodings: ORC_BF16 = IEEE bfloat16 stored as uint16_t,
 * ORC_F32 = IEEE binary32.
 */
#ifndef ISO_ORACLE_H
#define ISO_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_BF16 = 0, ORC_F32 = 1 };
enum { ORC_TA = 0, ORC_TIES = 1, ORC_ISO = 2, ORC_RAM = 3 };

/* per selection unit, as defined by the oracle's TopKMask */
typedef struct {
    uint32_t thresh_key;     /* key of the k-th largest |tau|; 0xFFFFFFFF when k == 0 */
    uint32_t pad;
    int64_t  k;              /* number of selected entries */
    int64_t  count_above;    /* entries with key > thresh_key */
    int64_t  ties_at_thresh; /* entries with key == thresh_key */
    int64_t  ties_taken;     /* ties selected, lowest position first */
} orc_unit_stats;

/* conversions */
float    orc_bf16_to_f32(uint16_t b);
uint16_t orc_f32_to_bf16(float f);    /* round to nearest, ties to even */
uint16_t orc_f64_to_bf16(double x);   /* one rounding from binary64, ties to even */
void     orc_f32_to_bf16_array(const float* x, int64_t n, uint16_t* out);
void     orc_f64_to_bf16_array(const double* x, int64_t n, uint16_t* out);

/* k = floor(rho * n + 1/2), clamped to [0, n] */
int64_t orc_topk_k(double rho, int64_t n);

/* load a tensor: value in f32 (decision precision) and f64 (value precision) */
void orc_load(const void* x, int32_t dtype, int64_t n, float* v32, double* v64);

/* tau = theta_i - theta_0: f32 subtraction (decision precision) and exact f64 */
void orc_delta(const void* theta_i, int32_t dtype_i, const void* theta_0, int32_t dtype_0,
               int64_t n, float* tau32, double* tau64);

/* TopKMask over one unit, entries in unit order.  Two independent methods:
 * full sort by (key desc, position asc), and k-th-largest selection plus an
 * in-order scan of the ties.  mask[p] = 1 for the selected entries. */
void orc_topk_sort(const float* tau32, int64_t n, int64_t k, uint8_t* mask, orc_unit_stats* st);
void orc_topk_select(const float* tau32, int64_t n, int64_t k, uint8_t* mask, orc_unit_stats* st);

/* merge one tensor of n entries from K task vectors.
 *   op      ORC_TA / ORC_TIES / ORC_ISO
 *   tau32   K arrays, decision precision (signs, TIES election)
 *   tau64   K arrays, value precision
 *   mask    K arrays (TIES, ISO 2-D); NULL = not trimmed (TA, ISO 1-D, and TIES
 *           tensors left untrimmed)
 *   is_1d   ISO only: 1-D parameters take the plain task-vector average
 *   out     merged values in f64
 *   gram    K*K (ISO 2-D, may be NULL), coef K (ISO 2-D, may be NULL) */
void orc_merge_tensor(int32_t op, int32_t K, int64_t n, int32_t is_1d,
                      const double* theta0,
                      const float* const* tau32, const double* const* tau64,
                      const uint8_t* const* mask,
                      double lambda, double ridge, double c_min, double c_max,
                      double* out, double* gram, double* coef);

/* RAM merge of one tensor (App. F, the RAM coordinate rule): per entry p the
 * active set A_p = { i : |tau_i^p| > eps_act } and c^p = |A_p|; the merged
 * coordinate is 0 for c^p = 0, tau_j^p for A_p = {j}, and the mean of the
 * active values for c^p >= 2; out = theta_0 + lambda tau_RAM (the paper's
 * RAM has no scale: lambda = 1 is the paper's rule).  Activity is decided on
 * tau32 (decision precision); the values come from tau64.  No trim. */
void orc_merge_ram(int32_t K, int64_t n, const double* theta0,
                   const float* const* tau32, const double* const* tau64,
                   double eps_act, double lambda, double* out);

/* retention coefficients from a K x K Gram matrix (App. E / Algorithm 1):
 * drop zero-norm experts, solve (G + ridge I) c = diag G, clip. */
void orc_retention(int32_t K, const double* gram, double ridge, double c_min, double c_max,
                   double* coef);

#ifdef __cplusplus
}
#endif
#endif
