// iso_frame.cu -- the frame-space ISO-Merger of one weight matrix (App. E)
// on one GPU.
//
// Given the thin SVDs W_0 = U_0 S_0 V_0^T (base) and W_i = U_i S_i V_i^T
// (experts, i = 1..K; their spectra are not used), the merge is
//   s_ik   = sign(<u_0k, u_ik>), sign(0) := 1                  (Sign canonicalization)
//   xi_Fi  = Pi_{F_0}(s_i F_i - F_0) D_keep,  F in {U, V}       (Stiefel tangent projection,
//            Pi_{F_0}(X) = X - F_0 sym(F_0^T X)                  Top-k_keep masking)
//   g_i    = xi_Ui S_0 V_0^T + U_0 S_0 xi_Vi^T, Gamma_ij = <g_i, g_j>_F
//   c*     = clip((Gamma + ridge I)^-1 diag Gamma)              (Retention coefficients)
//   xi_F*  = Pi_{F_0}(sum_i c*_i xi_Fi),  F* = polar(F_0 + xi_F*) (Retraction and
//   W*     = U* S_0 V*^T                                          reconstruction)
//
// How it is computed here (every identity below is pinned against the binary64
// oracle of the same definitions):
// * Nothing of size m x n is formed but the output.  With A_i = F_0^T dF_i
//   (dF_i = s_i F_i - F_0), Sym_i = sym(A_i), Kw_i = A_i - Sym_i:
//     F_0^T xi_Fi = Kw_i D,
//     (xi_Fi^T xi_Fj)_kk = D_k [(dF_i^T dF_j)_kk - (A_i^T Sym_j)_kk - (Sym_i A_j)_kk + (Sym_i Sym_j)_kk],
//     Gamma_ij = sum_k s_k^2 [(xi_Ui^T xi_Uj)_kk + (xi_Vi^T xi_Vj)_kk]
//                - sum_kl s_k s_l D_k D_l (KwU_i KwV_j + KwU_j KwV_i)[k, l],
//     xi_F* = D dF_c - F_0 Y,  dF_c = sum_i c*_i dF_i,
//     Y = (sum_i c*_i Sym_i) D + sym((sum_i c*_i Kw_i) D).
// * polar(F_0 + xi) = (F_0 + xi)(I + xi^T xi)^(-1/2), since F_0^T xi is skew;
//   the inverse square root comes from the coupled Newton-Schulz iteration
//   written in differences from the identity (Y = I + y, Z = I + z), so that
//   every product is of small matrices, scaled when ||xi^T xi||_F >= 0.9.
// * W* = W_0 + [E_U S_0 | U_0 S_0] [V* | E_V]^T with E_F = F* - F_0: the
//   difference form keeps the low-precision products on the small motion;
//   W_0 itself (the caller's matrix) replaces U_0 S_0 V_0^T.
// * Precision.  A_i = F_0^T dF_i is binary64 on the CUDA cores: on dense
//   spectra the frames rotate far inside near-degenerate singular subspaces
//   while the proxies stay small, so Gamma is a difference of terms up to
//   thousands of times larger than itself (the paper takes the merge in
//   binary64 throughout).  The other large contractions (F_0 Y, xi*^T xi*,
//   the Newton-Schulz products, (F_0 + xi*) R and the reconstruction) run on
//   the tensor cores (k_gemm_tf32) as three tf32 products per pair (hi hi +
//   hi lo + lo hi, x = hi + lo split in binary64) with binary32 accumulation,
//   about 2^-22 relative per product; what they feed is the merged frame,
//   whose error reaches W* only through products with the small motion.
//   Everything else is binary64 on the CUDA cores.
#include "iso_gemm.cuh"
#include "iso_internal.cuh"

#include <algorithm>
#include <cmath>
#include <vector>

namespace iso {

namespace {

constexpr int FR_PAD = 128;        // operand arrays padded to whole GEMM tiles
constexpr int FR_MAX_NS = 64;      // Newton-Schulz iteration limit
constexpr int FR_DEFAULT_NS = 16;
constexpr double FR_NS_TOL = 1e-9; // max |y + z + z y| at which the iteration has converged

long long pad_up(long long x) { return (x + FR_PAD - 1) / FR_PAD * FR_PAD; }

struct FrameHeader {
    int32_t status;
    int32_t conv[2];                // per side: the Newton-Schulz iteration has converged
    int32_t pad;
    double nu2[2];                  // per side: ||xi^T xi||_F^2
    double cs[2];                   // per side: the scaling of I + xi^T xi
    uint32_t wmax[2][FR_MAX_NS];    // per side and iteration: max |w| as binary32 bits
};

// binary64 -> (hi, lo) with hi a tf32 value (round to nearest, ties away) and
// lo the binary32 rest, so that hi + lo = x to about 2^-22 |x|
__device__ __forceinline__ void split_tf32(double x, float& hi, float& lo) {
    const float x32 = (float)x;
    uint32_t h;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(h) : "f"(x32));
    hi = __uint_as_float(h);
    const float l32 = (float)(x - (double)hi);
    uint32_t l;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(l) : "f"(l32));
    lo = __uint_as_float(l);
}

// An operand row of contraction length L (padded) is stored in four segments
// [hi | lo | hi | hi]: read from segment 0 it is (hi, lo, hi), from segment 1
// (lo, hi, hi); A from 0 and B from 1 pair up as hi lo + lo hi + hi hi.
__device__ __forceinline__ void put_split(float* row, long long L, long long k, double x) {
    float hi, lo;
    split_tf32(x, hi, lo);
    row[k] = hi;
    row[L + k] = lo;
    row[2 * L + k] = hi;
    row[3 * L + k] = hi;
}

struct Frames {                     // one side (U: d = m; V: d = n), d x q row-major binary64
    const double* F0;
    const double* F[MAXK];
    int K;
    long long d, q;
};

// ---------------------------------------------------------------------------
// layout helpers
// ---------------------------------------------------------------------------
// out (C x R) = in (R x C)^T, binary64, 32 x 32 tiles
__global__ void __launch_bounds__(256) k_fr_transpose(const double* in, double* out, long long R, long long C) {
    __shared__ double t[32][33];
    const long long r0 = (long long)blockIdx.y * 32, c0 = (long long)blockIdx.x * 32;
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        t[y][threadIdx.x] = (r < R && c < C) ? in[r * C + c] : 0.0;
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long c = c0 + y, r = r0 + threadIdx.x;
        if (c < C && r < R) out[c * R + r] = t[threadIdx.x][y];
    }
}

// s_ik = sign(<u_0k, u_ik>): the column dot products (U side), summed into dots[i][k]
__global__ void __launch_bounds__(256) k_fr_signdots(Frames f, double* dots, int row_chunks) {
    __shared__ double red[8][33];
    const long long k = (long long)blockIdx.x * 32 + threadIdx.x;
    const int i = blockIdx.y;
    const long long per = (f.d + row_chunks - 1) / row_chunks;
    const long long r0 = (long long)blockIdx.z * per, r1 = min(f.d, r0 + per);
    double acc = 0.0;
    if (k < f.q)
        for (long long r = r0 + threadIdx.y; r < r1; r += 8) acc = fma(f.F0[r * f.q + k], f.F[i][r * f.q + k], acc);
    red[threadIdx.y][threadIdx.x] = acc;
    __syncthreads();
    if (threadIdx.y == 0 && k < f.q) {
        double s = 0.0;
        for (int y = 0; y < 8; ++y) s += red[y][threadIdx.x];
        atomicAdd(&dots[(long long)i * f.q + k], s);
    }
}

__device__ __forceinline__ double sign_of(const double* dots, long long q, int i, long long k) {
    return dots[(long long)i * q + k] < 0.0 ? -1.0 : 1.0;
}

// (dF_i^T dF_j)_kk for i <= j, summed into cd[i][j][k]
__global__ void __launch_bounds__(256) k_fr_coldots(Frames f, const double* dots, double* cd, int row_chunks) {
    __shared__ double red[8][33];
    const long long k = (long long)blockIdx.x * 32 + threadIdx.x;
    const int K = f.K;
    const long long per = (f.d + row_chunks - 1) / row_chunks;
    const long long r0 = (long long)blockIdx.y * per, r1 = min(f.d, r0 + per);
    double acc[MAXK * (MAXK + 1) / 2];
#pragma unroll
    for (int p = 0; p < MAXK * (MAXK + 1) / 2; ++p) acc[p] = 0.0;
    double sg[MAXK];
#pragma unroll
    for (int i = 0; i < MAXK; ++i) sg[i] = (i < K && k < f.q) ? sign_of(dots, f.q, i, k) : 0.0;
    if (k < f.q) {
        for (long long r = r0 + threadIdx.y; r < r1; r += 8) {
            const double f0 = f.F0[r * f.q + k];
            double dv[MAXK];
#pragma unroll
            for (int i = 0; i < MAXK; ++i) dv[i] = (i < K) ? fma(sg[i], f.F[i][r * f.q + k], -f0) : 0.0;
            int p = 0;
#pragma unroll
            for (int i = 0; i < MAXK; ++i)
#pragma unroll
                for (int j = i; j < MAXK; ++j) acc[p] = fma(dv[i], dv[j], acc[p]), ++p;
        }
    }
    int p = 0;
    for (int i = 0; i < MAXK; ++i)
        for (int j = i; j < MAXK; ++j, ++p) {
            if (i >= K || j >= K) continue;
            red[threadIdx.y][threadIdx.x] = acc[p];
            __syncthreads();
            if (threadIdx.y == 0 && k < f.q) {
                double s = 0.0;
                for (int y = 0; y < 8; ++y) s += red[y][threadIdx.x];
                atomicAdd(&cd[((long long)i * K + j) * f.q + k], s);
            }
            __syncthreads();
        }
}

// Transposed split operand out[k][seg][j] (Qp rows of 4 Lr) of a d x q source,
// j the source row (Lr = Dp; the stacked modes 4 and 5 put two d-row sources
// one above the other, Lr = 2 Dp):
//   0  F_0[j, k];  1  dF_i = s_i F_i - F_0;  2  X[j, k];  3  X[j, k] S_0[k]
//   4  [F_0 ; X];  5  [X ; F_0 + X]
struct SplitT {
    Frames f;
    const double* dots;
    const double* X;
    const double* S0;
    int mode, i;
    float* out;
    long long Dp, Qp;
};
__global__ void __launch_bounds__(256) k_fr_split_t(SplitT a) {
    __shared__ double t[32][33];
    const long long Lr = (a.mode >= 4) ? 2 * a.Dp : a.Dp;
    const long long r0 = (long long)blockIdx.x * 32, k0 = (long long)blockIdx.y * 32;
    const long long d = a.f.d, q = a.f.q;
    for (int y = threadIdx.y; y < 32; y += 8) {
        long long r = r0 + y;
        const long long k = k0 + threadIdx.x;
        int half = 0;
        if (a.mode >= 4 && r >= a.Dp) { half = 1; r -= a.Dp; }
        double v = 0.0;
        if (r < d && k < q) {
            const long long e = r * q + k;
            switch (a.mode) {
                case 0: v = a.f.F0[e]; break;
                case 1: v = fma(sign_of(a.dots, q, a.i, k), a.f.F[a.i][e], -a.f.F0[e]); break;
                case 2: v = a.X[e]; break;
                case 3: v = a.X[e] * a.S0[k]; break;
                case 4: v = half ? a.X[e] : a.f.F0[e]; break;
                case 5: v = half ? a.f.F0[e] + a.X[e] : a.X[e]; break;
            }
        }
        t[y][threadIdx.x] = v;
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long k = k0 + y, r = r0 + threadIdx.x;
        if (k < a.Qp && r < Lr) put_split(a.out + k * 4 * Lr, Lr, r, t[threadIdx.x][y]);
    }
}

// Row-major split operand out[r][seg][c] (rows_p rows of 4 Lp), element value by mode:
//   0  F_0[r, c]                          (d x q)
//   1  F_0[r, c] + X[r, c]                (d x q)
//   2  M[r, c]                            (q x q binary64)
//   3  Y^T[r, c] of the aggregate          (q x q)
//   4  [E_U S_0 | U_0 S_0]                (m x 2 Qp: c < Qp from X = E_U, else U_0)
//   5  [V_0 + E_V | E_V]                  (n x 2 Qp: X = E_V)
//   6  R = (z + (1 - sqrt cs) I) / sqrt cs (q x q, M = z)
struct SplitR {
    Frames f;
    const double* X;
    const double* M;
    const double* S0;
    const double* sym;     // mode 3: K arrays q x q (Sym_i), then K arrays (Kw_i)
    const double* kw;
    const double* coef;
    const FrameHeader* hdr;
    int side;
    long long k_keep;
    int mode;
    float* out;
    long long rows, rows_p, Lp;
    const int32_t* skip;   // optional: nothing to do while *skip != 0
};
__global__ void __launch_bounds__(256) k_fr_split_r(SplitR a) {
    if (a.skip && *reinterpret_cast<const volatile int32_t*>(a.skip)) return;
    const long long total = a.rows_p * a.Lp;
    const long long q = a.f.q;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
        const long long r = e / a.Lp, c = e - r * a.Lp;
        double v = 0.0;
        if (r < a.rows) {
            switch (a.mode) {
                case 0: if (c < q) v = a.f.F0[r * q + c]; break;
                case 1: if (c < q) v = a.f.F0[r * q + c] + a.X[r * q + c]; break;
                case 2: if (c < q) v = a.M[r * q + c]; break;
                case 3:
                    if (c < q) {
                        // Y^T[j, k] = Y[k, j] = Sc[j, k] D_j - Kwc[j, k] (D_j - D_k) / 2
                        const double Dj = r < a.k_keep ? 1.0 : 0.0, Dk = c < a.k_keep ? 1.0 : 0.0;
                        double sc = 0.0, kc = 0.0;
                        for (int i = 0; i < a.f.K; ++i) {
                            sc = fma(a.coef[i], a.sym[((long long)i * q + r) * q + c], sc);
                            kc = fma(a.coef[i], a.kw[((long long)i * q + r) * q + c], kc);
                        }
                        v = sc * Dj - 0.5 * kc * (Dj - Dk);
                    }
                    break;
                case 4: {
                    const long long Qp = a.Lp / 2;
                    if (c < Qp) { if (c < q) v = a.X[r * q + c] * a.S0[c]; }
                    else if (c - Qp < q) v = a.f.F0[r * q + (c - Qp)] * a.S0[c - Qp];
                    break;
                }
                case 5: {
                    const long long Qp = a.Lp / 2;
                    if (c < Qp) { if (c < q) v = a.f.F0[r * q + c] + a.X[r * q + c]; }
                    else if (c - Qp < q) v = a.X[r * q + (c - Qp)];
                    break;
                }
                case 6:
                    if (c < q) {
                        const double sc = sqrt(a.hdr->cs[a.side]);
                        v = (a.M[r * q + c] + (r == c ? 1.0 - sc : 0.0)) / sc;
                    }
                    break;
            }
        }
        put_split(a.out + r * 4 * a.Lp, a.Lp, c, v);
    }
}

// A_i = F_0^T dF_i in binary64 on the CUDA cores (dF_i = s_i F_i - F_0 formed
// on the fly).  The Gram is a small difference of large terms whenever
// frames rotate inside near-degenerate singular subspaces while the proxies
// stay small, so this contraction (and only this one) is carried at the
// paper's binary64 precision.  64 x 64 output tile per block, 16 rows of the
// contraction per step, a 4 x 4 register tile per thread.
__global__ void __launch_bounds__(256) k_fr_ftdf(Frames f, const double* dots, int i, double* A) {
    __shared__ double sa[16][64], sb[16][64];
    __shared__ double sg[64];
    const long long q = f.q, d = f.d;
    const long long k0 = (long long)blockIdx.y * 64, l0 = (long long)blockIdx.x * 64;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    if (threadIdx.x < 64) sg[threadIdx.x] = (l0 + threadIdx.x < q) ? sign_of(dots, q, i, l0 + threadIdx.x) : 0.0;
    double acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.0;
    const double* F0 = f.F0;
    const double* Fi = f.F[i];
    __syncthreads();
    for (long long r0 = 0; r0 < d; r0 += 16) {
        for (int e = threadIdx.x; e < 16 * 64; e += 256) {
            const int rr = e >> 6, cc = e & 63;
            const long long r = r0 + rr;
            const long long ka = k0 + cc, lb = l0 + cc;
            sa[rr][cc] = (r < d && ka < q) ? F0[r * q + ka] : 0.0;
            sb[rr][cc] = (r < d && lb < q) ? fma(sg[cc], Fi[r * q + lb], -F0[r * q + lb]) : 0.0;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            double av[4], bv[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) av[a] = sa[kk][ty * 4 + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) bv[b] = sb[kk][tx * 4 + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = fma(av[a], bv[b], acc[a][b]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const long long k = k0 + ty * 4 + a, l = l0 + tx * 4 + b;
            if (k < q && l < q) A[((long long)i * q + k) * q + l] = acc[a][b];
        }
}

// N = (F + dF)^T (F + dF) - I in binary64, the polar retraction's argument
// (any departure of F^T F from I included, so the retraction also restores
// orthonormality lost to rounding).  N is symmetric: one block per 64 x 64
// tile on or above the diagonal (nt (nt + 1) / 2 blocks for nt tiles a side),
// written to both halves.  Entry (k, l) and entry (l, k) are the same sum of
// the same products in the same order, so the two halves agree bit for bit
// also inside a diagonal tile.  Tiling as in k_fr_ftdf.
__global__ void __launch_bounds__(256) k_op_gram64(const double* F, const double* dF, long long d, long long q,
                                                   double* N) {
    __shared__ double sa[16][64], sb[16][64];
    const long long nt = (q + 63) / 64;
    long long rest = blockIdx.x, tr = 0;
    while (rest >= nt - tr) { rest -= nt - tr; ++tr; }      // at most nt steps
    const long long k0 = tr * 64, l0 = (tr + rest) * 64;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    double acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.0;
    for (long long r0 = 0; r0 < d; r0 += 16) {
        for (int e = threadIdx.x; e < 16 * 64; e += 256) {
            const int rr = e >> 6, cc = e & 63;
            const long long r = r0 + rr;
            const long long ka = k0 + cc, lb = l0 + cc;
            sa[rr][cc] = (r < d && ka < q) ? F[r * q + ka] + dF[r * q + ka] : 0.0;
            sb[rr][cc] = (r < d && lb < q) ? F[r * q + lb] + dF[r * q + lb] : 0.0;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            double av[4], bv[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) av[a] = sa[kk][ty * 4 + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) bv[b] = sb[kk][tx * 4 + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = fma(av[a], bv[b], acc[a][b]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const long long k = k0 + ty * 4 + a, l = l0 + tx * 4 + b;
            if (k < q && l < q) {
                const double v = acc[a][b] - (k == l ? 1.0 : 0.0);
                N[k * q + l] = v;
                if (k0 != l0) N[l * q + k] = v;
            }
        }
}

// Split operands of an m x n bf16 / fp32 matrix G (row stride n): row-major
// (rows Mp of 4 Np, element G[r, c]) or transposed (rows Np of 4 Mp, element
// G[r, c] at row c, position r)
__device__ __forceinline__ double load_typed(const void* p, int dtype, long long e) {
    if (dtype == ISO_BF16) return (double)__uint_as_float((uint32_t)static_cast<const unsigned short*>(p)[e] << 16);
    return (double)static_cast<const float*>(p)[e];
}
__global__ void __launch_bounds__(256) k_op_split_g(const void* G, int dtype, long long m, long long n, long long Mp,
                                                    long long Np, float* out) {
    const long long total = Mp * Np;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
        const long long r = e / Np, c = e - r * Np;
        const double v = (r < m && c < n) ? load_typed(G, dtype, r * n + c) : 0.0;
        put_split(out + r * 4 * Np, Np, c, v);
    }
}
__global__ void __launch_bounds__(256) k_op_split_gt(const void* G, int dtype, long long m, long long n, long long Mp,
                                                     long long Np, float* out) {
    __shared__ double t[32][33];
    const long long r0 = (long long)blockIdx.x * 32, c0 = (long long)blockIdx.y * 32;
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        t[y][threadIdx.x] = (r < m && c < n) ? load_typed(G, dtype, r * n + c) : 0.0;
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long c = c0 + y, r = r0 + threadIdx.x;
        if (c < Np && r < Mp) put_split(out + c * 4 * Mp, Mp, r, t[threadIdx.x][y]);
    }
}

// F += E (binary64, d x q)
__global__ void __launch_bounds__(256) k_op_add(double* F, const double* E, long long total) {
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x)
        F[e] += E[e];
}

// Sym_i = sym(A_i), Kw_i = A_i - Sym_i (binary64; A is K arrays q x q)
__global__ void __launch_bounds__(256) k_fr_symskew(const double* A, long long Qp, long long q, double* sym, double* kw) {
    __shared__ double ta[32][33], tb[32][33];
    const int i = blockIdx.z;
    const double* Ai = A + (long long)i * q * q;
    const long long r0 = (long long)blockIdx.y * 32, c0 = (long long)blockIdx.x * 32;
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long ra = r0 + y, ca = c0 + threadIdx.x, rb = c0 + y, cb = r0 + threadIdx.x;
        ta[y][threadIdx.x] = (ra < q && ca < q) ? Ai[ra * q + ca] : 0.0;   // A[r0 + y, c0 + x]
        tb[y][threadIdx.x] = (rb < q && cb < q) ? Ai[rb * q + cb] : 0.0;   // A[c0 + y, r0 + x]
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        if (r < q && c < q) {
            const double a = ta[y][threadIdx.x], b = tb[threadIdx.x][y];   // A[r, c], A[c, r]
            sym[((long long)i * q + r) * q + c] = 0.5 * (a + b);
            kw[((long long)i * q + r) * q + c] = 0.5 * (a - b);
        }
    }
}

// Gamma_ij (i <= j), summed into gram[i][j]; block y covers a slice of the q x q entries
struct GramArgs {
    const double* A[2];         // per side: K arrays q x q
    const double* sym[2];
    const double* kw[2];
    const double* cd[2];        // per side: K x K x q
    const double* S0;
    double* gram;
    long long q, Qp, k_keep;
    int K;
};
__global__ void __launch_bounds__(256) k_fr_gram(GramArgs g) {
    __shared__ double red[32];
    // pair (i, j), i <= j, from blockIdx.x
    int i = 0, j = 0, p = blockIdx.x;
    for (i = 0; i < g.K; ++i) {
        if (p < g.K - i) { j = i + p; break; }
        p -= g.K - i;
    }
    const long long q = g.q, qq = q * q;
    const long long per = (qq + gridDim.y - 1) / gridDim.y;
    const long long e0 = (long long)blockIdx.y * per, e1 = min(qq, e0 + per);
    double acc = 0.0;
    for (long long e = e0 + threadIdx.x; e < e1; e += blockDim.x) {
        const long long r = e / q, c = e - r * q;
        const double sr = g.S0[r], sc = g.S0[c];
        const double Dr = r < g.k_keep ? 1.0 : 0.0, Dc = c < g.k_keep ? 1.0 : 0.0;
        // column terms (row l = r, column k = c), both sides
        double colt = 0.0;
#pragma unroll
        for (int s = 0; s < 2; ++s) {
            const double ai = g.A[s][(long long)i * qq + e];
            const double aj = g.A[s][(long long)j * qq + e];
            const double si = g.sym[s][(long long)i * qq + e], sj = g.sym[s][(long long)j * qq + e];
            colt += ai * sj + si * aj - si * sj;
        }
        acc -= sc * sc * Dc * colt;
        // cross terms (k = r, l = c)
        const double kui = g.kw[0][(long long)i * qq + e], kuj = g.kw[0][(long long)j * qq + e];
        const double kvi = g.kw[1][(long long)i * qq + e], kvj = g.kw[1][(long long)j * qq + e];
        acc -= sr * sc * Dr * Dc * (kui * kvj + kuj * kvi);
    }
    if (blockIdx.y == 0)
        for (long long k = threadIdx.x; k < min(q, g.k_keep); k += blockDim.x)
            acc += g.S0[k] * g.S0[k] *
                   (g.cd[0][((long long)i * g.K + j) * q + k] + g.cd[1][((long long)i * g.K + j) * q + k]);
    acc = block_sum(acc, red);
    if (threadIdx.x == 0) atomicAdd(&g.gram[i * g.K + j], acc);
}

// c* from Gamma (upper triangle), then the caller's stats
__global__ void k_fr_solve(double* gram, double* coef, int K, double ridge, double c_min, double c_max,
                           double* st_gram, double* st_coef) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    double G[MAXK * MAXK], c[MAXK];
    for (int a = 0; a < K; ++a)
        for (int b = a; b < K; ++b) {
            G[a * K + b] = gram[a * K + b];
            G[b * K + a] = gram[a * K + b];
        }
    for (int a = 0; a < K * K; ++a) gram[a] = G[a];
    retention_solve(G, K, ridge, c_min, c_max, c);
    for (int a = 0; a < K; ++a) coef[a] = c[a];
    if (st_gram) for (int a = 0; a < K * K; ++a) st_gram[a] = G[a];
    if (st_coef) for (int a = 0; a < K; ++a) st_coef[a] = c[a];
}

// xi* = D dF_c - E (E = F_0 Y from the GEMM, ld Qp)
__global__ void __launch_bounds__(256) k_fr_xi(Frames f, const double* dots, const double* coef, const float* E,
                                               long long Qp, long long k_keep, double* xi) {
    const long long total = f.d * f.q;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
        const long long r = e / f.q, k = e - r * f.q;
        double v = 0.0;
        if (k < k_keep) {
            const double f0 = f.F0[e];
            for (int i = 0; i < f.K; ++i) v = fma(coef[i], fma(sign_of(dots, f.q, i, k), f.F[i][e], -f0), v);
        }
        xi[e] = v - (double)E[r * Qp + k];
    }
}

// ||N||_F^2 of N = xi^T xi (binary32, ld Qp; or binary64, ld q), summed into the header
__global__ void __launch_bounds__(256) k_fr_norm(const float* N, const double* N64, long long Qp, long long q,
                                                 FrameHeader* h, int side) {
    __shared__ double red[32];
    double acc = 0.0;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < q * q; e += (long long)gridDim.x * blockDim.x) {
        const long long r = e / q, c = e - r * q;
        const double v = N64 ? N64[e] : (double)N[r * Qp + c];
        acc += v * v;
    }
    acc = block_sum(acc, red);
    if (threadIdx.x == 0) atomicAdd(&h->nu2[side], acc);
}

// The Newton-Schulz iterates y, z and the step m are symmetric in exact
// arithmetic (functions of N); the products treat them so (B = M^T = M).  Each
// kernel below symmetrises what it writes, one 32 x 32 tile and its mirror
// per block (blocks below the diagonal return), so that rounding cannot
// build an asymmetric component from one iteration to the next.  Reading
// both tiles before writing either makes the update safe in place.
struct NsArgs {
    const float* N;     // init: N = xi^T xi (binary32, ld Qp), unless N64 is given
    const double* N64;  // init: N in binary64 (ld q)
    const float* T1;    // m: z y;  update: y m
    const float* T2;    // update: m z
    double* y;
    double* z;
    double* m;
    FrameHeader* h;
    long long q, Qp;
    int side, it;
};

__device__ __forceinline__ bool ns_tile(long long q, long long& r0, long long& c0) {
    if (blockIdx.x < blockIdx.y) return false;
    r0 = (long long)blockIdx.y * 32;
    c0 = (long long)blockIdx.x * 32;
    return true;
}

// Y_0 = (I + N) / cs = I + y, Z_0 = I (z = 0); cs = 1 while ||N||_F < 0.9,
// else 1 + ||N||_F / 2, so that the eigenvalues of Y_0 lie in (0, 2)
__global__ void __launch_bounds__(256) k_fr_ns_init(NsArgs a) {
    __shared__ double ta[32][33], tb[32][33];
    long long r0, c0;
    if (!ns_tile(a.q, r0, c0)) return;
    const double nu = sqrt(a.h->nu2[a.side]);
    const double cs = nu < 0.9 ? 1.0 : 1.0 + 0.5 * nu;
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0 && threadIdx.y == 0) {
        a.h->cs[a.side] = cs;
        a.h->conv[a.side] = 0;
    }
    auto f = [&](long long r, long long c) -> double {
        if (r >= a.q || c >= a.q) return 0.0;
        const double id = r == c ? 1.0 : 0.0;
        const double nv = a.N64 ? a.N64[r * a.q + c] : (double)a.N[r * a.Qp + c];
        return (id + nv) / cs - id;
    };
    for (int y = threadIdx.y; y < 32; y += 8) {
        ta[y][threadIdx.x] = f(r0 + y, c0 + threadIdx.x);
        tb[y][threadIdx.x] = f(c0 + y, r0 + threadIdx.x);
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        if (r < a.q && c < a.q) {
            a.y[r * a.q + c] = 0.5 * (ta[y][threadIdx.x] + tb[threadIdx.x][y]);
            a.z[r * a.q + c] = 0.0;
        }
        const long long r2 = c0 + y, c2 = r0 + threadIdx.x;
        if (r2 < a.q && c2 < a.q) {
            a.y[r2 * a.q + c2] = 0.5 * (tb[y][threadIdx.x] + ta[threadIdx.x][y]);
            a.z[r2 * a.q + c2] = 0.0;
        }
    }
}

// w = y + z + z y (the residual Z Y - I), m = -w / 2; the largest |w| of the
// iteration goes to the header
__global__ void __launch_bounds__(256) k_fr_ns_m(NsArgs a) {
    __shared__ double ta[32][33], tb[32][33];
    if (*reinterpret_cast<volatile int32_t*>(&a.h->conv[a.side])) return;
    long long r0, c0;
    if (!ns_tile(a.q, r0, c0)) return;
    auto w = [&](long long r, long long c) -> double {
        if (r >= a.q || c >= a.q) return 0.0;
        const long long e = r * a.q + c;
        return a.y[e] + a.z[e] + (double)a.T1[r * a.Qp + c];
    };
    for (int y = threadIdx.y; y < 32; y += 8) {
        ta[y][threadIdx.x] = w(r0 + y, c0 + threadIdx.x);
        tb[y][threadIdx.x] = w(c0 + y, r0 + threadIdx.x);
    }
    __syncthreads();
    float wm = 0.0f;
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        if (r < a.q && c < a.q) {
            const double v = 0.5 * (ta[y][threadIdx.x] + tb[threadIdx.x][y]);
            a.m[r * a.q + c] = -0.5 * v;
            wm = fmaxf(wm, (float)fabs(v));
        }
        const long long r2 = c0 + y, c2 = r0 + threadIdx.x;
        if (r2 < a.q && c2 < a.q) a.m[r2 * a.q + c2] = -0.25 * (tb[y][threadIdx.x] + ta[threadIdx.x][y]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xFFFFFFFFu, wm, o));
    if ((threadIdx.x & 31) == 0) atomicMax(&a.h->wmax[a.side][a.it], __float_as_uint(wm));
}

// y += m + y m, z += m + m z, in place.  The iteration stops (this update and
// every later one skipped) once the residual is at the tolerance, or has
// stopped its quadratic fall below 1e-2 (the rounding floor of the products),
// or has grown.
__global__ void __launch_bounds__(256) k_fr_ns_update(NsArgs a) {
    __shared__ double ya[32][33], yb[32][33], za[32][33], zb[32][33];
    if (*reinterpret_cast<volatile int32_t*>(&a.h->conv[a.side])) return;
    const double wc = (double)__uint_as_float(a.h->wmax[a.side][a.it]);
    const double wp = a.it > 0 ? (double)__uint_as_float(a.h->wmax[a.side][a.it - 1]) : 1e300;
    const bool stop = !(wc > FR_NS_TOL) || wc >= wp || (wc < 1e-2 && wc > 0.25 * wp);
    if (stop) {
        if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0 && threadIdx.y == 0) a.h->conv[a.side] = 1;
        return;
    }
    long long r0, c0;
    if (!ns_tile(a.q, r0, c0)) return;
    auto fy = [&](long long r, long long c) -> double {
        if (r >= a.q || c >= a.q) return 0.0;
        const long long e = r * a.q + c;
        return a.y[e] + a.m[e] + (double)a.T1[r * a.Qp + c];
    };
    auto fz = [&](long long r, long long c) -> double {
        if (r >= a.q || c >= a.q) return 0.0;
        const long long e = r * a.q + c;
        return a.z[e] + a.m[e] + (double)a.T2[r * a.Qp + c];
    };
    for (int y = threadIdx.y; y < 32; y += 8) {
        ya[y][threadIdx.x] = fy(r0 + y, c0 + threadIdx.x);
        yb[y][threadIdx.x] = fy(c0 + y, r0 + threadIdx.x);
        za[y][threadIdx.x] = fz(r0 + y, c0 + threadIdx.x);
        zb[y][threadIdx.x] = fz(c0 + y, r0 + threadIdx.x);
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const long long r = r0 + y, c = c0 + threadIdx.x;
        if (r < a.q && c < a.q) {
            a.y[r * a.q + c] = 0.5 * (ya[y][threadIdx.x] + yb[threadIdx.x][y]);
            a.z[r * a.q + c] = 0.5 * (za[y][threadIdx.x] + zb[threadIdx.x][y]);
        }
        const long long r2 = c0 + y, c2 = r0 + threadIdx.x;
        if (r2 < a.q && c2 < a.q) {
            a.y[r2 * a.q + c2] = 0.5 * (yb[y][threadIdx.x] + ya[threadIdx.x][y]);
            a.z[r2 * a.q + c2] = 0.5 * (zb[y][threadIdx.x] + za[threadIdx.x][y]);
        }
    }
}

// E_F = xi* + (F_0 + xi*) R (P from the GEMM, ld Qp), in place over xi*
__global__ void __launch_bounds__(256) k_fr_motion(double* xi, const float* P, long long Qp, long long d, long long q) {
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < d * q; e += (long long)gridDim.x * blockDim.x) {
        const long long r = e / q, c = e - r * q;
        xi[e] += (double)P[r * Qp + c];
    }
}

__global__ void k_fr_status(const FrameHeader* h, int32_t* out) {
    if (threadIdx.x == 0 && blockIdx.x == 0) *out = h->status;
}

// ---------------------------------------------------------------------------
// host
// ---------------------------------------------------------------------------
size_t al256(size_t v) { return (v + 255) & ~(size_t)255; }

struct FrameLayout {
    long long m, n, q, Mp, Np, Qp, K;
    size_t hdr, gram, coef, dots, vcopy;
    size_t cd[2], ft4[2], aq[2], sym[2], kw[2], fr4[2], y4[2], e[2], xi[2], nq[2];
    size_t ns_y, ns_z, ns_m, ns_y4, ns_z4, ns_m4, ns_t1, ns_t2, ns_t3;
    size_t a6, b6, total;
};

FrameLayout frame_layout(long long m, long long n, int K) {
    FrameLayout L;
    L.m = m; L.n = n; L.K = K;
    L.q = std::min(m, n);
    L.Mp = pad_up(m); L.Np = pad_up(n); L.Qp = pad_up(L.q);
    const long long q = L.q, Qp = L.Qp;
    size_t o = 0;
    auto take = [&](size_t bytes) { const size_t at = o; o = al256(o + bytes); return at; };
    L.hdr = take(sizeof(FrameHeader));
    L.gram = take(sizeof(double) * K * K);
    L.coef = take(sizeof(double) * K);
    L.dots = take(sizeof(double) * K * q);
    for (int s = 0; s < 2; ++s) L.cd[s] = take(sizeof(double) * K * K * q);
    L.vcopy = take(sizeof(double) * (K + 1) * n * q);
    for (int s = 0; s < 2; ++s) {
        const long long Dp = s == 0 ? L.Mp : L.Np, d = s == 0 ? m : n;
        L.ft4[s] = take(sizeof(float) * Qp * 4 * Dp);      // xi*^T split
        L.aq[s] = take(sizeof(double) * K * q * q);        // A_i = F_0^T dF_i (binary64)
        L.sym[s] = take(sizeof(double) * K * q * q);
        L.kw[s] = take(sizeof(double) * K * q * q);
        L.fr4[s] = take(sizeof(float) * Dp * 4 * Qp);      // F_0 split, later (F_0 + xi*) split
        L.y4[s] = take(sizeof(float) * Qp * 4 * Qp);       // Y^T split, later R split
        L.e[s] = take(sizeof(float) * Dp * Qp);            // F_0 Y, later (F_0 + xi*) R
        L.xi[s] = take(sizeof(double) * d * q);            // xi*, later E_F
        L.nq[s] = take(sizeof(float) * Qp * Qp);
    }
    L.ns_y = take(sizeof(double) * q * q);
    L.ns_z = take(sizeof(double) * q * q);
    L.ns_m = take(sizeof(double) * q * q);
    L.ns_y4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_z4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_m4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_t1 = take(sizeof(float) * Qp * Qp);
    L.ns_t2 = take(sizeof(float) * Qp * Qp);
    L.ns_t3 = take(sizeof(float) * Qp * Qp);
    L.a6 = take(sizeof(float) * L.Mp * 4 * 2 * Qp);
    L.b6 = take(sizeof(float) * L.Np * 4 * 2 * Qp);
    L.total = o;
    return L;
}

int grid_of(long long work, int sms) {
    const long long b = (work + 255) / 256;
    return (int)std::max(1LL, std::min(b, (long long)sms * 8));
}

int gemm_smem_optin() {
    static int done = 0;
    if (done) return ISO_OK;
    if (cudaFuncSetAttribute(k_gemm_tf32, cudaFuncAttributeMaxDynamicSharedMemorySize, GEMM_SMEM) != cudaSuccess)
        return ISO_ERR_CUDA;
    done = 1;
    return ISO_OK;
}

// C (a_rows x b_rows) = A B^T over the three-product split: A and B are
// four-segment operand arrays of segment length L (rows a_rows / b_rows,
// multiples of 128).
int frame_gemm(cudaStream_t s, const float* A, long long a_rows, const float* B, long long b_rows, long long L,
               GemmArgs g) {
    CUtensorMap ta, tb;
    ISO_TRY(gemm_tensor_map(&ta, A, a_rows, 4 * L, 4 * L));
    ISO_TRY(gemm_tensor_map(&tb, B, b_rows, 4 * L, 4 * L));
    g.k_tiles = (int)(3 * L / GEMM_BK);
    g.a_k0 = 0;
    g.b_k0 = (int)L;
    ISO_TRY(gemm_smem_optin());
    const dim3 grid((unsigned)(b_rows / GEMM_BN), (unsigned)(a_rows / GEMM_BM));
    const int slot = prof_begin(0, s);
    k_gemm_tf32<<<grid, GEMM_THREADS, GEMM_SMEM, s>>>(ta, tb, g);
    prof_end(slot, s);
    return cudaGetLastError() == cudaSuccess ? ISO_OK : ISO_ERR_CUDA;
}

struct OptLayout {
    long long m, n, q, Mp, Np, Qp, Dmax;
    size_t hdr, gw4, gwt4, su4, sv4, dF[2], n64, xb4, r4, p, a6, b6;
    size_t ns_y, ns_z, ns_m, ns_y4, ns_z4, ns_m4, ns_t1, ns_t2, ns_t3, total;
};

OptLayout opt_layout(long long m, long long n) {
    OptLayout L;
    L.m = m; L.n = n; L.q = std::min(m, n);
    L.Mp = pad_up(m); L.Np = pad_up(n); L.Qp = pad_up(L.q);
    L.Dmax = std::max(L.Mp, L.Np);
    const long long q = L.q, Qp = L.Qp;
    size_t o = 0;
    auto take = [&](size_t bytes) { const size_t at = o; o = al256(o + bytes); return at; };
    L.hdr = take(sizeof(FrameHeader));
    L.gw4 = take(sizeof(float) * L.Mp * 4 * L.Np);      // G_W, rows m, contraction n
    L.gwt4 = take(sizeof(float) * L.Np * 4 * L.Mp);     // G_W^T, rows n, contraction m
    L.su4 = take(sizeof(float) * Qp * 4 * L.Mp);        // (U S_0)^T
    L.sv4 = take(sizeof(float) * Qp * 4 * L.Np);        // (V S_0)^T
    L.dF[0] = take(sizeof(double) * m * q);             // U_bar - U, later E_U
    L.dF[1] = take(sizeof(double) * n * q);             // V_bar - V, later E_V
    L.n64 = take(sizeof(double) * q * q);               // (F + dF)^T (F + dF) - I
    L.xb4 = take(sizeof(float) * L.Dmax * 4 * Qp);      // F + dF
    L.r4 = take(sizeof(float) * Qp * 4 * Qp);
    L.p = take(sizeof(float) * L.Dmax * Qp);
    L.a6 = take(sizeof(float) * L.Mp * 4 * 2 * Qp);
    L.b6 = take(sizeof(float) * L.Np * 4 * 2 * Qp);
    L.ns_y = take(sizeof(double) * q * q);
    L.ns_z = take(sizeof(double) * q * q);
    L.ns_m = take(sizeof(double) * q * q);
    L.ns_y4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_z4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_m4 = take(sizeof(float) * Qp * 4 * Qp);
    L.ns_t1 = take(sizeof(float) * Qp * Qp);
    L.ns_t2 = take(sizeof(float) * Qp * Qp);
    L.ns_t3 = take(sizeof(float) * Qp * Qp);
    L.total = o;
    return L;
}

// launch one CUDA-core kernel of the frame merge / optimizer step on stream s
#define FR_LAUNCH(...) do { const int _slot = prof_begin(1, s); __VA_ARGS__; prof_end(_slot, s); \
                                if (cudaGetLastError() != cudaSuccess) return ISO_ERR_CUDA; } while (0)

// Scratch of the inverse square root
struct NsBufs {
    double *y, *z, *m;
    float *y4, *z4, *m4, *t1, *t2, *t3;
};

// R = (I + N)^(-1/2) - I for N = X^T X (binary32, ld Qp) with X^T F_0 skew,
// by the difference-form Newton-Schulz iteration (k_fr_ns_*), written as
// the split operand R4 (Qp rows of 4 Qp; R is symmetric, so it serves as B
// of (F_0 + X) R).  Header slot `side` holds its scaling and state.
int ns_root(cudaStream_t s, int sms, FrameHeader* hdr, int side, const float* Nq, const double* N64, long long q,
            long long Qp, const NsBufs& b, int ns_iters, float* R4) {
    FR_LAUNCH((k_fr_norm<<<grid_of(q * q, sms), 256, 0, s>>>(Nq, N64, Qp, q, hdr, side)));
    NsArgs na{};
    na.N = Nq; na.N64 = N64; na.y = b.y; na.z = b.z; na.m = b.m; na.h = hdr;
    na.q = q; na.Qp = Qp; na.side = side;
    const dim3 tiles((unsigned)((q + 31) / 32), (unsigned)((q + 31) / 32)), tb(32, 8);
    FR_LAUNCH((k_fr_ns_init<<<tiles, tb, 0, s>>>(na)));
    SplitR sq{};
    sq.f.q = q; sq.hdr = hdr; sq.side = side; sq.mode = 2; sq.rows = q; sq.rows_p = Qp; sq.Lp = Qp;
    sq.skip = &hdr->conv[side];
    auto split_q = [&](const double* M_, float* out) -> int {
        sq.M = M_; sq.out = out;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Qp * Qp, sms), 256, 0, s>>>(sq)));
        return ISO_OK;
    };
    ISO_TRY(split_q(b.y, b.y4));
    ISO_TRY(split_q(b.z, b.z4));
    for (int it = 0; it < ns_iters; ++it) {
        GemmArgs g{};
        g.mode = GEMM_STORE_F32; g.ldc = Qp; g.M = (int)Qp; g.N = (int)Qp; g.status = &hdr->status;
        g.skip = &hdr->conv[side];
        g.C = b.t1;
        ISO_TRY(frame_gemm(s, b.z4, Qp, b.y4, Qp, Qp, g));     // z y
        na.it = it;
        na.T1 = b.t1;
        FR_LAUNCH((k_fr_ns_m<<<tiles, tb, 0, s>>>(na)));
        ISO_TRY(split_q(b.m, b.m4));
        g.C = b.t2;
        ISO_TRY(frame_gemm(s, b.y4, Qp, b.m4, Qp, Qp, g));     // y m
        g.C = b.t3;
        ISO_TRY(frame_gemm(s, b.m4, Qp, b.z4, Qp, Qp, g));     // m z
        na.T1 = b.t2;
        na.T2 = b.t3;
        FR_LAUNCH((k_fr_ns_update<<<tiles, tb, 0, s>>>(na)));
        ISO_TRY(split_q(b.y, b.y4));
        ISO_TRY(split_q(b.z, b.z4));
    }
    SplitR sr{};
    sr.f.q = q; sr.hdr = hdr; sr.side = side; sr.mode = 6; sr.M = b.z; sr.out = R4;
    sr.rows = q; sr.rows_p = Qp; sr.Lp = Qp;
    FR_LAUNCH((k_fr_split_r<<<grid_of(Qp * Qp, sms), 256, 0, s>>>(sr)));
    return ISO_OK;
}

}  // namespace
}  // namespace iso

using namespace iso;

extern "C" {

int32_t iso_frame_workspace_size(int64_t m, int64_t n, int32_t K, size_t* bytes) {
    if (!bytes || m < 1 || n < 1 || K < 1) return ISO_ERR_ARG;
    if (K > ISO_MAX_EXPERTS) return ISO_ERR_UNSUPPORTED;
    if (m >= (1LL << 24) || n >= (1LL << 24) || std::min(m, n) > 32768) return ISO_ERR_UNSUPPORTED;
    *bytes = frame_layout(m, n, K).total;
    return ISO_OK;
}

int32_t iso_frame_merge(const double* U0, const double* S0, const double* Vt0, const double* const* U,
                        const double* const* Vt, int32_t K, int64_t m, int64_t n, const iso_tensor* W0,
                        const iso_tensor* out, const iso_frame_cfg* cfg, void* workspace, size_t ws_bytes,
                        const iso_merge_stats* stats, void* stream) {
    size_t need = 0;
    ISO_TRY(iso_frame_workspace_size(m, n, K, &need));
    if (!U0 || !S0 || !Vt0 || !U || !Vt || !W0 || !out || !cfg) return ISO_ERR_ARG;
    for (int i = 0; i < K; ++i)
        if (!U[i] || !Vt[i]) return ISO_ERR_ARG;
    auto al8 = [](const void* p) { return ((uintptr_t)p & 7u) == 0; };
    if (!al8(U0) || !al8(S0) || !al8(Vt0)) return ISO_ERR_ALIGN;
    for (int i = 0; i < K; ++i)
        if (!al8(U[i]) || !al8(Vt[i])) return ISO_ERR_ALIGN;
    if (!(cfg->rho_keep > 0.0 && cfg->rho_keep <= 1.0)) return ISO_ERR_ARG;
    if (!(cfg->ridge >= 0.0) || !std::isfinite(cfg->ridge)) return ISO_ERR_ARG;
    if (!std::isfinite(cfg->c_min) || !std::isfinite(cfg->c_max) || cfg->c_min > cfg->c_max) return ISO_ERR_ARG;
    if (cfg->ns_iters < 0 || cfg->ns_iters > FR_MAX_NS || cfg->reserved != 0) return ISO_ERR_ARG;
    if (W0->rows != m || W0->cols != n || out->rows != m || out->cols != n) return ISO_ERR_SHAPE;
    if ((W0->dtype != ISO_BF16 && W0->dtype != ISO_F32) || out->dtype != W0->dtype) return ISO_ERR_DTYPE;
    if (!W0->data || !out->data) return ISO_ERR_ARG;
    if (((uintptr_t)W0->data & 15u) || ((uintptr_t)out->data & 15u)) return ISO_ERR_ALIGN;
    if (!workspace || ((uintptr_t)workspace & 255u)) return ISO_ERR_WORKSPACE;
    if (ws_bytes < need) return ISO_ERR_WORKSPACE;
    // out may coincide with W0 (each entry is read and written by one thread);
    // it may share no other byte with an input
    {
        const size_t es = W0->dtype == ISO_BF16 ? 2 : 4;
        const uintptr_t o0 = (uintptr_t)out->data, o1 = o0 + (uintptr_t)(m * n) * es;
        const uintptr_t w0 = (uintptr_t)W0->data;
        if (o0 != w0 && o0 < w0 + (uintptr_t)(m * n) * es && w0 < o1) return ISO_ERR_ARG;
    }
    const FrameLayout L = frame_layout(m, n, K);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    char* ws = static_cast<char*>(workspace);
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return ISO_ERR_CUDA;
    const long long q = L.q, Qp = L.Qp;
    long long k_keep = (long long)std::floor(cfg->rho_keep * (double)q + 0.5);
    k_keep = std::max(0LL, std::min(q, k_keep));
    const int ns_iters = cfg->ns_iters ? cfg->ns_iters : FR_DEFAULT_NS;
    FrameHeader* hdr = reinterpret_cast<FrameHeader*>(ws + L.hdr);
    double* gram = reinterpret_cast<double*>(ws + L.gram);
    double* coef = reinterpret_cast<double*>(ws + L.coef);
    double* dots = reinterpret_cast<double*>(ws + L.dots);
    auto F = [&](size_t off) { return reinterpret_cast<float*>(ws + off); };
    auto D = [&](size_t off) { return reinterpret_cast<double*>(ws + off); };

    // header, Gamma, c*, the sign dots and the column dots start at zero
    if (cudaMemsetAsync(ws, 0, L.cd[1] + sizeof(double) * K * K * q, s) != cudaSuccess) return ISO_ERR_CUDA;

    // the V side as n x q row-major frames
    Frames fr[2];
    fr[0].F0 = U0; fr[0].K = K; fr[0].d = m; fr[0].q = q;
    fr[1].F0 = D(L.vcopy); fr[1].K = K; fr[1].d = n; fr[1].q = q;
    for (int i = 0; i < MAXK; ++i) {
        fr[0].F[i] = i < K ? U[i] : nullptr;
        fr[1].F[i] = i < K ? D(L.vcopy) + (size_t)(i + 1) * n * q : nullptr;
    }
    {
        const dim3 blk(32, 8), grd((unsigned)((n + 31) / 32), (unsigned)((q + 31) / 32));
        FR_LAUNCH((k_fr_transpose<<<grd, blk, 0, s>>>(Vt0, D(L.vcopy), q, n)));
        for (int i = 0; i < K; ++i)
            FR_LAUNCH((k_fr_transpose<<<grd, blk, 0, s>>>(Vt[i], D(L.vcopy) + (size_t)(i + 1) * n * q, q, n)));
    }
    // signs (from the U frames), then the column dot products of each side
    {
        const int rc = (int)std::max(1LL, std::min(64LL, ((long long)m + 511) / 512));
        FR_LAUNCH((k_fr_signdots<<<dim3((unsigned)((q + 31) / 32), K, rc), dim3(32, 8), 0, s>>>(fr[0], dots, rc)));
        for (int sd = 0; sd < 2; ++sd) {
            const int r2 = (int)std::max(1LL, std::min(256LL, (fr[sd].d + 255) / 256));
            FR_LAUNCH((k_fr_coldots<<<dim3((unsigned)((q + 31) / 32), r2), dim3(32, 8), 0, s>>>(
                fr[sd], dots, D(L.cd[sd]), r2)));
        }
    }
    // A_i = F_0^T dF_i (binary64), then Sym_i and Kw_i
    for (int sd = 0; sd < 2; ++sd) {
        const dim3 grd((unsigned)((q + 63) / 64), (unsigned)((q + 63) / 64));
        for (int i = 0; i < K; ++i)
            FR_LAUNCH((k_fr_ftdf<<<grd, 256, 0, s>>>(fr[sd], dots, i, D(L.aq[sd]))));
        FR_LAUNCH((k_fr_symskew<<<dim3((unsigned)(Qp / 32), (unsigned)(Qp / 32), K), dim3(32, 8), 0, s>>>(
            D(L.aq[sd]), Qp, q, D(L.sym[sd]), D(L.kw[sd]))));
    }
    // Gamma and c*
    {
        GramArgs ga{};
        for (int sd = 0; sd < 2; ++sd) {
            ga.A[sd] = D(L.aq[sd]); ga.sym[sd] = D(L.sym[sd]); ga.kw[sd] = D(L.kw[sd]); ga.cd[sd] = D(L.cd[sd]);
        }
        ga.S0 = S0; ga.gram = gram; ga.q = q; ga.Qp = Qp; ga.k_keep = k_keep; ga.K = K;
        const int pairs = K * (K + 1) / 2;
        const int slices = (int)std::max(1LL, std::min((long long)sms * 4, (q * q + 4095) / 4096));
        FR_LAUNCH((k_fr_gram<<<dim3(pairs, slices), 256, 0, s>>>(ga)));
        FR_LAUNCH((k_fr_solve<<<1, 32, 0, s>>>(gram, coef, K, cfg->ridge, cfg->c_min, cfg->c_max,
                                                stats ? stats->gram : nullptr, stats ? stats->coef : nullptr)));
    }
    // per side: aggregate tangent, polar factor, motion E_F
    for (int sd = 0; sd < 2; ++sd) {
        const long long Dp = sd == 0 ? L.Mp : L.Np, d = fr[sd].d;
        SplitR sr{};
        sr.f = fr[sd]; sr.S0 = S0; sr.sym = D(L.sym[sd]); sr.kw = D(L.kw[sd]); sr.coef = coef; sr.hdr = hdr;
        sr.side = sd; sr.k_keep = k_keep;
        // Y^T, F_0, then E = F_0 Y
        sr.mode = 3; sr.out = F(L.y4[sd]); sr.rows = q; sr.rows_p = Qp; sr.Lp = Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Qp * Qp, sms), 256, 0, s>>>(sr)));
        sr.mode = 0; sr.out = F(L.fr4[sd]); sr.rows = d; sr.rows_p = Dp; sr.Lp = Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Dp * Qp, sms), 256, 0, s>>>(sr)));
        {
            GemmArgs g{};
            g.mode = GEMM_STORE_F32; g.C = F(L.e[sd]); g.ldc = Qp; g.M = (int)Dp; g.N = (int)Qp; g.status = &hdr->status;
            ISO_TRY(frame_gemm(s, F(L.fr4[sd]), Dp, F(L.y4[sd]), Qp, Qp, g));
        }
        FR_LAUNCH((k_fr_xi<<<grid_of(d * q, sms), 256, 0, s>>>(fr[sd], dots, coef, F(L.e[sd]), Qp, k_keep, D(L.xi[sd]))));
        // N = xi*^T xi*
        {
            SplitT st{};
            st.f = fr[sd]; st.dots = dots; st.X = D(L.xi[sd]); st.mode = 2; st.out = F(L.ft4[sd]); st.Dp = Dp; st.Qp = Qp;
            FR_LAUNCH((k_fr_split_t<<<dim3((unsigned)(Dp / 32), (unsigned)(Qp / 32)), dim3(32, 8), 0, s>>>(st)));
            GemmArgs g{};
            g.mode = GEMM_STORE_F32; g.C = F(L.nq[sd]); g.ldc = Qp; g.M = (int)Qp; g.N = (int)Qp; g.status = &hdr->status;
            ISO_TRY(frame_gemm(s, F(L.ft4[sd]), Qp, F(L.ft4[sd]), Qp, Dp, g));
        }
        // (I + N)^(-1/2) = I + R by the difference-form Newton-Schulz iteration,
        // then F_0 + xi*, and E_F = xi* + (F_0 + xi*) R
        {
            NsBufs nb{D(L.ns_y), D(L.ns_z), D(L.ns_m), F(L.ns_y4), F(L.ns_z4), F(L.ns_m4), F(L.ns_t1),
                      F(L.ns_t2), F(L.ns_t3)};
            ISO_TRY(ns_root(s, sms, hdr, sd, F(L.nq[sd]), nullptr, q, Qp, nb, ns_iters, F(L.y4[sd])));
        }
        sr.mode = 1; sr.X = D(L.xi[sd]); sr.out = F(L.fr4[sd]); sr.rows = d; sr.rows_p = Dp; sr.Lp = Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Dp * Qp, sms), 256, 0, s>>>(sr)));
        {
            GemmArgs g{};
            g.mode = GEMM_STORE_F32; g.C = F(L.e[sd]); g.ldc = Qp; g.M = (int)Dp; g.N = (int)Qp; g.status = &hdr->status;
            ISO_TRY(frame_gemm(s, F(L.fr4[sd]), Dp, F(L.y4[sd]), Qp, Qp, g));
        }
        FR_LAUNCH((k_fr_motion<<<grid_of(d * q, sms), 256, 0, s>>>(D(L.xi[sd]), F(L.e[sd]), Qp, d, q)));
        // the reconstruction's operand of this side
        sr.X = D(L.xi[sd]);
        sr.mode = sd == 0 ? 4 : 5;
        sr.out = F(sd == 0 ? L.a6 : L.b6);
        sr.rows = d; sr.rows_p = Dp; sr.Lp = 2 * Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Dp * 2 * Qp, sms), 256, 0, s>>>(sr)));
    }
    // W* = W_0 + [E_U S_0 | U_0 S_0] [V* | E_V]^T
    {
        GemmArgs g{};
        g.mode = GEMM_ADD_BASE; g.M = (int)m; g.N = (int)n; g.out = out->data; g.w0 = W0->data; g.ldo = n;
        g.out_dtype = W0->dtype; g.status = &hdr->status;
        ISO_TRY(frame_gemm(s, F(L.a6), L.Mp, F(L.b6), L.Np, 2 * Qp, g));
    }
    if (stats && stats->status) FR_LAUNCH((k_fr_status<<<1, 32, 0, s>>>(hdr, stats->status)));
    return ISO_OK;
}

int32_t iso_opt_workspace_size(int64_t m, int64_t n, size_t* bytes) {
    if (!bytes || m < 1 || n < 1) return ISO_ERR_ARG;
    if (m >= (1LL << 24) || n >= (1LL << 24) || std::min(m, n) > 32768) return ISO_ERR_UNSUPPORTED;
    *bytes = opt_layout(m, n).total;
    return ISO_OK;
}

int32_t iso_opt_step(double* U, double* V, const double* S0, const iso_tensor* G_W, float* mU, float* vU,
                     float* mV, float* vV, const iso_tensor* W, const iso_tensor* W_out, int64_t m, int64_t n,
                     const iso_adamw_cfg* cfg, void* workspace, size_t ws_bytes, const iso_merge_stats* stats,
                     void* stream) {
    size_t need = 0;
    ISO_TRY(iso_opt_workspace_size(m, n, &need));
    if (!U || !V || !S0 || !G_W || !mU || !vU || !mV || !vV || !W || !W_out || !cfg) return ISO_ERR_ARG;
    auto al8 = [](const void* p) { return ((uintptr_t)p & 7u) == 0; };
    auto al4 = [](const void* p) { return ((uintptr_t)p & 3u) == 0; };
    if (!al8(U) || !al8(V) || !al8(S0) || !al4(mU) || !al4(vU) || !al4(mV) || !al4(vV)) return ISO_ERR_ALIGN;
    if (!(cfg->lr >= 0.0) || !std::isfinite(cfg->lr)) return ISO_ERR_ARG;
    if (!(cfg->beta1 >= 0.0 && cfg->beta1 < 1.0) || !(cfg->beta2 >= 0.0 && cfg->beta2 < 1.0)) return ISO_ERR_ARG;
    if (!(cfg->eps > 0.0) || !std::isfinite(cfg->eps)) return ISO_ERR_ARG;
    if (!(cfg->weight_decay >= 0.0) || !std::isfinite(cfg->weight_decay)) return ISO_ERR_ARG;
    if (cfg->step < 1 || cfg->ns_iters < 0 || cfg->ns_iters > FR_MAX_NS || cfg->reserved != 0) return ISO_ERR_ARG;
    for (const iso_tensor* t : {G_W, W, W_out}) {
        if (t->rows != m || t->cols != n) return ISO_ERR_SHAPE;
        if (t->dtype != ISO_BF16 && t->dtype != ISO_F32) return ISO_ERR_DTYPE;
        if (!t->data) return ISO_ERR_ARG;
        if ((uintptr_t)t->data & 15u) return ISO_ERR_ALIGN;
    }
    if (W_out->dtype != W->dtype) return ISO_ERR_DTYPE;
    {
        const size_t es = W->dtype == ISO_BF16 ? 2 : 4;
        const uintptr_t o0 = (uintptr_t)W_out->data, o1 = o0 + (uintptr_t)(m * n) * es, w0 = (uintptr_t)W->data;
        if (o0 != w0 && o0 < w0 + (uintptr_t)(m * n) * es && w0 < o1) return ISO_ERR_ARG;
    }
    if (!workspace || ((uintptr_t)workspace & 255u)) return ISO_ERR_WORKSPACE;
    if (ws_bytes < need) return ISO_ERR_WORKSPACE;
    const OptLayout L = opt_layout(m, n);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    char* ws = static_cast<char*>(workspace);
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return ISO_ERR_CUDA;
    const long long q = L.q, Qp = L.Qp;
    const int ns_iters = cfg->ns_iters ? cfg->ns_iters : FR_DEFAULT_NS;
    FrameHeader* hdr = reinterpret_cast<FrameHeader*>(ws + L.hdr);
    auto F = [&](size_t off) { return reinterpret_cast<float*>(ws + off); };
    auto D = [&](size_t off) { return reinterpret_cast<double*>(ws + off); };
    if (cudaMemsetAsync(ws + L.hdr, 0, sizeof(FrameHeader), s) != cudaSuccess) return ISO_ERR_CUDA;

    Frames fr[2];
    fr[0] = Frames{}; fr[0].F0 = U; fr[0].d = m; fr[0].q = q;
    fr[1] = Frames{}; fr[1].F0 = V; fr[1].d = n; fr[1].q = q;
    // operands of the factor gradients G_U = G_W (V S_0), G_V = G_W^T (U S_0)
    FR_LAUNCH((k_op_split_g<<<grid_of(L.Mp * L.Np, sms), 256, 0, s>>>(G_W->data, G_W->dtype, m, n, L.Mp, L.Np,
                                                                      F(L.gw4))));
    FR_LAUNCH((k_op_split_gt<<<dim3((unsigned)(L.Mp / 32), (unsigned)(L.Np / 32)), dim3(32, 8), 0, s>>>(
        G_W->data, G_W->dtype, m, n, L.Mp, L.Np, F(L.gwt4))));
    for (int sd = 0; sd < 2; ++sd) {
        SplitT st{};
        st.f = fr[sd]; st.X = sd == 0 ? U : V; st.S0 = S0; st.mode = 3; st.Dp = sd == 0 ? L.Mp : L.Np; st.Qp = Qp;
        st.out = F(sd == 0 ? L.su4 : L.sv4);
        FR_LAUNCH((k_fr_split_t<<<dim3((unsigned)(st.Dp / 32), (unsigned)(Qp / 32)), dim3(32, 8), 0, s>>>(st)));
    }
    // the factor gradients on the tensor cores with AdamW in the epilogue:
    // dF = F_bar - F, the moments updated in place
    const double bc1 = 1.0 - std::pow(cfg->beta1, (double)cfg->step);
    const double bc2 = 1.0 - std::pow(cfg->beta2, (double)cfg->step);
    for (int sd = 0; sd < 2; ++sd) {
        GemmArgs g{};
        g.mode = GEMM_ADAMW; g.M = (int)(sd == 0 ? m : n); g.N = (int)q; g.ldo = q; g.status = &hdr->status;
        g.adam = AdamwArgs{sd == 0 ? U : V, sd == 0 ? mU : mV, sd == 0 ? vU : vV, D(L.dF[sd]),
                           cfg->lr, cfg->beta1, cfg->beta2, cfg->eps, cfg->weight_decay, bc1, bc2};
        if (sd == 0) ISO_TRY(frame_gemm(s, F(L.gw4), L.Mp, F(L.sv4), Qp, L.Np, g));
        else ISO_TRY(frame_gemm(s, F(L.gwt4), L.Np, F(L.su4), Qp, L.Mp, g));
    }
    // the polar retraction of each side: N = (F + dF)^T (F + dF) - I in
    // binary64, R = (I + N)^(-1/2) - I, E_F = dF + (F + dF) R
    for (int sd = 0; sd < 2; ++sd) {
        const long long Dp = sd == 0 ? L.Mp : L.Np, d = fr[sd].d;
        const unsigned nt = (unsigned)((q + 63) / 64);
        FR_LAUNCH((k_op_gram64<<<nt * (nt + 1) / 2, 256, 0, s>>>(sd == 0 ? U : V, D(L.dF[sd]), d, q, D(L.n64))));
        NsBufs nb{D(L.ns_y), D(L.ns_z), D(L.ns_m), F(L.ns_y4), F(L.ns_z4), F(L.ns_m4), F(L.ns_t1),
                  F(L.ns_t2), F(L.ns_t3)};
        ISO_TRY(ns_root(s, sms, hdr, sd, nullptr, D(L.n64), q, Qp, nb, ns_iters, F(L.r4)));
        SplitR sr{};
        sr.f = fr[sd]; sr.X = D(L.dF[sd]); sr.mode = 1; sr.out = F(L.xb4); sr.rows = d; sr.rows_p = Dp; sr.Lp = Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Dp * Qp, sms), 256, 0, s>>>(sr)));
        {
            GemmArgs g{};
            g.mode = GEMM_STORE_F32; g.C = F(L.p); g.ldc = Qp; g.M = (int)Dp; g.N = (int)Qp; g.status = &hdr->status;
            ISO_TRY(frame_gemm(s, F(L.xb4), Dp, F(L.r4), Qp, Qp, g));
        }
        FR_LAUNCH((k_fr_motion<<<grid_of(d * q, sms), 256, 0, s>>>(D(L.dF[sd]), F(L.p), Qp, d, q)));
        // the reconstruction's operand of this side ([E_U S_0 | U S_0] or [V + E_V | E_V])
        sr.S0 = S0; sr.X = D(L.dF[sd]); sr.mode = sd == 0 ? 4 : 5; sr.out = F(sd == 0 ? L.a6 : L.b6);
        sr.rows = d; sr.rows_p = Dp; sr.Lp = 2 * Qp;
        FR_LAUNCH((k_fr_split_r<<<grid_of(Dp * 2 * Qp, sms), 256, 0, s>>>(sr)));
    }
    // F+ = F + E_F, then W+ = W + [E_U S_0 | U S_0] [V+ | E_V]^T
    FR_LAUNCH((k_op_add<<<grid_of(m * q, sms), 256, 0, s>>>(U, D(L.dF[0]), m * q)));
    FR_LAUNCH((k_op_add<<<grid_of(n * q, sms), 256, 0, s>>>(V, D(L.dF[1]), n * q)));
    {
        GemmArgs g{};
        g.mode = GEMM_ADD_BASE; g.M = (int)m; g.N = (int)n; g.out = W_out->data; g.w0 = W->data; g.ldo = n;
        g.out_dtype = W->dtype; g.status = &hdr->status;
        ISO_TRY(frame_gemm(s, F(L.a6), L.Mp, F(L.b6), L.Np, 2 * Qp, g));
    }
    if (stats && stats->status) FR_LAUNCH((k_fr_status<<<1, 32, 0, s>>>(hdr, stats->status)));
    return ISO_OK;
}

// The tcgen05 product on its own, for tests of the contraction: C (M x N,
// ldc) = A[:, a_k0 : a_k0 + Kc] B[:, b_k0 : b_k0 + Kc]^T with A (M x lda) and
// B (N x ldb) row-major binary32 read as tf32.
int32_t iso_gemm_tf32(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                      int64_t N, int64_t Kc, int64_t a_k0, int64_t b_k0, void* stream) {
    if (!A || !B || !C) return ISO_ERR_ARG;
    if (M <= 0 || N <= 0 || Kc <= 0 || a_k0 < 0 || b_k0 < 0) return ISO_ERR_ARG;
    if (M % GEMM_BM || N % GEMM_BN || Kc % GEMM_BK || a_k0 % GEMM_BK || b_k0 % GEMM_BK) return ISO_ERR_SHAPE;
    if (a_k0 + Kc > lda || b_k0 + Kc > ldb || ldc < N || lda % 4 || ldb % 4 || ldc % 4) return ISO_ERR_SHAPE;
    if (M >= (1LL << 31) || N >= (1LL << 31) || lda >= (1LL << 31) || ldb >= (1LL << 31)) return ISO_ERR_UNSUPPORTED;
    if (((uintptr_t)A & 15u) || ((uintptr_t)B & 15u) || ((uintptr_t)C & 15u)) return ISO_ERR_ALIGN;
    CUtensorMap ta, tb;
    ISO_TRY(gemm_tensor_map(&ta, A, M, lda, lda));
    ISO_TRY(gemm_tensor_map(&tb, B, N, ldb, ldb));
    ISO_TRY(gemm_smem_optin());
    GemmArgs g{};
    g.mode = GEMM_STORE_F32; g.C = C; g.ldc = ldc; g.M = (int)M; g.N = (int)N;
    g.k_tiles = (int)(Kc / GEMM_BK); g.a_k0 = (int)a_k0; g.b_k0 = (int)b_k0;
    const int slot = prof_begin(0, static_cast<cudaStream_t>(stream));
    k_gemm_tf32<<<dim3((unsigned)(N / GEMM_BN), (unsigned)(M / GEMM_BM)), GEMM_THREADS, GEMM_SMEM,
                  static_cast<cudaStream_t>(stream)>>>(ta, tb, g);
    prof_end(slot, static_cast<cudaStream_t>(stream));
    return cudaGetLastError() == cudaSuccess ? ISO_OK : ISO_ERR_CUDA;
}

}  // extern "C"
