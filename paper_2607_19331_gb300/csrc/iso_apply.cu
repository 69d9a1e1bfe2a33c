// iso_apply.cu -- the streaming passes that apply a resolved TopKMask.
//
//   k_apply  out = theta_0 + update, one read of theta_0 and the K experts
//            and one write:                                         (App. F)
//              TA    update = lambda * sum_i tau_i
//              TIES  gamma = sign(sum_i m_i tau_i); A = {i : m_i tau_i != 0,
//                    sign = gamma}; update = lambda * mean_{i in A} tau_i
//              ISO   2-D: update = sum_i c_i m_i tau_i          (Sec. 4.2, App. E)
//                    1-D: update = (1/K) sum_i tau_i            (App. E, Algorithm 1)
//            An update of exactly zero leaves theta_0 untouched.
//   k_gram   Gamma_ij = <m_i tau_i, m_j tau_j> per 2-D tensor  (Sec. 4.2 Gram eq.)
//   k_solve  (Gamma + ridge I) c = diag Gamma on the non-zero experts, clip
//   k_mask   the mask itself as a packed bitmask
//   k_delta  tau = theta_i - theta_0 in binary32
//
// Arithmetic: binary32 with explicit round-to-nearest intrinsics (no
// contraction), experts summed in the fixed order i = 1..K.
#include "iso_kernels.cuh"

namespace iso {

// ---------------------------------------------------------------------------
// vector load / store with a ragged tail
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ void load8_tail(const void* p, long long e, long long n, float (&v)[8]) {
    if (e + 8 <= n) {
        Load8<T>::run(p, e, v);
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = (e + j < n) ? Load8<T>::one(p, e + j) : 0.0f;
    }
}

template <typename T> struct Store8;
template <> struct Store8<__nv_bfloat16> {
    static __device__ __forceinline__ void run(void* p, long long e, long long n, const float (&v)[8]) {
        __nv_bfloat16* q = static_cast<__nv_bfloat16*>(p) + e;
        if (e + 8 <= n) {
            uint4 u;
            __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]);
            __nv_bfloat162 b = __floats2bfloat162_rn(v[2], v[3]);
            __nv_bfloat162 c = __floats2bfloat162_rn(v[4], v[5]);
            __nv_bfloat162 d = __floats2bfloat162_rn(v[6], v[7]);
            u.x = *reinterpret_cast<uint32_t*>(&a);
            u.y = *reinterpret_cast<uint32_t*>(&b);
            u.z = *reinterpret_cast<uint32_t*>(&c);
            u.w = *reinterpret_cast<uint32_t*>(&d);
            *reinterpret_cast<uint4*>(q) = u;
        } else {
            for (int j = 0; j < 8; ++j)
                if (e + j < n) q[j] = __float2bfloat16_rn(v[j]);
        }
    }
};
template <> struct Store8<float> {
    static __device__ __forceinline__ void run(void* p, long long e, long long n, const float (&v)[8]) {
        float* q = static_cast<float*>(p) + e;
        if (e + 8 <= n) {
            reinterpret_cast<float4*>(q)[0] = make_float4(v[0], v[1], v[2], v[3]);
            reinterpret_cast<float4*>(q)[1] = make_float4(v[4], v[5], v[6], v[7]);
        } else {
            for (int j = 0; j < 8; ++j)
                if (e + j < n) q[j] = v[j];
        }
    }
};

// ---------------------------------------------------------------------------
// per-entry selection
// ---------------------------------------------------------------------------
struct SelParam { uint32_t t; long long cut; };

__device__ __forceinline__ bool kept(uint32_t key, long long pos, const SelParam& s) {
    return key > s.t || (key == s.t && pos < s.cut);
}

// BLOCK scope: unit of entry e of tensor d
__device__ __forceinline__ int block_unit(const Plan& P, const TensorDesc& d, long long row, long long col) {
    return d.unit + (int)(row / P.block_rows) * d.bpr + (int)(col / P.block_cols);
}

__device__ __forceinline__ int sgn(float v) { return (v > 0.0f) - (v < 0.0f); }

// ---------------------------------------------------------------------------
// apply
// ---------------------------------------------------------------------------
template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB) k_apply(Plan P) {
    const int K = KC ? KC : P.K;
    for (long long g = blockIdx.x; g < P.n_tiles; g += gridDim.x) {
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const bool is1d = (d.flags & TF_1D) != 0;
        const bool iso2d = (P.op == ISO_OP_ISO) && !is1d;
        const bool iso1d = (P.op == ISO_OP_ISO) && is1d;
        const bool blk = (P.scope == ISO_SCOPE_BLOCK) && (d.flags & TF_TRIM);
        const long long pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
        SelParam sp[KC ? KC : MAXK];
        float cf[KC ? KC : MAXK];
        const void* xs[KC ? KC : MAXK];
#pragma unroll
        for (int i = 0; i < (KC ? KC : MAXK); ++i) {
            if (i >= K) break;
            xs[i] = P.xptr[i * P.n_tensors + t];
            cf[i] = iso2d ? (float)P.coef[(long long)t * K + i] : 0.0f;
            if (!blk) {
                const Unit& U = P.units[(long long)i * P.n_units + ((P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit)];
                sp[i].t = U.t;
                sp[i].cut = U.cut;
            }
        }
        for (int v = 0; v < NVEC; ++v) {
            const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
            if (e >= n) continue;
            float th0[VEC];
            load8_tail<BT>(d.base, e, n, th0);
            float acc0[VEC], acc1[VEC];   // TA / ISO: running sums; TIES: election sum
#pragma unroll
            for (int j = 0; j < VEC; ++j) { acc0[j] = 0.0f; acc1[j] = 0.0f; }
            float tau[KC ? KC : MAXK][VEC];
            bool sel[KC ? KC : MAXK][VEC];
            long long row = 0, col = 0;
            if (blk) { row = e / d.cols; col = e - row * d.cols; }
#pragma unroll
            for (int i = 0; i < (KC ? KC : MAXK); ++i) {
                if (i >= K) break;
                TauSrc<XT, BT, CK>::load8(xs[i], d.base, e, n, tau[i]);
                long long r = row, c = col;
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    SelParam s;
                    if (blk) {
                        const Unit& U = P.units[(long long)i * P.n_units + block_unit(P, d, r, c)];
                        s.t = U.t;
                        s.cut = U.cut;
                        if (++c == d.cols) { c = 0; ++r; }
                    } else {
                        s = sp[i];
                    }
                    sel[i][j] = kept(key_of(tau[i][j]), pos_off + e + j, s);
                }
            }
            float o[VEC];
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                float upd;
                if (P.op == ISO_OP_TA || iso1d) {
                    float s = 0.0f;
#pragma unroll
                    for (int i = 0; i < (KC ? KC : MAXK); ++i) {
                        if (i >= K) break;
                        s = __fadd_rn(s, tau[i][j]);
                    }
                    upd = iso1d ? __fdiv_rn(s, (float)K) : __fmul_rn(P.lambda, s);
                } else if (P.op == ISO_OP_TIES) {
                    float s = 0.0f;
#pragma unroll
                    for (int i = 0; i < (KC ? KC : MAXK); ++i) {
                        if (i >= K) break;
                        s = __fadd_rn(s, sel[i][j] ? tau[i][j] : 0.0f);
                    }
                    const int gam = sgn(s);
                    float a = 0.0f;
                    int cnt = 0;
#pragma unroll
                    for (int i = 0; i < (KC ? KC : MAXK); ++i) {
                        if (i >= K) break;
                        const float x = tau[i][j];
                        if (sel[i][j] && x != 0.0f && sgn(x) == gam) { a = __fadd_rn(a, x); cnt++; }
                    }
                    const float merged = cnt ? __fdiv_rn(a, (float)cnt) : 0.0f;
                    upd = __fmul_rn(P.lambda, merged);
                } else {
                    float s = 0.0f;
#pragma unroll
                    for (int i = 0; i < (KC ? KC : MAXK); ++i) {
                        if (i >= K) break;
                        if (sel[i][j]) s = __fadd_rn(s, __fmul_rn(cf[i], tau[i][j]));
                    }
                    upd = s;
                }
                o[j] = (upd == 0.0f) ? th0[j] : __fadd_rn(th0[j], upd);
            }
            Store8<BT>::run(d.out, e, n, o);
        }
    }
}

// ---------------------------------------------------------------------------
// Gram of the trimmed task vectors (per 2-D tensor, upper triangle)
// ---------------------------------------------------------------------------
template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(TPB) k_gram(Plan P) {
    constexpr int NP = MAXK * (MAXK + 1) / 2;
    __shared__ double s_g[NP];
    const int K = P.K;
    const int np = K * (K + 1) / 2;
    const long long per = (P.n_tiles + gridDim.x - 1) / gridDim.x;
    const long long g0 = blockIdx.x * per;
    const long long g1 = (g0 + per < P.n_tiles) ? g0 + per : P.n_tiles;
    for (int q = threadIdx.x; q < NP; q += blockDim.x) s_g[q] = 0.0;
    __syncthreads();
    int cur = -1;
    for (long long g = g0; g < g1; ++g) {
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        if ((d.flags & TF_1D) || !(d.flags & TF_TRIM)) continue;
        if (t != cur) {
            __syncthreads();
            if (cur >= 0)
                for (int q = threadIdx.x; q < np; q += blockDim.x) {
                    if (s_g[q] != 0.0) {
                        int a = 0, b = q;   // q -> (a, b) in the upper triangle, row-major
                        while (b >= K - a) { b -= K - a; ++a; }
                        atomicAdd(&P.gram[((long long)cur * K + a) * K + a + b], s_g[q]);
                    }
                    s_g[q] = 0.0;
                }
            __syncthreads();
            cur = t;
        }
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const bool blk = (P.scope == ISO_SCOPE_BLOCK);
        const long long pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
        float acc[NP];
#pragma unroll
        for (int q = 0; q < NP; ++q) acc[q] = 0.0f;
        for (int v = 0; v < NVEC; ++v) {
            const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
            if (e >= n) continue;
            float m[MAXK][VEC];
            long long row = 0, col = 0;
            if (blk) { row = e / d.cols; col = e - row * d.cols; }
#pragma unroll
            for (int i = 0; i < MAXK; ++i) {
                if (i >= K) break;
                float tau[VEC];
                TauSrc<XT, BT, CK>::load8(P.xptr[i * P.n_tensors + t], d.base, e, n, tau);
                SelParam s;
                if (!blk) {
                    const Unit& U = P.units[(long long)i * P.n_units + ((P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit)];
                    s.t = U.t; s.cut = U.cut;
                }
                long long r = row, c = col;
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    if (blk) {
                        const Unit& U = P.units[(long long)i * P.n_units + block_unit(P, d, r, c)];
                        s.t = U.t; s.cut = U.cut;
                        if (++c == d.cols) { c = 0; ++r; }
                    }
                    m[i][j] = kept(key_of(tau[j]), pos_off + e + j, s) ? tau[j] : 0.0f;
                }
            }
            int q = 0;
#pragma unroll
            for (int a = 0; a < MAXK; ++a) {
#pragma unroll
                for (int b = a; b < MAXK; ++b) {
                    if (a < K && b < K) {
#pragma unroll
                        for (int j = 0; j < VEC; ++j) acc[q] = __fadd_rn(acc[q], __fmul_rn(m[a][j], m[b][j]));
                    }
                    ++q;
                }
            }
        }
        // warp partials in binary32 (<= 1024 entries), then binary64 in shared memory
        const int lane = threadIdx.x & 31;
        int q = 0;
#pragma unroll
        for (int a = 0; a < MAXK; ++a) {
#pragma unroll
            for (int b = a; b < MAXK; ++b) {
                if (a < K && b < K) {
                    const float w = warp_sum(acc[q]);
                    if (lane == 0 && w != 0.0f) {
                        // compact index over the K x K upper triangle
                        const int cq = a * K - a * (a - 1) / 2 + (b - a);
                        atomicAdd(&s_g[cq], (double)w);
                    }
                }
                ++q;
            }
        }
    }
    __syncthreads();
    if (cur >= 0)
        for (int q = threadIdx.x; q < np; q += blockDim.x) {
            if (s_g[q] != 0.0) {
                int a = 0, b = q;
                while (b >= K - a) { b -= K - a; ++a; }
                atomicAdd(&P.gram[((long long)cur * K + a) * K + a + b], s_g[q]);
            }
        }
}

// ---------------------------------------------------------------------------
// retention coefficients: one thread per tensor
// ---------------------------------------------------------------------------
__global__ void k_solve(Plan P, int gram_mode) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= P.n_tensors) return;
    const int K = P.K;
    const TensorDesc& d = P.tens[t];
    double G[MAXK * MAXK];
    double c[MAXK];
    for (int q = 0; q < K * K; ++q) G[q] = 0.0;
    for (int i = 0; i < K; ++i) c[i] = 0.0;
    const bool active = (P.op == ISO_OP_ISO) && !(d.flags & TF_1D) && (d.flags & TF_TRIM);
    if (active) {
        if (gram_mode == GRAM_UNIT) {
            G[0] = P.units[d.unit].gamma;           // K == 1, TENSOR scope
        } else {
            for (int a = 0; a < K; ++a)
                for (int b = a; b < K; ++b) {
                    const double v = P.gram[((long long)t * K + a) * K + b];
                    G[a * K + b] = v;
                    G[b * K + a] = v;
                }
        }
        // I = {i : Gamma_ii > 0}; (Gamma_II + ridge I) c_I = diag(Gamma)_I; clip
        int idx[MAXK];
        int m = 0;
        for (int i = 0; i < K; ++i)
            if (G[i * K + i] > 0.0) idx[m++] = i;
        double A[MAXK * MAXK], rhs[MAXK], x[MAXK];
        for (int r = 0; r < m; ++r) {
            for (int q = 0; q < m; ++q) A[r * m + q] = G[idx[r] * K + idx[q]];
            A[r * m + r] = __dadd_rn(A[r * m + r], P.ridge);
            rhs[r] = G[idx[r] * K + idx[r]];
        }
        // Gaussian elimination with partial pivoting
        for (int col = 0; col < m; ++col) {
            int piv = col;
            for (int r = col + 1; r < m; ++r)
                if (fabs(A[r * m + col]) > fabs(A[piv * m + col])) piv = r;
            if (piv != col) {
                for (int q = 0; q < m; ++q) { double s = A[col * m + q]; A[col * m + q] = A[piv * m + q]; A[piv * m + q] = s; }
                double s = rhs[col]; rhs[col] = rhs[piv]; rhs[piv] = s;
            }
            for (int r = col + 1; r < m; ++r) {
                const double f = A[r * m + col] / A[col * m + col];
                for (int q = col; q < m; ++q) A[r * m + q] = __dadd_rn(A[r * m + q], -__dmul_rn(f, A[col * m + q]));
                rhs[r] = __dadd_rn(rhs[r], -__dmul_rn(f, rhs[col]));
            }
        }
        for (int r = m - 1; r >= 0; --r) {
            double s = rhs[r];
            for (int q = r + 1; q < m; ++q) s = __dadd_rn(s, -__dmul_rn(A[r * m + q], x[q]));
            x[r] = s / A[r * m + r];
        }
        for (int r = 0; r < m; ++r) {
            double v = x[r];
            if (v < P.c_min) v = P.c_min;
            if (v > P.c_max) v = P.c_max;
            c[idx[r]] = v;
        }
    }
    for (int i = 0; i < K; ++i) P.coef[(long long)t * K + i] = c[i];
    const long long tg = P.st_tensor_base + t;
    if (P.st_gram)
        for (int q = 0; q < K * K; ++q) P.st_gram[tg * K * K + q] = G[q];
    if (P.st_coef)
        for (int i = 0; i < K; ++i) P.st_coef[tg * K + i] = c[i];
}

// ---------------------------------------------------------------------------
// packed mask: bit j of word w is entry 32 w + j
// ---------------------------------------------------------------------------
template <typename XT>
__global__ void __launch_bounds__(TPB) k_mask(Plan P, uint32_t* const* mptr) {
    for (long long g = blockIdx.x; g < P.n_tiles; g += gridDim.x) {
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        uint32_t* mw = mptr[t];
        if (!mw) continue;
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const bool blk = (P.scope == ISO_SCOPE_BLOCK);
        const long long pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
        SelParam s0;
        if (!blk) {
            const Unit& U = P.units[(P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit];
            s0.t = U.t; s0.cut = U.cut;
        }
        for (int v = 0; v < NVEC; ++v) {
            const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
            uint32_t bits = 0;
            if (e < n) {
                float tau[VEC];
                TauSrc<XT, XT, false>::load8(P.xptr[t], nullptr, e, n, tau);
                long long r = 0, c = 0;
                if (blk) { r = e / d.cols; c = e - r * d.cols; }
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    if (e + j >= n) break;
                    SelParam s = s0;
                    if (blk) {
                        const Unit& U = P.units[block_unit(P, d, r, c)];
                        s.t = U.t; s.cut = U.cut;
                        if (++c == d.cols) { c = 0; ++r; }
                    }
                    if (kept(key_of(tau[j]), pos_off + e + j, s)) bits |= 1u << j;
                }
            }
            // four consecutive threads hold 32 consecutive entries
            const int sub = threadIdx.x & 3;
            uint32_t w = bits << (8 * sub);
            w |= __shfl_xor_sync(0xFFFFFFFFu, w, 1);
            w |= __shfl_xor_sync(0xFFFFFFFFu, w, 2);
            if (sub == 0 && e < n) mw[e >> 5] = w;
        }
    }
}

__global__ void k_status(const Header* h, int32_t* out) {
    if (threadIdx.x == 0 && blockIdx.x == 0) *out = h->status;
}

__global__ void k_upload(UploadChunk c) {
    uint4* dst = reinterpret_cast<uint4*>(c.dst);
    for (uint32_t q = threadIdx.x; q < c.nbytes / 16; q += blockDim.x) dst[q] = c.data[q];
}

// ---------------------------------------------------------------------------
// tau = theta_i - theta_0
// ---------------------------------------------------------------------------
template <typename AT, typename BT>
__global__ void __launch_bounds__(TPB) k_delta(DeltaArgs A) {
    const long long n_tiles = A.tile_base[A.n];
    for (long long g = blockIdx.x; g < n_tiles; g += gridDim.x) {
        int t = 0;
        while (t + 1 < A.n && A.tile_base[t + 1] <= g) ++t;
        const long long n = A.numel[t];
        const long long e0 = (g - A.tile_base[t]) * TILE;
#pragma unroll
        for (int v = 0; v < NVEC; ++v) {
            const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
            if (e >= n) continue;
            float a[VEC], b[VEC], o[VEC];
            load8_tail<AT>(A.a[t], e, n, a);
            load8_tail<BT>(A.b[t], e, n, b);
#pragma unroll
            for (int j = 0; j < VEC; ++j) o[j] = __fsub_rn(a[j], b[j]);
            Store8<float>::run(A.out[t], e, n, o);
        }
    }
}

// ---------------------------------------------------------------------------
// instantiations
// ---------------------------------------------------------------------------
#define ISO_APPLY_INST(XT, BT, CK)                                             \
    template __global__ void k_apply<XT, BT, CK, 1>(Plan);                    \
    template __global__ void k_apply<XT, BT, CK, 0>(Plan);                    \
    template __global__ void k_gram<XT, BT, CK>(Plan);

ISO_APPLY_INST(__nv_bfloat16, __nv_bfloat16, false)
ISO_APPLY_INST(__nv_bfloat16, float, false)
ISO_APPLY_INST(float, __nv_bfloat16, false)
ISO_APPLY_INST(float, float, false)
ISO_APPLY_INST(__nv_bfloat16, __nv_bfloat16, true)
ISO_APPLY_INST(__nv_bfloat16, float, true)
ISO_APPLY_INST(float, __nv_bfloat16, true)
ISO_APPLY_INST(float, float, true)

template __global__ void k_mask<__nv_bfloat16>(Plan, uint32_t* const*);
template __global__ void k_mask<float>(Plan, uint32_t* const*);
template __global__ void k_delta<__nv_bfloat16, __nv_bfloat16>(DeltaArgs);
template __global__ void k_delta<__nv_bfloat16, float>(DeltaArgs);
template __global__ void k_delta<float, __nv_bfloat16>(DeltaArgs);
template __global__ void k_delta<float, float>(DeltaArgs);

}  // namespace iso
