// iso_merge.cu -- the streaming passes of a merge of K >= 2 experts, and the
// Gram pass of the ISO retention rule for any K.
//
//   k_merge   out = theta_0 + update from the K masked task vectors   (App. F)
//               TA    update = lambda * sum_i tau_i
//               TIES  gamma = sign(sum_i m_i tau_i); A = {i : m_i tau_i != 0,
//                     sign(tau_i) = gamma}; update = lambda * mean_{i in A} tau_i
//               ISO   2-D: update = sum_i c_i m_i tau_i           (Sec. 4.2, App. E)
//                     1-D: update = (1/K) sum_i tau_i             (App. E, Algorithm 1)
//             An update of exactly zero leaves theta_0 untouched.
//   k_gramk   Gamma_ab = <m_a tau_a, m_b tau_b> per trimmed 2-D tensor   (Sec. 4.2)
//
// Both read theta_0 and the K experts once, streaming: each lane takes one
// 16-byte vector of every expert per step (4 fp32 or 8 bf16 entries), a warp
// 512 contiguous bytes of each, and the K loads of U steps are issued before
// any of them is used.  The expert count is a compile-time bound KC (2, 4 or
// 8; the call's K <= KC), so every per-expert array is a register array and
// all loops over experts unroll; experts K..KC-1 are predicated off.
//
// Arithmetic: binary32, experts taken in the fixed order i = 1..K; the merge
// uses explicit round-to-nearest operations (no contraction) so that every
// output is the one the sequential definition gives.
#include "iso_kernels.cuh"

namespace iso {

namespace {

// raw words of E consecutive entries of T (E * sizeof(T) is 8, 16 or 32 bytes)
template <typename T, int E>
struct Words {
    static constexpr int N = E * (int)sizeof(T) / 4;
    uint32_t w[N];
};

__device__ __forceinline__ uint2 ld_stream2(const void* p) {
    uint2 r;
    asm("ld.global.nc.L1::no_allocate.L2::256B.v2.u32 {%0, %1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(p));
    return r;
}

// entries [e, e + E) of p (e a multiple of E); entries at or past n read as 0
template <typename T, int E>
__device__ __forceinline__ void load_words(const void* p, long long e, long long n, Words<T, E>& r) {
    constexpr int N = Words<T, E>::N;
    const char* a = static_cast<const char*>(p) + e * (long long)sizeof(T);
    if (e + E <= n) {
        if (N == 2) {
            const uint2 v = ld_stream2(a);
            r.w[0] = v.x; r.w[1] = v.y;
        } else {
#pragma unroll
            for (int q = 0; q < N / 4; ++q) {
                const uint4 v = ld_stream(a + 16 * q);
                r.w[4 * q] = v.x; r.w[4 * q + 1] = v.y; r.w[4 * q + 2] = v.z; r.w[4 * q + 3] = v.w;
            }
        }
    } else {
#pragma unroll
        for (int q = 0; q < N; ++q) r.w[q] = 0;
        if (sizeof(T) == 2) {
            const unsigned short* s = static_cast<const unsigned short*>(p);
#pragma unroll
            for (int j = 0; j < E; ++j)
                if (e + j < n) r.w[j >> 1] |= (uint32_t)s[e + j] << (16 * (j & 1));
        } else {
            const uint32_t* s = static_cast<const uint32_t*>(p);
#pragma unroll
            for (int j = 0; j < E; ++j)
                if (e + j < n) r.w[j] = s[e + j];
        }
    }
}

template <typename T, int E>
__device__ __forceinline__ float word_f32(const Words<T, E>& r, int j) {
    if (sizeof(T) == 2)
        return __uint_as_float((j & 1) ? (r.w[j >> 1] & 0xFFFF0000u) : (r.w[j >> 1] << 16));
    return __uint_as_float(r.w[j]);
}

// E outputs of type T at [e, e + E), rounded to nearest even for bf16
template <typename T, int E>
__device__ __forceinline__ void store_out(void* p, long long e, long long n, const float (&v)[E]) {
    constexpr int N = Words<T, E>::N;
    uint32_t w[N];
    if (sizeof(T) == 2) {
#pragma unroll
        for (int q = 0; q < N; ++q) {
            __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * q], v[2 * q + 1]);
            w[q] = *reinterpret_cast<uint32_t*>(&h);
        }
    } else {
#pragma unroll
        for (int q = 0; q < N; ++q) w[q] = __float_as_uint(v[q]);
    }
    char* a = static_cast<char*>(p) + e * (long long)sizeof(T);
    if (e + E <= n) {
        if (N == 2) {
            __stcs(reinterpret_cast<uint2*>(a), make_uint2(w[0], w[1]));
        } else {
#pragma unroll
            for (int q = 0; q < N / 4; ++q)
                __stcs(reinterpret_cast<uint4*>(a) + q, make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]));
        }
    } else if (sizeof(T) == 2) {
        unsigned short* s = reinterpret_cast<unsigned short*>(a);
#pragma unroll
        for (int j = 0; j < E; ++j)
            if (e + j < n) s[j] = (unsigned short)(w[j >> 1] >> (16 * (j & 1)));
    } else {
        uint32_t* s = reinterpret_cast<uint32_t*>(a);
#pragma unroll
        for (int j = 0; j < E; ++j)
            if (e + j < n) s[j] = w[j];
    }
}

// how the entries of one tensor are tested against their units' thresholds
enum SelMode : int {
    SEL_ALL = 0,      // no mask (TA, ISO 1-D)
    SEL_PACKED = 1,   // one unit per tensor and expert: (key, ~pos) > (t, ~cut)
    SEL_BLOCK = 2,    // BLOCK scope: the unit of each entry's block
};

enum OpKind : int { OPK_SUM = 0, OPK_TIES = 1, OPK_ISO = 2 };

template <int KC>
struct MergeParams {
    const void* xs[KC];
    unsigned long long thr[KC];   // SEL_PACKED, tensor-local positions
    float cf[KC];                 // ISO 2-D coefficients
    int sel, opk;
    bool iso1d, trimmed2d;
};

// the warp's copy of one tensor's parameters lives in shared memory (written
// by lane 0), which keeps the registers for the data in flight
template <int KC>
__device__ __forceinline__ void merge_params(const Plan& P, int t, int K, MergeParams<KC>& mp) {
    __syncwarp();
    if ((threadIdx.x & 31) != 0) { __syncwarp(); return; }
    const TensorDesc& d = P.tens[t];
    const bool is1d = (d.flags & TF_1D) != 0;
    const bool trim = (d.flags & TF_TRIM) != 0;
    mp.iso1d = (P.op == ISO_OP_ISO) && is1d;
    mp.trimmed2d = trim && !is1d;
    mp.opk = (P.op == ISO_OP_TA || mp.iso1d) ? OPK_SUM : (P.op == ISO_OP_TIES ? OPK_TIES : OPK_ISO);
    if (mp.opk == OPK_SUM) mp.sel = SEL_ALL;
    else if (trim && P.scope == ISO_SCOPE_BLOCK) mp.sel = SEL_BLOCK;
    else mp.sel = SEL_PACKED;
    // GLOBAL scope: the unit's cut is a position in the concatenation; entry
    // e of this tensor sits at uoff + e, so the tensor-local cut is cut - uoff
    // clamped to [0, 2^32 - 1] (numel < 2^32 keeps every local position below)
    const long long pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
#pragma unroll
    for (int i = 0; i < KC; ++i) {
        mp.xs[i] = (i < K) ? P.xptr[i * P.n_tensors + t] : nullptr;
        mp.cf[i] = (i < K && mp.opk == OPK_ISO) ? (float)P.coef[(long long)t * K + i] : 0.0f;
        uint32_t tk = 0;
        long long cut = CUT_ALL;
        if (i < K && trim && mp.sel != SEL_BLOCK) {
            const Unit& U = P.units[(long long)i * P.n_units + ((P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit)];
            tk = U.t;
            cut = U.cut;
        }
        const long long lc = (cut == CUT_ALL) ? cut : cut - pos_off;
        const uint32_t c32 = (lc >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (lc <= 0 ? 0u : (uint32_t)lc);
        mp.thr[i] = ((unsigned long long)tk << 32) | (uint32_t)~c32;
    }
    __syncwarp();
}

__device__ __forceinline__ int sgnf(float v) { return (v > 0.0f) - (v < 0.0f); }

// selection bits of the K experts at entry e (tensor-local), bit i for expert i
template <int KC>
__device__ __forceinline__ uint32_t select_bits(const Plan& P, const TensorDesc& d, const MergeParams<KC>& mp,
                                                int K, const float (&tau)[KC], long long e, long long& r,
                                                long long& c) {
    uint32_t bits = 0;
    if (mp.sel == SEL_ALL) return (1u << KC) - 1u;
    if (mp.sel == SEL_PACKED) {
        const uint32_t np = ~(uint32_t)e;
#pragma unroll
        for (int i = 0; i < KC; ++i) {
            const unsigned long long kp = ((unsigned long long)key_of(tau[i]) << 32) | np;
            if (i < K && kp > mp.thr[i]) bits |= 1u << i;
        }
    } else {
        const int u = d.unit + (int)(r / P.block_rows) * d.bpr + (int)(c / P.block_cols);
#pragma unroll
        for (int i = 0; i < KC; ++i) {
            if (i < K) {
                const Unit& U = P.units[(long long)i * P.n_units + u];
                SelParam s;
                s.t = U.t;
                s.cut = U.cut;
                if (kept(key_of(tau[i]), e, s)) bits |= 1u << i;
            }
        }
        if (++c == d.cols) { c = 0; ++r; }
    }
    return bits;
}

// the merged output of one entry; every argument is in registers
template <int KC>
__device__ __forceinline__ float merged_value(int opk, bool iso1d, float lambda, int K, float th0,
                                              const float (&tau)[KC], const float (&cf)[KC], uint32_t bits) {
    float upd;
    if (opk == OPK_SUM) {
        float s = 0.0f;
#pragma unroll
        for (int i = 0; i < KC; ++i)
            if (i < K) s = __fadd_rn(s, tau[i]);
        upd = iso1d ? __fdiv_rn(s, (float)K) : __fmul_rn(lambda, s);
    } else if (opk == OPK_TIES) {
        // gamma = sign(sum of the trimmed values); the agreeing set holds the
        // non-zero trimmed values of that sign (none when the sum is 0)
        float tt[KC];
        float s = 0.0f;
#pragma unroll
        for (int i = 0; i < KC; ++i) {
            tt[i] = (i < K && ((bits >> i) & 1u)) ? tau[i] : 0.0f;
            if (i < K) s = __fadd_rn(s, tt[i]);
        }
        const uint32_t sbit = __float_as_uint(s) & 0x80000000u;
        float a = 0.0f;
        int cnt = 0;
#pragma unroll
        for (int i = 0; i < KC; ++i) {
            const bool agree = (i < K) && (tt[i] != 0.0f) && ((__float_as_uint(tt[i]) & 0x80000000u) == sbit);
            a = agree ? __fadd_rn(a, tt[i]) : a;
            cnt += agree;
        }
        if (s == 0.0f) cnt = 0;
        const float m = cnt ? __fdiv_rn(a, (float)cnt) : 0.0f;
        upd = __fmul_rn(lambda, m);
    } else {
        float s = 0.0f;
#pragma unroll
        for (int i = 0; i < KC; ++i)
            if (i < K && ((bits >> i) & 1u)) s = __fadd_rn(s, __fmul_rn(cf[i], tau[i]));
        upd = s;
    }
    return (upd == 0.0f) ? th0 : __fadd_rn(th0, upd);
}

// Per-tile thresholds.  Inside a tile that lies wholly before (after) a unit's
// cut, an entry with key == t is kept (dropped), so the selection is the
// single comparison  (int)key > T  with T = t - 1 (T = t); keys are below 2^31.
// A tile holding the cut, and BLOCK scope, take the exact per-entry test.
template <int KC>
__device__ __forceinline__ bool tile_thresholds(const MergeParams<KC>& mp, int K, uint32_t e0, uint32_t e1,
                                                int (&T)[KC]) {
    bool exact = (mp.sel == SEL_BLOCK);
#pragma unroll
    for (int i = 0; i < KC; ++i) {
        T[i] = -1;
        if (i < K && mp.sel == SEL_PACKED) {
            const unsigned long long th = mp.thr[i];
            const uint32_t tk = (uint32_t)(th >> 32), c32 = ~(uint32_t)th;
            if (tk > 0x7FFFFFFEu) T[i] = 0x7FFFFFFF;          // nothing is kept
            else if (e1 <= c32) T[i] = (int)tk - 1;            // ties kept
            else if (e0 >= c32) T[i] = (int)tk;                // ties dropped
            else exact = true;
        }
    }
    return exact;
}

template <int KC>
__device__ __forceinline__ uint32_t fast_bits(const int (&T)[KC], int K, const float (&tau)[KC]) {
    uint32_t bits = 0;
#pragma unroll
    for (int i = 0; i < KC; ++i)
        if (i < K && (int)key_of(tau[i]) > T[i]) bits |= 1u << i;
    return bits;
}

// the warp's contiguous tile range
struct WarpRange { long long beg, end; };
__device__ __forceinline__ WarpRange warp_range(const Plan& P) {
    const long long W = (long long)gridDim.x * WPB;
    const long long wid = (long long)blockIdx.x * WPB + (threadIdx.x >> 5);
    const long long per = (P.n_tiles + W - 1) / W;
    WarpRange r;
    r.beg = wid * per;
    r.end = (r.beg + per < P.n_tiles) ? r.beg + per : P.n_tiles;
    return r;
}

__device__ __forceinline__ long long tensor_tile_end(const Plan& P, int t) {
    return P.tens[t].tile_base + (P.tens[t].numel + TILE - 1) / TILE;
}

}  // namespace

// One warp per tile, a contiguous tile range per warp.  Each lane takes one
// 16-byte vector of every expert per step (4 fp32 or 8 bf16 entries); up to
// four experts, the next step's loads are issued before the current step is
// merged.
template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB, MERGE_BLOCKS_PER_SM) k_merge(Plan P) {
    constexpr int E = 16 / (int)sizeof(XT);          // entries per lane per step
    constexpr int SPT = TILE / (32 * E);             // steps per tile (4 or 8)
    static_assert(SPT % 2 == 0, "steps alternate between two buffers");
    const int K = P.K;
    const int lane = threadIdx.x & 31;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    int t = tensor_of_tile(P.tens, P.n_tensors, wr.beg);
    long long t_end = tensor_tile_end(P, t);
    __shared__ MergeParams<KC> s_mp[WPB];
    MergeParams<KC>& mp = s_mp[threadIdx.x >> 5];
    merge_params<KC>(P, t, K, mp);
    for (long long g = wr.beg; g < wr.end; ++g) {
        if (g >= t_end) {
            while (g >= t_end) t_end = tensor_tile_end(P, ++t);
            merge_params<KC>(P, t, K, mp);
        }
        const TensorDesc& d = P.tens[t];
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
        // this tile's parameters, in registers
        const void* xs[KC];
        float cf[KC];
        int T[KC];
#pragma unroll
        for (int i = 0; i < KC; ++i) { xs[i] = mp.xs[i]; cf[i] = mp.cf[i]; }
        const bool exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
        const int opk = mp.opk;
        const bool iso1d = mp.iso1d;
        const void* bp = d.base;
        void* op = d.out;

        Words<XT, E> xa[KC], xb[KC];
        Words<BT, E> ba, bb;
        auto load = [&](int st, Words<XT, E> (&x)[KC], Words<BT, E>& b) {
            const long long e = e0 + (long long)st * (32 * E) + lane * E;
            if (e < n) {
                load_words<BT, E>(bp, e, n, b);
#pragma unroll
                for (int i = 0; i < KC; ++i)
                    if (i < K) load_words<XT, E>(xs[i], e, n, x[i]);
            }
        };
        auto merge_step = [&](int st, const Words<XT, E> (&x)[KC], const Words<BT, E>& b) {
            const long long e = e0 + (long long)st * (32 * E) + lane * E;
            if (e >= n) return;
            long long r = 0, c = 0;
            if (exact && mp.sel == SEL_BLOCK) { r = e / d.cols; c = e - r * d.cols; }
            float o[E];
#pragma unroll
            for (int j = 0; j < E; ++j) {
                const float th0 = word_f32<BT, E>(b, j);
                float tau[KC];
#pragma unroll
                for (int i = 0; i < KC; ++i) {
                    tau[i] = (i < K) ? word_f32<XT, E>(x[i], j) : 0.0f;
                    if (CK) tau[i] = __fsub_rn(tau[i], th0);
                }
                const uint32_t bits = exact ? select_bits<KC>(P, d, mp, K, tau, e + j, r, c)
                                            : fast_bits<KC>(T, K, tau);
                o[j] = merged_value<KC>(opk, iso1d, P.lambda, K, th0, tau, cf, bits);
            }
            store_out<BT, E>(op, e, n, o);
        };
        if (KC <= 4) {
            load(0, xa, ba);
#pragma unroll 1
            for (int st = 0; st < SPT; st += 2) {
                load(st + 1, xb, bb);
                merge_step(st, xa, ba);
                if (st + 2 < SPT) load(st + 2, xa, ba);
                merge_step(st + 1, xb, bb);
            }
        } else {
            // eight experts: one buffer (the registers of a second would spill)
#pragma unroll 1
            for (int st = 0; st < SPT; ++st) {
                load(st, xa, ba);
                merge_step(st, xa, ba);
            }
        }
    }
}

// steps of one warp whose loads are issued together in the Gram pass: KC
// 16-byte loads per step, 4 KB in flight per warp; eight experts take two
// steps (8 KB) and one block per SM, whose registers hold the 36 pair sums
// and both steps
template <int KC, int SPT>
struct Batch {
    static constexpr int U0 = KC >= 8 ? 2 : 8 / KC;
    static constexpr int U = U0 < SPT ? U0 : SPT;
};

// Gram of the trimmed task vectors, upper triangle, per 2-D trimmed tensor.
// Tile partials in binary32 (fused multiply-add over one lane's entries of
// the tile, then a warp sum), accumulated per warp in binary64 and added to
// the tensor's Gamma with one atomic per pair when the warp leaves the tensor.
template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB, gram_blocks_per_sm(KC)) k_gramk(Plan P) {
    constexpr int E = 16 / (int)sizeof(XT);
    constexpr int SPT = TILE / (32 * E);
    constexpr int U = Batch<KC, SPT>::U;
    constexpr int NP = KC * (KC + 1) / 2;
    static_assert(NP <= 64, "two pair sums per lane");
    const int K = P.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // lane L accumulates pairs L and 32 + L over the warp's tiles of one
    // tensor as binary32 two-sum pairs (no binary64 arithmetic per tile)
    float gs0 = 0.0f, ge0 = 0.0f, gs1 = 0.0f, ge1 = 0.0f;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    int t = tensor_of_tile(P.tens, P.n_tensors, wr.beg);
    long long t_end = tensor_tile_end(P, t);
    __shared__ MergeParams<KC> s_mp[WPB];
    MergeParams<KC>& mp = s_mp[warp];
    merge_params<KC>(P, t, K, mp);
    auto flush = [&](int tt) {
        int q = 0;
#pragma unroll
        for (int a = 0; a < KC; ++a) {
#pragma unroll
            for (int b = a; b < KC; ++b, ++q) {
                if (a < K && b < K && (lane == q || lane + 32 == q)) {
                    const double v = (lane == q) ? (double)gs0 + (double)ge0 : (double)gs1 + (double)ge1;
                    if (v != 0.0) atomicAdd(&P.gram[((long long)tt * K + a) * K + b], v);
                }
            }
        }
        gs0 = ge0 = gs1 = ge1 = 0.0f;
    };
    for (long long g = wr.beg; g < wr.end; ++g) {
        if (g >= t_end) {
            flush(t);
            while (g >= t_end) t_end = tensor_tile_end(P, ++t);
            merge_params<KC>(P, t, K, mp);
        }
        const TensorDesc& d = P.tens[t];
        if (!mp.trimmed2d) continue;
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
        int T[KC];
        const bool exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
        float acc[NP];
#pragma unroll
        for (int q = 0; q < NP; ++q) acc[q] = 0.0f;
#pragma unroll 1
        for (int s0 = 0; s0 < SPT; s0 += U) {
            Words<XT, E> xr[U][KC];
            Words<BT, E> br[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const long long e = e0 + (long long)(s0 + u) * (32 * E) + lane * E;
                if (e < n) {
                    if (CK) load_words<BT, E>(d.base, e, n, br[u]);
#pragma unroll
                    for (int i = 0; i < KC; ++i)
                        if (i < K) load_words<XT, E>(mp.xs[i], e, n, xr[u][i]);
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const long long e = e0 + (long long)(s0 + u) * (32 * E) + lane * E;
                if (e >= n) continue;
                long long r = 0, c = 0;
                if (exact && mp.sel == SEL_BLOCK) { r = e / d.cols; c = e - r * d.cols; }
#pragma unroll
                for (int j = 0; j < E; ++j) {
                    float tau[KC];
                    const float th0 = CK ? word_f32<BT, E>(br[u], j) : 0.0f;
#pragma unroll
                    for (int i = 0; i < KC; ++i) {
                        tau[i] = (i < K) ? word_f32<XT, E>(xr[u][i], j) : 0.0f;
                        if (CK) tau[i] = __fsub_rn(tau[i], th0);
                    }
                    uint32_t bits = 0;
                    if (e + j < n) bits = exact ? select_bits<KC>(P, d, mp, K, tau, e + j, r, c)
                                                : fast_bits<KC>(T, K, tau);
                    float m[KC];
#pragma unroll
                    for (int i = 0; i < KC; ++i) m[i] = ((bits >> i) & 1u) ? tau[i] : 0.0f;
                    int q = 0;
#pragma unroll
                    for (int a = 0; a < KC; ++a)
#pragma unroll
                        for (int b = a; b < KC; ++b, ++q) acc[q] = __fmaf_rn(m[a], m[b], acc[q]);
                }
            }
        }
        float w0 = 0.0f, w1 = 0.0f;
        int q = 0;
#pragma unroll
        for (int a = 0; a < KC; ++a) {
#pragma unroll
            for (int b = a; b < KC; ++b, ++q) {
                if (a < K && b < K) {
                    const float w = warp_sum(acc[q]);
                    if (q < 32) w0 = (lane == q) ? w : w0;
                    else w1 = (lane + 32 == q) ? w : w1;
                }
            }
        }
        two_sum_add(gs0, ge0, w0);
        if (NP > 32) two_sum_add(gs1, ge1, w1);
    }
    flush(t);
}

#define ISO_MERGE_INST(XT, BT, CK)                                             \
    template __global__ void k_merge<XT, BT, CK, 2>(Plan);                    \
    template __global__ void k_merge<XT, BT, CK, 4>(Plan);                    \
    template __global__ void k_merge<XT, BT, CK, 8>(Plan);                    \
    template __global__ void k_gramk<XT, BT, CK, 1>(Plan);                    \
    template __global__ void k_gramk<XT, BT, CK, 2>(Plan);                    \
    template __global__ void k_gramk<XT, BT, CK, 4>(Plan);                    \
    template __global__ void k_gramk<XT, BT, CK, 8>(Plan);

ISO_MERGE_INST(__nv_bfloat16, __nv_bfloat16, false)
ISO_MERGE_INST(__nv_bfloat16, float, false)
ISO_MERGE_INST(float, __nv_bfloat16, false)
ISO_MERGE_INST(float, float, false)
ISO_MERGE_INST(__nv_bfloat16, __nv_bfloat16, true)
ISO_MERGE_INST(__nv_bfloat16, float, true)
ISO_MERGE_INST(float, __nv_bfloat16, true)
ISO_MERGE_INST(float, float, true)

}  // namespace iso
