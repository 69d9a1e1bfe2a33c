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

enum OpKind : int { OPK_SUM = 0, OPK_TIES = 1, OPK_ISO = 2, OPK_RAM = 3 };

template <int KC>
struct MergeParams {
    const void* xs[KC];
    unsigned long long thr[KC];   // SEL_PACKED, tensor-local positions
    float cf[KC];                 // ISO 2-D coefficients
    int sel, opk;
    int teps;                     // RAM: key of eps_act (active: key > teps)
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
    mp.opk = (P.op == ISO_OP_TA || mp.iso1d) ? OPK_SUM
           : (P.op == ISO_OP_TIES ? OPK_TIES : (P.op == ISO_OP_RAM ? OPK_RAM : OPK_ISO));
    mp.teps = (int)__float_as_uint(P.eps_act);   // eps_act >= +0 and finite: below 2^31
    if (mp.opk == OPK_SUM || mp.opk == OPK_RAM) mp.sel = SEL_ALL;
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

// the merged output of one entry; every argument is in registers.  RAM never
// comes here: its tensors are untrimmed (SEL_ALL), so every tile takes the
// per-tile form below.
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
        T[i] = (i < K) ? -1 : 0x7FFFFFFF;                      // experts past K: nothing kept
        if (i < K && mp.opk == OPK_RAM) T[i] = mp.teps;        // RAM: active where |tau| > eps_act
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

// merged output of one entry inside a tile with per-tile thresholds: the
// selection of expert q is (int)key > T[q] (never for q >= K), unselected
// terms enter the sums as +0, which leaves every sum and the output as the
// skipping form gives them
template <int KC>
__device__ __forceinline__ float merged_fast(int opk, bool iso1d, float lambda, int K, float th0,
                                             const float (&tau)[KC], const float (&cf)[KC], const int (&T)[KC],
                                             uint32_t& kmax) {
    float upd;
    if (opk == OPK_RAM) {
        // RAM (App. F): active experts key > T (|tau| > eps_act; T is past
        // every key for q >= K); the active values summed in expert order,
        // divided by their count -- one active value is kept whole (0 + v
        // and v / 1 are exact), none leaves theta_0
        float s = 0.0f;
        int cnt = 0;
#pragma unroll
        for (int q = 0; q < KC; ++q) {
            const uint32_t k = key_of(tau[q]);
            kmax = (q < K && k > kmax) ? k : kmax;
            const bool a = (int)k > T[q];
            s = __fadd_rn(s, a ? tau[q] : 0.0f);
            cnt += a;
        }
        const float m = cnt ? __fdiv_rn(s, (float)cnt) : 0.0f;
        upd = __fmul_rn(lambda, m);
    } else if (opk == OPK_TIES) {
        // gamma = sign of the trimmed sum; the agreeing set: the non-zero
        // trimmed values of that sign.  u = tt with the sign of the sum
        // cleared is |tt| exactly for the agreeing ones, so their sum in
        // order is the magnitude of the signed sum, bit for bit.
        float tt[KC];
        float s = 0.0f;
#pragma unroll
        for (int q = 0; q < KC; ++q) {
            tt[q] = ((int)key_of(tau[q]) > T[q]) ? tau[q] : 0.0f;
            s = __fadd_rn(s, tt[q]);
        }
        const uint32_t sb = __float_as_uint(s) & 0x80000000u;
        float a = 0.0f;
        int cnt = 0;
#pragma unroll
        for (int q = 0; q < KC; ++q) {
            const float u = __uint_as_float(__float_as_uint(tt[q]) ^ sb);
            const bool ag = u > 0.0f;
            a = ag ? __fadd_rn(a, u) : a;
            cnt += ag;
        }
        if (s == 0.0f) cnt = 0;
        float m = cnt ? __fdiv_rn(a, (float)cnt) : 0.0f;
        m = __uint_as_float(__float_as_uint(m) ^ sb);
        upd = __fmul_rn(lambda, m);
    } else if (opk == OPK_ISO) {
        float s = 0.0f;
#pragma unroll
        for (int q = 0; q < KC; ++q)
            s = __fadd_rn(s, ((int)key_of(tau[q]) > T[q]) ? __fmul_rn(cf[q], tau[q]) : 0.0f);
        upd = s;
    } else {
        float s = 0.0f;
#pragma unroll
        for (int q = 0; q < KC; ++q)
            if (q < K) s = __fadd_rn(s, tau[q]);
        upd = iso1d ? __fdiv_rn(s, (float)K) : __fmul_rn(lambda, s);
    }
    return (upd == 0.0f) ? th0 : __fadd_rn(th0, upd);
}

template <int KC>
__device__ __forceinline__ uint32_t fast_bits(const int (&T)[KC], int K, const float (&tau)[KC]) {
    uint32_t bits = 0;
#pragma unroll
    for (int i = 0; i < KC; ++i)
        if (i < K && (int)key_of(tau[i]) > T[i]) bits |= 1u << i;
    return bits;
}

// the warp's tiles: beg, beg + step, ... below end -- dealt round-robin over
// the warps (all warps sweep one window of the tensors together, for DRAM
// page locality) or one contiguous range per warp
struct WarpRange {
    long long beg, end, step;
    __device__ __forceinline__ long long count() const { return beg < end ? (end - beg + step - 1) / step : 0; }
    __device__ __forceinline__ long long tile(long long j) const { return beg + j * step; }
};
__device__ __forceinline__ WarpRange warp_range(const Plan& P) {
    const long long W = (long long)gridDim.x * WPB;
    const long long wid = (long long)blockIdx.x * WPB + (threadIdx.x >> 5);
    WarpRange r;
    if (PASS_INTERLEAVE) {
        r.beg = wid;
        r.end = P.n_tiles;
        r.step = W;
    } else {
        const long long per = (P.n_tiles + W - 1) / W;
        r.beg = wid * per;
        r.end = (r.beg + per < P.n_tiles) ? r.beg + per : P.n_tiles;
        r.step = 1;
    }
    return r;
}

__device__ __forceinline__ long long tensor_tile_end(const Plan& P, int t) {
    return P.tens[t].tile_base + (P.tens[t].numel + TILE - 1) / TILE;
}

}  // namespace

// ---------------------------------------------------------------------------
// Staged streaming of the K experts and the base.  A warp walks its steps
// (tile, 32 lanes x E entries) in order; each lane copies its own 16-byte
// vector of every expert, and its base entries, into a per-warp ring of DEPTH
// stages in shared memory with cp.async, DEPTH - 1 steps ahead of the step it
// merges.  The data in flight then lives in shared memory instead of
// registers, which holds enough of it to keep HBM busy with eight experts.
// Each lane reads back only what it copied itself, so no barrier is needed.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" :: "r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" :: "r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory"); }

__device__ __forceinline__ uint32_t clamp_bytes(long long avail, uint32_t cap) {
    return avail <= 0 ? 0u : (avail >= (long long)cap ? cap : (uint32_t)avail);
}

template <typename XT, typename BT, int KC, int BLK = 2>
struct StageGeom {
    static constexpr int E = 16 / (int)sizeof(XT);          // entries per lane per step
    static constexpr int SPT = TILE / (32 * E);              // steps per tile
    static constexpr int BB = E * (int)sizeof(BT);           // base bytes per lane per step (8, 16, 32)
    static constexpr int BYTES = KC * 512 + 32 * BB;         // one stage of one warp
    // two blocks per SM: about 108 KB of ring per block; a kernel run at one
    // block per SM (BLK = 1) gets about 216 KB, a deeper ring
    static constexpr int BUDGET = BLK == 1 ? 221184 : 110592;
    static constexpr int DMAX = BLK == 1 ? 6 : 4;
    static constexpr int D0 = BUDGET / (WPB * BYTES);
    static constexpr int DEPTH = D0 < 2 ? 2 : (D0 > DMAX ? DMAX : D0);
    static constexpr int SMEM = WPB * DEPTH * BYTES;
};

// the tile a step belongs to and where its data comes from (issue side)
template <int KC, bool SMEM_PTRS>
struct IssueCursor;
// the tensor's expert pointers in registers
template <int KC>
struct IssueCursor<KC, false> {
    long long g = -1;        // tile of the cached tensor data
    int t = 0;
    long long t_end = 0, e0 = 0, n = 0;
    const void* xs[KC];
    const void* bp = nullptr;
};
// ... or in the warp's shared-memory copy (frees registers for two blocks per SM)
template <int KC>
struct IssueCursor<KC, true> {
    long long g = -1;
    int t = 0;
    long long t_end = 0, e0 = 0, n = 0;
    const void** xs;
    const void* bp = nullptr;
};

// copy step (g, s) of lane `lane` into stage `st` (shared-space address);
// NB = false leaves the base out (a pass over task vectors that never reads it)
template <typename XT, typename BT, int KC, bool SP, bool NB = true>
__device__ __forceinline__ void issue_step(const Plan& P, int K, IssueCursor<KC, SP>& ic, long long g, int s,
                                           uint32_t st, int lane) {
    using G = StageGeom<XT, BT, KC>;
    if (g != ic.g) {
        if (ic.g < 0 || g >= ic.t_end) {
            if (ic.g < 0) ic.t = tensor_of_tile(P.tens, P.n_tensors, g);
            while (g >= P.tens[ic.t].tile_base + (P.tens[ic.t].numel + TILE - 1) / TILE) ++ic.t;
            const TensorDesc& d = P.tens[ic.t];
            ic.t_end = d.tile_base + (d.numel + TILE - 1) / TILE;
            ic.n = d.numel;
            ic.bp = d.base;
#pragma unroll
            for (int i = 0; i < KC; ++i) ic.xs[i] = (i < K) ? P.xptr[i * P.n_tensors + ic.t] : nullptr;
            if (SP) __syncwarp();
        }
        ic.g = g;
        ic.e0 = (g - P.tens[ic.t].tile_base) * TILE;
    }
    const long long e = ic.e0 + (long long)s * (32 * G::E) + lane * G::E;
    const bool in = e < ic.n;
    const uint32_t xb = clamp_bytes((ic.n - e) * (long long)sizeof(XT), 16);
#pragma unroll
    for (int i = 0; i < KC; ++i) {
        if (i < K) {
            const char* src = static_cast<const char*>(ic.xs[i]) + (in ? e * (long long)sizeof(XT) : 0);
            cp_async16(st + i * 512 + lane * 16, src, xb);
        }
    }
    if (!NB) return;
    const uint32_t bdst = st + KC * 512 + lane * G::BB;
    const char* bsrc = static_cast<const char*>(ic.bp) + (in ? e * (long long)sizeof(BT) : 0);
    const long long bavail = (ic.n - e) * (long long)sizeof(BT);
    if (G::BB == 8) {
        cp_async8(bdst, bsrc, clamp_bytes(bavail, 8));
    } else {
#pragma unroll
        for (int q = 0; q < G::BB / 16; ++q)
            cp_async16(bdst + 16 * q, bsrc + (in && bavail > 16 * q ? 16 * q : 0), clamp_bytes(bavail - 16 * q, 16));
    }
}

// the step's words back from the stage
template <typename XT, typename BT, int KC>
__device__ __forceinline__ void read_step(const char* st, int K, int lane, Words<XT, 16 / (int)sizeof(XT)> (&x)[KC],
                                          Words<BT, 16 / (int)sizeof(XT)>& b) {
    using G = StageGeom<XT, BT, KC>;
    constexpr int E = G::E;
#pragma unroll
    for (int i = 0; i < KC; ++i) {
        if (i < K) {
            const uint4 v = *reinterpret_cast<const uint4*>(st + i * 512 + lane * 16);
            x[i].w[0] = v.x; x[i].w[1] = v.y; x[i].w[2] = v.z; x[i].w[3] = v.w;
        }
    }
    const char* bs = st + KC * 512 + lane * G::BB;
    if (G::BB == 8) {
        const uint2 v = *reinterpret_cast<const uint2*>(bs);
        b.w[0] = v.x; b.w[1] = v.y;
    } else {
#pragma unroll
        for (int q = 0; q < G::BB / 16; ++q) {
            const uint4 v = *reinterpret_cast<const uint4*>(bs + 16 * q);
            b.w[4 * q] = v.x; b.w[4 * q + 1] = v.y; b.w[4 * q + 2] = v.z; b.w[4 * q + 3] = v.w;
        }
    }
    (void)E;
}

// One warp per tile, a contiguous tile range per warp; every step staged
// through shared memory (above).
template <typename XT, typename BT, bool CK, int KC, int OPF>
__global__ void __launch_bounds__(TPB, merge_blocks_per_sm(KC, OPF)) k_merge(Plan P) {
    using G = StageGeom<XT, BT, KC, merge_blocks_per_sm(KC, OPF)>;
    constexpr int E = G::E;
    constexpr int SPT = G::SPT;
    constexpr int D = G::DEPTH;
    extern __shared__ __align__(16) char s_stage[];
    const int K = P.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    char* ring = s_stage + warp * D * G::BYTES;
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring);
    const long long NS = wr.count() * SPT;
    constexpr bool SP = merge_blocks_per_sm(KC, OPF) == 2 && KC >= 8;
    __shared__ const void* s_xs[WPB][KC];
    IssueCursor<KC, SP> ic;
    if constexpr (SP) ic.xs = s_xs[warp];
#pragma unroll
    for (int p = 0; p < D - 1; ++p) {
        if (p < NS) issue_step<XT, BT, KC, SP>(P, K, ic, wr.tile(p / SPT), p % SPT, ring_s + p * G::BYTES, lane);
        cp_async_commit();
    }
    int t = tensor_of_tile(P.tens, P.n_tensors, wr.beg);
    long long t_end = tensor_tile_end(P, t);
    __shared__ MergeParams<KC> s_mp[WPB];
    MergeParams<KC>& mp = s_mp[warp];
    merge_params<KC>(P, t, K, mp);
    float cf[KC];
    int T[KC];
    uint32_t kmax = 0;   // RAM: largest key seen (non-finite inputs)
    bool exact = false;
    int opk = 0;
    bool iso1d = false;
    long long n = 0, e0 = 0;
    void* op = nullptr;
    const TensorDesc* dp = nullptr;
#pragma unroll 1
    for (long long i = 0; i < NS; ++i) {
        const long long g = wr.tile(i / SPT);
        const int s = (int)(i % SPT);
        if (s == 0) {
            if (g >= t_end) {
                while (g >= t_end) t_end = tensor_tile_end(P, ++t);
                merge_params<KC>(P, t, K, mp);
            }
            dp = &P.tens[t];
            n = dp->numel;
            e0 = (g - dp->tile_base) * TILE;
            const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
#pragma unroll
            for (int q = 0; q < KC; ++q) cf[q] = (OPF == OPF_TIES) ? 0.0f : mp.cf[q];
            exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
            opk = (OPF == OPF_TIES) ? (int)OPK_TIES : mp.opk;
            iso1d = mp.iso1d;
            op = dp->out;
        }
        cp_async_wait<D - 2>();
        // eight experts: the step's words are read from the stage entry by
        // entry (the stage is the lane's own and is refilled only after this
        // step) -- fewer live registers, two blocks per SM without spills;
        // fewer experts read the whole step at once
        constexpr bool LAZY = KC >= 8;
        Words<XT, E> x[LAZY ? 1 : KC];
        Words<BT, E> b;
        const char* stg = ring + (int)(i % D) * G::BYTES;
        if constexpr (!LAZY) read_step<XT, BT, KC>(stg, K, lane, x, b);
        auto xw = [&](int q, int j) -> float {
            if constexpr (!LAZY) return word_f32<XT, E>(x[q], j);
            const char* p = stg + q * 512 + lane * 16;
            if (sizeof(XT) == 4) return *reinterpret_cast<const float*>(p + 4 * j);
            const uint32_t w = *reinterpret_cast<const uint32_t*>(p + 4 * (j >> 1));
            return __uint_as_float((j & 1) ? (w & 0xFFFF0000u) : (w << 16));
        };
        auto bw = [&](int j) -> float {
            if constexpr (!LAZY) return word_f32<BT, E>(b, j);
            const char* p = stg + KC * 512 + lane * G::BB;
            if (sizeof(BT) == 4) return *reinterpret_cast<const float*>(p + 4 * j);
            const uint32_t w = *reinterpret_cast<const uint32_t*>(p + 4 * (j >> 1));
            return __uint_as_float((j & 1) ? (w & 0xFFFF0000u) : (w << 16));
        };
        const long long ni = i + D - 1;
        if (ni < NS) issue_step<XT, BT, KC, SP>(P, K, ic, wr.tile(ni / SPT), (int)(ni % SPT), ring_s + (int)(ni % D) * G::BYTES, lane);
        cp_async_commit();
        const long long e = e0 + (long long)s * (32 * E) + lane * E;
        if (e >= n) continue;
        long long r = 0, c = 0;
        if (exact && mp.sel == SEL_BLOCK) { r = e / dp->cols; c = e - r * dp->cols; }
        float o[E];
#pragma unroll
        for (int j = 0; j < E; ++j) {
            const float th0 = bw(j);
            float tau[KC];
#pragma unroll
            for (int q = 0; q < KC; ++q) {
                tau[q] = (q < K) ? xw(q, j) : 0.0f;
                if (CK) tau[q] = __fsub_rn(tau[q], th0);
            }
            if (exact) {
                const uint32_t bits = select_bits<KC>(P, *dp, mp, K, tau, e + j, r, c);
                o[j] = merged_value<KC>(opk, iso1d, P.lambda, K, th0, tau, cf, bits);
            } else {
                o[j] = merged_fast<KC>(opk, iso1d, P.lambda, K, th0, tau, cf, T, kmax);
            }
        }
        store_out<BT, E>(op, e, n, o);
    }
    cp_async_wait<0>();
    // RAM reads every entry's magnitude: a NaN or infinity is reported
    // (entries past a tensor's end are staged as zeros)
    if (__any_sync(0xFFFFFFFFu, kmax >= KEY_INF) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
}

// Gram of the trimmed task vectors, upper triangle, per 2-D trimmed tensor.
// The experts stream through the same shared-memory ring as the merge.  Tile
// partials in binary32 (fused multiply-add over one lane's entries of the
// tile, then a warp sum), accumulated per warp as binary32 two-sum pairs and
// added to the tensor's Gamma with one atomic per pair when the warp leaves
// the tensor.
template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB, gram_blocks_per_sm(KC)) k_gramk(Plan P) {
    using G = StageGeom<XT, BT, KC, gram_blocks_per_sm(KC)>;
    constexpr int E = G::E;
    constexpr int SPT = G::SPT;
    constexpr int D = G::DEPTH;
    constexpr int NP = KC * (KC + 1) / 2;
    static_assert(NP <= 64, "two pair sums per lane");
    extern __shared__ __align__(16) char s_stage[];
    const int K = P.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // lane L accumulates pairs L and 32 + L over the warp's tiles of one
    // tensor as binary32 two-sum pairs (no binary64 arithmetic per tile)
    float gs0 = 0.0f, ge0 = 0.0f, gs1 = 0.0f, ge1 = 0.0f;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    char* ring = s_stage + warp * D * G::BYTES;
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring);
    const long long NS = wr.count() * SPT;
    constexpr bool SP = KC >= 8;   // eight experts: their pointers in shared memory (two blocks per SM)
    IssueCursor<KC, SP> ic;
    __shared__ const void* s_xs[WPB][KC];
    if constexpr (SP) ic.xs = s_xs[warp];
#pragma unroll
    for (int p = 0; p < D - 1; ++p) {
        if (p < NS) issue_step<XT, BT, KC, SP, CK>(P, K, ic, wr.tile(p / SPT), p % SPT, ring_s + p * G::BYTES, lane);
        cp_async_commit();
    }
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
    int T[KC];
    bool exact = false, active = false;
    long long n = 0, e0 = 0;
    const TensorDesc* dp = nullptr;
    float acc[NP];
#pragma unroll 1
    for (long long i = 0; i < NS; ++i) {
        const long long g = wr.tile(i / SPT);
        const int s = (int)(i % SPT);
        if (s == 0) {
            if (g >= t_end) {
                flush(t);
                while (g >= t_end) t_end = tensor_tile_end(P, ++t);
                merge_params<KC>(P, t, K, mp);
            }
            dp = &P.tens[t];
            active = mp.trimmed2d;
            n = dp->numel;
            e0 = (g - dp->tile_base) * TILE;
            const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
            exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
#pragma unroll
            for (int q = 0; q < NP; ++q) acc[q] = 0.0f;
        }
        cp_async_wait<D - 2>();
        // the step's words are read from the stage entry by entry (the stage is
        // the lane's own and is refilled only after this step): fewer live
        // registers than a whole step's words, two blocks per SM
        const char* stg = ring + (int)(i % D) * G::BYTES;
        auto xw = [&](int q, int j) -> float {
            const char* p = stg + q * 512 + lane * 16;
            if (sizeof(XT) == 4) return *reinterpret_cast<const float*>(p + 4 * j);
            const uint32_t w = *reinterpret_cast<const uint32_t*>(p + 4 * (j >> 1));
            return __uint_as_float((j & 1) ? (w & 0xFFFF0000u) : (w << 16));
        };
        auto bw = [&](int j) -> float {
            const char* p = stg + KC * 512 + lane * G::BB;
            if (sizeof(BT) == 4) return *reinterpret_cast<const float*>(p + 4 * j);
            const uint32_t w = *reinterpret_cast<const uint32_t*>(p + 4 * (j >> 1));
            return __uint_as_float((j & 1) ? (w & 0xFFFF0000u) : (w << 16));
        };
        const long long ni = i + D - 1;
        if (ni < NS) issue_step<XT, BT, KC, SP, CK>(P, K, ic, wr.tile(ni / SPT), (int)(ni % SPT), ring_s + (int)(ni % D) * G::BYTES, lane);
        cp_async_commit();
        const long long e = e0 + (long long)s * (32 * E) + lane * E;
        if (active && e < n) {
            long long r = 0, c = 0;
            if (exact && mp.sel == SEL_BLOCK) { r = e / dp->cols; c = e - r * dp->cols; }
#pragma unroll
            for (int j = 0; j < E; ++j) {
                float tau[KC];
                const float th0 = CK ? bw(j) : 0.0f;
#pragma unroll
                for (int q = 0; q < KC; ++q) {
                    tau[q] = (q < K) ? xw(q, j) : 0.0f;
                    if (CK) tau[q] = __fsub_rn(tau[q], th0);
                }
                float m[KC];
                if (exact) {
                    const uint32_t bits = (e + j < n) ? select_bits<KC>(P, *dp, mp, K, tau, e + j, r, c) : 0u;
#pragma unroll
                    for (int q = 0; q < KC; ++q) m[q] = ((bits >> q) & 1u) ? tau[q] : 0.0f;
                } else {
                    // past the tensor's end the loads read zeros: key 0 is never selected by T >= 0,
                    // and T = -1 (everything kept) only leaves zeros in the sums
#pragma unroll
                    for (int q = 0; q < KC; ++q) m[q] = ((int)key_of(tau[q]) > T[q]) ? tau[q] : 0.0f;
                }
                int q = 0;
#pragma unroll
                for (int a2 = 0; a2 < KC; ++a2)
#pragma unroll
                    for (int b2 = a2; b2 < KC; ++b2, ++q) acc[q] = __fmaf_rn(m[a2], m[b2], acc[q]);
            }
        }
        if (s == SPT - 1 && active) {
            // the tile's partial sums: warp sums, then one two-sum per lane
            float w0 = 0.0f, w1 = 0.0f;
            int q = 0;
#pragma unroll
            for (int a2 = 0; a2 < KC; ++a2) {
#pragma unroll
                for (int b2 = a2; b2 < KC; ++b2, ++q) {
                    if (a2 < K && b2 < K) {
                        const float w = warp_sum(acc[q]);
                        if (q < 32) w0 = (lane == q) ? w : w0;
                        else w1 = (lane + 32 == q) ? w : w1;
                    }
                }
            }
            two_sum_add(gs0, ge0, w0);
            if (NP > 32) two_sum_add(gs1, ge1, w1);
        }
    }
    cp_async_wait<0>();
    flush(t);
}

// ---------------------------------------------------------------------------
// Compact candidates (Plan::ccv).  The count pass has written, per expert and
// tile, the binary32 task-vector values whose key is at least the low edge of
// the unit's band, in position order, and a 32-word mask of their positions.
// When the unit's threshold lies in its band (Unit::v_ok) those values hold
// every entry the selection can keep, so the Gram and merge passes read them
// (about the kept fraction of each expert's bytes) instead of the full task
// vectors; any other expert of the tensor (an untrimmed tensor, a unit whose
// band missed or whose value segment overflowed) is read in full.  An entry
// absent from the values has key < lo <= t: never kept, it enters every sum
// as +0 exactly as an unkept entry does in k_merge / k_gramk, so both give
// the same results.  One warp per tile, lane l taking entries 4 l .. 4 l + 3
// of each 128-entry step: the four bits of word 4 s + l / 8 at 4 (l % 8).
// ---------------------------------------------------------------------------
template <int KC>
struct CompactParams {
    uint32_t vok;                      // bit q: expert q reads its compact values
    unsigned long long voff[KC];       // the unit's value segment in the pool
};

template <int KC>
__device__ __forceinline__ void compact_params(const Plan& P, int t, int K, CompactParams<KC>& cp) {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) {
        const TensorDesc& d = P.tens[t];
        uint32_t ok = 0;
#pragma unroll
        for (int q = 0; q < KC; ++q) {
            cp.voff[q] = 0;
            if (q < K && (d.flags & TF_TRIM)) {
                const Unit& U = P.units[(long long)q * P.n_units + d.unit];
                if (U.v_ok) { ok |= 1u << q; cp.voff[q] = U.v_off; }
            }
        }
        cp.vok = ok;
    }
    __syncwarp();
}

// the tile's mask words, their exclusive popcount prefix and the value
// pointer of each compact expert, in the warp's shared memory (registers
// stay free for the data); the tile's values of each expert (when they fit
// CC_STAGE slots) and the tile's theta_0 are copied into the warp's stage
// with cp.async before the tile is merged, so that the merge reads shared
// memory only: two round trips to memory per tile (mask words, then values)
// instead of one per step.
constexpr int CC_STAGE = 256;
template <int KC, typename BT>
struct CompactTile {
    uint32_t mw[KC][32], pre[KC][32];
    const float* vb[KC];
    uint32_t staged;                   // bit q: expert q's values are in sv[q]
    float sv[KC][CC_STAGE];
    __align__(16) char th0[TILE * sizeof(BT)];
};

__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" :: "r"(dst), "l"(src) : "memory");
}

template <int KC, typename BT>
__device__ __forceinline__ void compact_tile(const Plan& P, const CompactParams<KC>& cp, int K, long long g, int lane,
                                             const void* base, long long e0, long long n, bool want_base,
                                             CompactTile<KC, BT>& ct) {
    __syncwarp();
    uint32_t cnt[KC];
#pragma unroll
    for (int q = 0; q < KC; ++q) {
        cnt[q] = 0;
        if (q < K && ((cp.vok >> q) & 1u)) {
            const long long rec = (long long)q * P.n_tiles + g;
            const uint32_t w = P.vmask[rec * 32 + lane];
            ct.pre[q][lane] = warp_excl_scan((uint32_t)__popc(w), &cnt[q]);
            ct.mw[q][lane] = w;
            if (lane == 0) ct.vb[q] = P.vals + cp.voff[q] + P.tval[rec];
        }
    }
    __syncwarp();
    uint32_t staged = 0;
#pragma unroll
    for (int q = 0; q < KC; ++q) {
        if (q < K && ((cp.vok >> q) & 1u) && cnt[q] <= (uint32_t)CC_STAGE) {
            staged |= 1u << q;
            const float* src = ct.vb[q];
            const uint32_t dst = (uint32_t)__cvta_generic_to_shared(&ct.sv[q][0]);
            for (uint32_t i = lane; i < cnt[q]; i += 32) cp_async4(dst + 4 * i, src + i);
        }
    }
    if (want_base) {
        // the tile's theta_0, 16 bytes per lane per copy, zero-filled past the tensor's end
        const uint32_t dst = (uint32_t)__cvta_generic_to_shared(ct.th0);
        const char* src = static_cast<const char*>(base) + e0 * (long long)sizeof(BT);
        const long long avail = (n - e0) * (long long)sizeof(BT);
#pragma unroll
        for (int k = 0; k < (int)(TILE * sizeof(BT)) / 512; ++k) {
            const long long off = (long long)k * 512 + lane * 16;
            cp_async16(dst + (uint32_t)off, src + (avail > off ? off : 0), clamp_bytes(avail - off, 16));
        }
    }
    cp_async_commit();
    cp_async_wait<0>();
    if (lane == 0) ct.staged = staged;
    __syncwarp();
}

template <typename BT>
__device__ __forceinline__ float staged_base(const char* th0, int p) {
    if (sizeof(BT) == 4) return reinterpret_cast<const float*>(th0)[p];
    return __uint_as_float((uint32_t)reinterpret_cast<const unsigned short*>(th0)[p] << 16);
}

// tau of entries e .. e + 3 (step s of the tile) for every expert: compact
// values, or the full task vector; entries past the tensor's end read 0
template <typename XT, typename BT, bool CK, int KC>
__device__ __forceinline__ void compact_step(const CompactParams<KC>& cp, const CompactTile<KC, BT>& ct,
                                             const void* const* xs, int K, long long e, long long n, int s, int lane,
                                             const float (&th0)[4], float (&tau)[KC][4]) {
    const int w = s * 4 + (lane >> 3), bo = (lane & 7) * 4;
#pragma unroll
    for (int q = 0; q < KC; ++q) {
#pragma unroll
        for (int j = 0; j < 4; ++j) tau[q][j] = 0.0f;
        if (q >= K) continue;
        if ((cp.vok >> q) & 1u) {
            const uint32_t word = ct.mw[q][w];
            const uint32_t at = ct.pre[q][w] + (uint32_t)__popc(word & ((1u << bo) - 1u));
            const uint32_t nib = (word >> bo) & 0xFu;
            const bool st = (ct.staged >> q) & 1u;
            const float* vb = (st ? &ct.sv[q][0] : ct.vb[q]) + at;
            uint32_t r = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if ((nib >> j) & 1u) { tau[q][j] = st ? vb[r] : __ldg(vb + r); ++r; }
            }
        } else {
            Words<XT, 4> x;
            load_words<XT, 4>(xs[q], e, n, x);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                tau[q][j] = word_f32<XT, 4>(x, j);
                if (CK) tau[q][j] = __fsub_rn(tau[q][j], th0[j]);
            }
        }
    }
}

template <typename XT, typename BT, bool CK, int KC, int OPF>
__global__ void __launch_bounds__(TPB, 2) k_merge_c(Plan P) {
    constexpr int E = 4, SPT = TILE / (32 * E);
    const int K = P.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    __shared__ MergeParams<KC> s_mp[WPB];
    __shared__ CompactParams<KC> s_cp[WPB];
    extern __shared__ __align__(16) char s_cstage[];
    CompactTile<KC, BT>& ct = reinterpret_cast<CompactTile<KC, BT>*>(s_cstage)[warp];
    MergeParams<KC>& mp = s_mp[warp];
    CompactParams<KC>& cp = s_cp[warp];
    int t = tensor_of_tile(P.tens, P.n_tensors, wr.beg);
    long long t_end = tensor_tile_end(P, t);
    merge_params<KC>(P, t, K, mp);
    compact_params<KC>(P, t, K, cp);
    const long long nt = wr.count();
#pragma unroll 1
    for (long long jt = 0; jt < nt; ++jt) {
        const long long g = wr.tile(jt);
        if (g >= t_end) {
            while (g >= t_end) t_end = tensor_tile_end(P, ++t);
            merge_params<KC>(P, t, K, mp);
            compact_params<KC>(P, t, K, cp);
        }
        const TensorDesc& d = P.tens[t];
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
        int T[KC];
        float cf[KC];
        const bool exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
#pragma unroll
        for (int q = 0; q < KC; ++q) cf[q] = (OPF == OPF_TIES) ? 0.0f : mp.cf[q];
        const int opk = (OPF == OPF_TIES) ? (int)OPK_TIES : mp.opk;
        const bool iso1d = mp.iso1d;
        compact_tile<KC, BT>(P, cp, K, g, lane, d.base, e0, n, true, ct);
        uint32_t kmax = 0;
#pragma unroll 1
        for (int s = 0; s < SPT; ++s) {
            const long long e = e0 + (long long)s * (32 * E) + lane * E;
            float th0[E];
#pragma unroll
            for (int j = 0; j < E; ++j) th0[j] = staged_base<BT>(ct.th0, s * (32 * E) + lane * E + j);
            float tau[KC][E];
            compact_step<XT, BT, CK, KC>(cp, ct, mp.xs, K, e, n, s, lane, th0, tau);
            long long r = 0, c = 0;
            if (exact && mp.sel == SEL_BLOCK) { r = e / d.cols; c = e - r * d.cols; }
            float o[E];
#pragma unroll
            for (int j = 0; j < E; ++j) {
                float tj[KC];
#pragma unroll
                for (int q = 0; q < KC; ++q) tj[q] = tau[q][j];
                if (exact) {
                    const uint32_t bits = (e + j < n) ? select_bits<KC>(P, d, mp, K, tj, e + j, r, c) : 0u;
                    o[j] = merged_value<KC>(opk, iso1d, P.lambda, K, th0[j], tj, cf, bits);
                } else {
                    o[j] = merged_fast<KC>(opk, iso1d, P.lambda, K, th0[j], tj, cf, T, kmax);
                }
            }
            store_out<BT, E>(d.out, e, n, o);
        }
    }
}

// Gram of the trimmed task vectors from the compact candidates (see above);
// partial sums as in k_gramk: per lane over the tile's entries in order,
// warp sums per tile, binary32 two-sum pairs per tensor, one atomic per pair.
template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB, 2) k_gramk_c(Plan P) {
    constexpr int E = 4, SPT = TILE / (32 * E);
    constexpr int NP = KC * (KC + 1) / 2;
    static_assert(NP <= 64, "two pair sums per lane");
    const int K = P.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float gs0 = 0.0f, ge0 = 0.0f, gs1 = 0.0f, ge1 = 0.0f;
    const WarpRange wr = warp_range(P);
    if (wr.beg >= wr.end) return;
    __shared__ MergeParams<KC> s_mp[WPB];
    __shared__ CompactParams<KC> s_cp[WPB];
    extern __shared__ __align__(16) char s_cstage[];
    CompactTile<KC, BT>& ct = reinterpret_cast<CompactTile<KC, BT>*>(s_cstage)[warp];
    MergeParams<KC>& mp = s_mp[warp];
    CompactParams<KC>& cp = s_cp[warp];
    int t = tensor_of_tile(P.tens, P.n_tensors, wr.beg);
    long long t_end = tensor_tile_end(P, t);
    merge_params<KC>(P, t, K, mp);
    compact_params<KC>(P, t, K, cp);
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
    const long long nt = wr.count();
#pragma unroll 1
    for (long long jt = 0; jt < nt; ++jt) {
        const long long g = wr.tile(jt);
        if (g >= t_end) {
            flush(t);
            while (g >= t_end) t_end = tensor_tile_end(P, ++t);
            merge_params<KC>(P, t, K, mp);
            compact_params<KC>(P, t, K, cp);
        }
        if (!mp.trimmed2d) continue;
        const TensorDesc& d = P.tens[t];
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const long long e1 = (e0 + TILE < n) ? e0 + TILE : n;
        int T[KC];
        const bool exact = tile_thresholds<KC>(mp, K, (uint32_t)e0, (uint32_t)e1, T);
        const bool want_base = CK && cp.vok != ((1u << K) - 1u);
        compact_tile<KC, BT>(P, cp, K, g, lane, d.base, e0, n, want_base, ct);
        float acc[NP];
#pragma unroll
        for (int q = 0; q < NP; ++q) acc[q] = 0.0f;
#pragma unroll 1
        for (int s = 0; s < SPT; ++s) {
            const long long e = e0 + (long long)s * (32 * E) + lane * E;
            float th0[E] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (want_base) {
#pragma unroll
                for (int j = 0; j < E; ++j) th0[j] = staged_base<BT>(ct.th0, s * (32 * E) + lane * E + j);
            }
            float tau[KC][E];
            compact_step<XT, BT, CK, KC>(cp, ct, mp.xs, K, e, n, s, lane, th0, tau);
            long long r = 0, c = 0;
            if (exact && mp.sel == SEL_BLOCK) { r = e / d.cols; c = e - r * d.cols; }
#pragma unroll
            for (int j = 0; j < E; ++j) {
                float tj[KC], m[KC];
#pragma unroll
                for (int q = 0; q < KC; ++q) tj[q] = tau[q][j];
                if (exact) {
                    const uint32_t bits = (e + j < n) ? select_bits<KC>(P, d, mp, K, tj, e + j, r, c) : 0u;
#pragma unroll
                    for (int q = 0; q < KC; ++q) m[q] = ((bits >> q) & 1u) ? tj[q] : 0.0f;
                } else {
#pragma unroll
                    for (int q = 0; q < KC; ++q) m[q] = ((int)key_of(tj[q]) > T[q]) ? tj[q] : 0.0f;
                }
                int q = 0;
#pragma unroll
                for (int a2 = 0; a2 < KC; ++a2)
#pragma unroll
                    for (int b2 = a2; b2 < KC; ++b2, ++q) acc[q] = __fmaf_rn(m[a2], m[b2], acc[q]);
            }
        }
        float w0 = 0.0f, w1 = 0.0f;
        int q = 0;
#pragma unroll
        for (int a2 = 0; a2 < KC; ++a2) {
#pragma unroll
            for (int b2 = a2; b2 < KC; ++b2, ++q) {
                if (a2 < K && b2 < K) {
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

template <typename XT, typename BT, int KC, int OPF>
int merge_smem_bytes() { return StageGeom<XT, BT, KC, merge_blocks_per_sm(KC, OPF)>::SMEM; }
template <typename BT, int KC>
int compact_smem_bytes() { return WPB * (int)sizeof(CompactTile<KC, BT>); }
template <typename XT, typename BT, int KC>
int gram_smem_bytes() { return StageGeom<XT, BT, KC, gram_blocks_per_sm(KC)>::SMEM; }

#define ISO_MERGE_SMEM(XT, BT)                                                 \
    template int merge_smem_bytes<XT, BT, 2, OPF_TIES>();                     \
    template int merge_smem_bytes<XT, BT, 4, OPF_TIES>();                     \
    template int merge_smem_bytes<XT, BT, 8, OPF_TIES>();                     \
    template int merge_smem_bytes<XT, BT, 2, OPF_OTHER>();                    \
    template int merge_smem_bytes<XT, BT, 4, OPF_OTHER>();                    \
    template int merge_smem_bytes<XT, BT, 8, OPF_OTHER>();                    \
    template int gram_smem_bytes<XT, BT, 1>();                                \
    template int gram_smem_bytes<XT, BT, 2>();                                \
    template int gram_smem_bytes<XT, BT, 4>();                                \
    template int gram_smem_bytes<XT, BT, 8>();
template int compact_smem_bytes<__nv_bfloat16, 2>();
template int compact_smem_bytes<__nv_bfloat16, 4>();
template int compact_smem_bytes<__nv_bfloat16, 8>();
template int compact_smem_bytes<float, 2>();
template int compact_smem_bytes<float, 4>();
template int compact_smem_bytes<float, 8>();
ISO_MERGE_SMEM(__nv_bfloat16, __nv_bfloat16)
ISO_MERGE_SMEM(__nv_bfloat16, float)
ISO_MERGE_SMEM(float, __nv_bfloat16)
ISO_MERGE_SMEM(float, float)

#define ISO_MERGE_INST(XT, BT, CK)                                             \
    template __global__ void k_merge_c<XT, BT, CK, 2, OPF_TIES>(Plan);        \
    template __global__ void k_merge_c<XT, BT, CK, 4, OPF_TIES>(Plan);        \
    template __global__ void k_merge_c<XT, BT, CK, 8, OPF_TIES>(Plan);        \
    template __global__ void k_merge_c<XT, BT, CK, 2, OPF_OTHER>(Plan);       \
    template __global__ void k_merge_c<XT, BT, CK, 4, OPF_OTHER>(Plan);       \
    template __global__ void k_merge_c<XT, BT, CK, 8, OPF_OTHER>(Plan);       \
    template __global__ void k_gramk_c<XT, BT, CK, 2>(Plan);                  \
    template __global__ void k_gramk_c<XT, BT, CK, 4>(Plan);                  \
    template __global__ void k_gramk_c<XT, BT, CK, 8>(Plan);                  \
    template __global__ void k_merge<XT, BT, CK, 2, OPF_TIES>(Plan);          \
    template __global__ void k_merge<XT, BT, CK, 4, OPF_TIES>(Plan);          \
    template __global__ void k_merge<XT, BT, CK, 8, OPF_TIES>(Plan);          \
    template __global__ void k_merge<XT, BT, CK, 2, OPF_OTHER>(Plan);         \
    template __global__ void k_merge<XT, BT, CK, 4, OPF_OTHER>(Plan);         \
    template __global__ void k_merge<XT, BT, CK, 8, OPF_OTHER>(Plan);         \
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
