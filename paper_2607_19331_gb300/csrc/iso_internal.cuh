// iso_internal.cuh -- device-side data structures and helpers shared by the
// kernels of the GB300 delta-merge library.
//
// Element-wise path (App. F of the paper for TopKMask / TA / TIES; Sec. 4.2,
// App. E and Algorithm 1 for the retention combiner):
//   tau   = theta_i - theta_0          (binary32, one subtraction)
//   key   = bits(|tau|)                (binary32 pattern, sign cleared: monotone in |tau|)
//   mask  = key > t || (key == t && index < cut)   per selection unit
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "iso.h"

namespace iso {

// ---------------------------------------------------------------------------
// geometry
// ---------------------------------------------------------------------------
// A tile is 1024 consecutive entries of one tensor, processed by one warp:
// lane L holds entries e0 + v*256 + 8L .. +8 for v = 0..3 (each warp-wide
// vector step reads 256 consecutive entries).
constexpr int TILE = 1024;                  // entries per tile
constexpr int VEC = 8;                      // entries per lane per vector step
constexpr int WVEC = TILE / (32 * VEC);     // vector steps per tile (4)
constexpr int TPB = 256;                    // threads per streaming block
constexpr int WPB = TPB / 32;               // warps per streaming block
static_assert(WVEC * 32 * VEC == TILE, "tile geometry");
constexpr int CHUNK_MAX = 1024;             // candidate slots a warp reserves at once
constexpr int VCHUNK = 8192;                // compact-candidate value slots a warp reserves at most at once

constexpr int SAMPLE_MAX = 24576;           // sampled keys per unit (96 KB of smem: two blocks per SM)
constexpr int SAMPLE_CHUNK = 256;           // contiguous entries per sample chunk
constexpr int SAMPLE_TPB = 512;             // two sample blocks per SM
constexpr int SAMPLE_SEL_R = 5;             // ranks selected at once from the sample
constexpr int CUT_TPB = 1024;
constexpr int CS_SPLIT = 4;                 // count-sample blocks per unit
constexpr int CS_TPB = 256;
constexpr double SAMPLE_Z = 5.0;            // band half-width in sample standard deviations
constexpr int COUNT_CHUNKS = 512;           // fused K = 1 pass: 256-entry chunks counted for the cut estimate

constexpr int RADIX_BITS = 11;
constexpr int RADIX_BINS = 1 << RADIX_BITS;
// A unit whose candidate pool holds at least this many slots is histogrammed
// as one flat array (the count pass seals the unused slots of its chunks with
// KEY_NONE), not tile by tile.
constexpr unsigned long long RADIX_FLAT_MIN = 1ull << 20;
constexpr int RADIX_FLAT_SMEM = (WPB + 2) * RADIX_BINS * 4;   // k_radix_flat's dynamic shared memory
constexpr int COUNT_EMIT_SMEM = WPB * 32 * 33 * 4;               // k_count<..., true>'s dynamic shared memory
// A unit with at least this many tiles finds the tile of its cut from
// per-chunk tie sums (k_cut_part, RADIX_BINS chunks) before it scans tiles.
constexpr long long CUT_SPLIT_MIN = 1ll << 16;
constexpr int BLOCK_MAX_ENTRIES = 16384;    // BLOCK scope: entries per unit held on chip
constexpr int BLOCK_KEYS_WORDS = BLOCK_MAX_ENTRIES + BLOCK_MAX_ENTRIES / 32;   // padded key array

constexpr int MAXK = ISO_MAX_EXPERTS;
constexpr uint32_t KEY_NONE = 0xFFFFFFFFu;  // threshold of a unit that selects nothing
constexpr uint32_t KEY_MAX = 0x7FFFFFFFu;   // largest key
constexpr uint32_t KEY_INF = 0x7F800000u;   // keys >= this are not finite
constexpr long long CUT_ALL = 0x7FFFFFFFFFFFFFFFLL;

// ---------------------------------------------------------------------------
// tables (in the caller's workspace)
// ---------------------------------------------------------------------------
enum TensorFlags : int32_t { TF_1D = 1, TF_TRIM = 2 };

struct TensorDesc {
    const void* base;        // theta_0 (or tau for iso_topk_mask)
    void*       out;         // merged output (NULL for mask-only calls)
    long long   numel;
    long long   uoff;        // GLOBAL scope: position of entry 0 in the unit order
    long long   tile_base;   // first tile id (group-local)
    long long   rows, cols;
    int32_t     flags;
    int32_t     unit;        // TENSOR: this tensor's unit; BLOCK: first block unit
    int32_t     bpr;         // BLOCK: blocks per block row
    int32_t     nblocks;     // BLOCK: blocks in this tensor
    unsigned long long cand_off;  // TENSOR: expert 0's candidate segment (expert i adds i*cand_cap)
    unsigned long long cand_cap;
    unsigned long long brec_off;  // fused K = 1 pass: band-record segment
    unsigned long long brec_cap;
    unsigned long long v_off;     // compact candidates: expert 0's value segment (expert i adds i*v_cap)
    unsigned long long v_cap;
};

enum UnitState : int32_t {
    ST_OFF = 0,      // not trimmed: every entry is kept
    ST_NONE = 1,     // k == 0: nothing is kept
    ST_SAMPLE = 2,   // waiting for the band
    ST_BAND = 3,     // band set; the count pass fills the counters
    ST_RADIX = 4,    // exact select in progress (interior candidates or full data)
    ST_TKNOWN = 5,   // threshold known; cut pending
    ST_DONE = 6
};
enum RadixSource : int32_t { SRC_CAND = 0, SRC_DATA = 1 };
enum TieSource : int32_t { TIE_EQ_HI = 0, TIE_EQ_LO = 1, TIE_ARRAY = 2 };

struct Unit {
    // static
    long long n, k;
    long long tile_begin, tile_end;     // group-local tiles covering the unit
    unsigned long long cand_off, cand_cap;
    int32_t tensor;                     // TENSOR / BLOCK: owning tensor; GLOBAL: -1
    int32_t expert;
    int32_t state;
    int32_t want_gamma;                 // accumulate sum of squares of the kept entries
    // band
    uint32_t lo, hi;
    // count-pass accumulators
    unsigned long long c_gt;            // keys above the band
    unsigned long long n_int;           // keys in the band (the candidates)
    unsigned long long c_hi, c_lo;      // band keys equal to hi / to lo (lo != hi)
    unsigned long long n_alloc;         // candidate slots handed out (>= n_int)
    int32_t overflow;                   // the segment could not hold every band key
    int32_t pad0;
    unsigned long long b_alloc;         // band-record slots handed out (fused K = 1 pass)
    unsigned long long brec_off, brec_cap;
    int32_t b_overflow;                 // the band records did not fit
    int32_t pad1;
    double gamma_acc;                   // sum tau^2 over key > hi (count pass)
    double gamma_band;                  // sum tau^2 over the band keys above lo (count pass)
    double gamma_rad;                   // sum tau^2 over the candidates (or, on the fallback, all entries) above t
    // radix select
    int32_t r_src;
    int32_t r_shift, r_pshift;
    uint32_t r_base;                    // key offset: lo for candidates, 0 for data
    uint32_t r_prefix;
    int32_t fallback;
    long long r_rank;                   // rank (1-based, from the top) inside the current set
    long long r_above;                  // entries above the current set
    // result
    uint32_t t;
    int32_t tie_src;
    long long count_above, ties, need;
    long long cut;                      // kept iff key > t || (key == t && pos < cut)
    double gamma;
    // fused K = 1 pass: the sample's estimate t^ of the threshold (that) and
    // of the cut among its ties (chat); the band's other keys are the
    // candidates, the keys equal to t^ are counted per tile (teq_hi)
    int32_t mode_t;
    uint32_t that;
    long long chat;
    unsigned long long c_eq;            // keys == t^
    unsigned long long c_abv;           // candidates above t^
    long long fix0, fix1;               // positions k_fix re-applies (k_fix_plan)
    long long fix_off;                  // tiles to fix in the units before this one
    unsigned long long cs_gt;           // count sample: keys above t^
    uint32_t cs_done;                   // count-sample blocks finished
    int32_t pad2;
    // compact candidates (K >= 2 merges): the values with key >= lo, per
    // tile in position order, in this unit's value segment
    unsigned long long v_off, v_cap;    // segment in the value pool, slots
    unsigned long long v_alloc;         // slots handed out (above v_cap: overflow)
    int32_t v_ok;                       // every kept entry is in the compact candidates (set by k_decide)
    int32_t pad3;
};

// Per (expert, tile) records of the count pass, as separate arrays:
//   tcand  (first slot of the tile's band keys in the unit's candidate
//          segment, band keys stored; count 0 when the segment overflowed)
//   teq_lo / teq_hi  band keys == lo / == hi in the tile
//   tcnt   keys == t in the tile (interior thresholds; written by k_tie)
//   tval   compact candidates: first slot of the tile's values in the unit's
//          value segment (KEY_NONE when the segment overflowed); vmask holds
//          32 words per record, bit p of word w for position 32 w + p of the
//          tile (key >= lo), and the tile's values follow the set bits in
//          position order

struct Header {             // first bytes of the workspace
    int32_t status;
    int32_t n_radix;        // units in ST_RADIX after the last pick
    int32_t n_tknown;
    int32_t fix_tiles;      // fused K = 1 pass: tiles k_fix re-applies (k_fix_plan)
};

// Everything a kernel needs to find its tables.
struct Plan {
    Header*       hdr;
    TensorDesc*   tens;
    const void**  xptr;     // [K][n_tensors] expert data
    Unit*         units;    // [K][n_units]
    uint2*        tcand;    // [K][n_tiles] (start, count) of the tile's band keys
    uint32_t*     teq_lo;   // [K][n_tiles]
    uint32_t*     teq_hi;   // [K][n_tiles]
    uint32_t*     tcnt;     // [K][n_tiles] ties at t per tile
    uint32_t*     hist;     // [K * n_units][RADIX_BINS]
    uint32_t*     hmxc;     // [K * n_units][RADIX_BINS] per bin: max of ~key (its smallest key)
    uint32_t*     hmx;      // [K * n_units][RADIX_BINS] per bin: largest key
    uint32_t*     cand;     // candidate pool
    uint2*        brec;     // fused K = 1 pass: band records (position, theta_0 bits << 16 | x bits)
    uint2*        tband;    // fused K = 1 pass: [n_tiles] (start, count) of the tile's band records
    uint32_t*     csamp;    // fused K = 1 pass: [n_units][COUNT_CHUNKS] sampled ties of t^ per chunk
    int32_t*      repair;   // fused K = 1 pass: [n_tensors] tensor needs the full exact apply
    uint32_t*     vmask;    // compact candidates: [K][n_tiles][32] words
    uint32_t*     tval;     // compact candidates: [K][n_tiles] first value slot (KEY_NONE: overflow)
    float*        vals;     // compact candidates: value pool (binary32 tau)
    double*       gram;     // [n_tensors][K][K]
    double*       coef;     // [n_tensors][K]
    int32_t n_tensors;
    int32_t K;
    int32_t n_units;        // per expert
    int32_t scope;
    long long n_tiles;
    int32_t xdt;            // expert dtype
    int32_t bdt;            // base dtype
    int32_t ckpt;           // experts are checkpoints (tau = x - base)
    int32_t op;
    int32_t fused;          // the K = 1 update runs the fused single pass
    int32_t fuse_block;     // BLOCK scope, K = 1 TIES: k_block_select writes the outputs
    int32_t ccv;            // K >= 2 TIES / ISO: the count pass writes compact candidates and
                            // the Gram and merge passes read them for every unit with v_ok
    int32_t block_rows, block_cols;
    float lambda;
    float eps_act;          // RAM: expert active where the binary32 |tau| > eps_act (>= +0)
    double density, ridge, c_min, c_max;
    // stats destinations (device, may be NULL) and the unit offset of this group
    iso_unit_stats* st_units;
    long long st_units_stride;          // units per expert in the caller's array
    int32_t st_unit_base;               // this group's first unit in the caller's array
    int32_t st_tensor_base;             // this group's first tensor
    double* st_gram;
    double* st_coef;
};

// ---------------------------------------------------------------------------
// element access
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t b16) {
    return __uint_as_float(b16 << 16);
}
__device__ __forceinline__ uint32_t key_of(float tau) {
    return __float_as_uint(tau) & 0x7FFFFFFFu;
}

// 8 consecutive entries (16-byte aligned start) of a tensor as binary32.
template <typename T> struct Load8;
template <> struct Load8<__nv_bfloat16> {
    static __device__ __forceinline__ void run(const void* p, long long e, float (&v)[8]) {
        uint4 u = __ldg(reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p) + e));
        v[0] = bf16_bits_to_f32(u.x & 0xFFFFu); v[1] = bf16_bits_to_f32(u.x >> 16);
        v[2] = bf16_bits_to_f32(u.y & 0xFFFFu); v[3] = bf16_bits_to_f32(u.y >> 16);
        v[4] = bf16_bits_to_f32(u.z & 0xFFFFu); v[5] = bf16_bits_to_f32(u.z >> 16);
        v[6] = bf16_bits_to_f32(u.w & 0xFFFFu); v[7] = bf16_bits_to_f32(u.w >> 16);
    }
    static __device__ __forceinline__ float one(const void* p, long long e) {
        return bf16_bits_to_f32(static_cast<const unsigned short*>(p)[e]);
    }
};
template <> struct Load8<float> {
    static __device__ __forceinline__ void run(const void* p, long long e, float (&v)[8]) {
        const float4* q = reinterpret_cast<const float4*>(static_cast<const float*>(p) + e);
        float4 a = __ldg(q), b = __ldg(q + 1);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    static __device__ __forceinline__ float one(const void* p, long long e) {
        return static_cast<const float*>(p)[e];
    }
};

// Task-vector source: tau = x (delta) or x - base (checkpoint), binary32.
template <typename XT, typename BT, bool CKPT>
struct TauSrc {
    // 8 entries starting at e (e % 8 == 0); entries at or beyond n read as 0
    static __device__ __forceinline__ void load8(const void* x, const void* base, long long e,
                                                 long long n, float (&tau)[8]) {
        if (e + 8 <= n) {
            Load8<XT>::run(x, e, tau);
            if (CKPT) {
                float b[8];
                Load8<BT>::run(base, e, b);
#pragma unroll
                for (int j = 0; j < 8; ++j) tau[j] = __fsub_rn(tau[j], b[j]);
            }
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                float v = 0.0f;
                if (e + j < n) {
                    v = Load8<XT>::one(x, e + j);
                    if (CKPT) v = __fsub_rn(v, Load8<BT>::one(base, e + j));
                }
                tau[j] = v;
            }
        }
    }
    static __device__ __forceinline__ float load1(const void* x, const void* base, long long e) {
        float v = Load8<XT>::one(x, e);
        if (CKPT) v = __fsub_rn(v, Load8<BT>::one(base, e));
        return v;
    }
};

// ---------------------------------------------------------------------------
// streaming loads / stores
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
    return r;
}

template <typename T> struct Lanes;   // uint4 words per 8 entries
template <> struct Lanes<__nv_bfloat16> { static constexpr int N = 1; };
template <> struct Lanes<float> { static constexpr int N = 2; };

// 8 entries (start e, e % 8 == 0) as raw words; entries at or beyond n read as 0
template <typename T>
__device__ __forceinline__ void load_raw8(const void* p, long long e, long long n, uint4 (&w)[Lanes<T>::N]) {
    if (e + 8 <= n) {
#pragma unroll
        for (int q = 0; q < Lanes<T>::N; ++q)
            w[q] = ld_stream(static_cast<const char*>(p) + (e * sizeof(T)) + 16 * q);
    } else {
        uint32_t u[4 * Lanes<T>::N];
#pragma unroll
        for (int q = 0; q < 4 * Lanes<T>::N; ++q) u[q] = 0;
        if (sizeof(T) == 2) {
            const unsigned short* s = static_cast<const unsigned short*>(p);
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (e + j < n) u[j >> 1] |= (uint32_t)s[e + j] << (16 * (j & 1));
        } else {
            const uint32_t* s = static_cast<const uint32_t*>(p);
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (e + j < n) u[j] = s[e + j];
        }
#pragma unroll
        for (int q = 0; q < Lanes<T>::N; ++q) w[q] = make_uint4(u[4 * q], u[4 * q + 1], u[4 * q + 2], u[4 * q + 3]);
    }
}

template <typename T>
__device__ __forceinline__ void raw_to_f32(const uint4 (&w)[Lanes<T>::N], float (&v)[8]) {
    if (sizeof(T) == 2) {
        const uint32_t u[4] = {w[0].x, w[0].y, w[0].z, w[0].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[2 * j] = __uint_as_float(u[j] << 16);
            v[2 * j + 1] = __uint_as_float(u[j] & 0xFFFF0000u);
        }
    } else {
#pragma unroll
        for (int q = 0; q < Lanes<T>::N; ++q) {
            v[4 * q] = __uint_as_float(w[q].x); v[4 * q + 1] = __uint_as_float(w[q].y);
            v[4 * q + 2] = __uint_as_float(w[q].z); v[4 * q + 3] = __uint_as_float(w[q].w);
        }
    }
}

// One lane's share of a tile of a task-vector source, as raw words, so the
// next tile's loads can be in flight while the current one is processed.
template <typename XT, typename BT, bool CK>
struct RawTile {
    static constexpr int NX = Lanes<XT>::N;
    static constexpr int NB = CK ? Lanes<BT>::N : 1;
    uint4 x[WVEC][NX];
    uint4 b[WVEC][NB];
    __device__ __forceinline__ void load(const void* xp, const void* bp, long long e0, long long n, int lane) {
#pragma unroll
        for (int v = 0; v < WVEC; ++v) {
            const long long e = e0 + v * (32 * VEC) + lane * VEC;
            if (e < n) {
                load_raw8<XT>(xp, e, n, x[v]);
                if (CK) load_raw8<BT>(bp, e, n, reinterpret_cast<uint4(&)[Lanes<BT>::N]>(b[v]));
            } else {
#pragma unroll
                for (int q = 0; q < NX; ++q) x[v][q] = make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int q = 0; q < NB; ++q) b[v][q] = make_uint4(0, 0, 0, 0);
            }
        }
    }
    // vector step v of the tile starting at tensor entry e0, with rem = numel - e0
    // entries left in the tensor (32-bit offsets; no bounds tests on a whole tile)
    __device__ __forceinline__ void load_step(int v, const void* xp, const void* bp, uint32_t e0,
                                              uint32_t rem, int lane) {
        const uint32_t o = (uint32_t)(v * (32 * VEC) + lane * VEC);
        if (rem >= TILE) {
            const char* xq = static_cast<const char*>(xp) + ((size_t)e0 + o) * sizeof(XT);
#pragma unroll
            for (int q = 0; q < NX; ++q) x[v][q] = ld_stream(xq + 16 * q);
            if (CK) {
                const char* bq = static_cast<const char*>(bp) + ((size_t)e0 + o) * sizeof(BT);
#pragma unroll
                for (int q = 0; q < NB; ++q) b[v][q] = ld_stream(bq + 16 * q);
            }
        } else if (o < rem) {
            load_raw8<XT>(xp, (long long)e0 + o, (long long)e0 + rem, x[v]);
            if (CK) load_raw8<BT>(bp, (long long)e0 + o, (long long)e0 + rem,
                                  reinterpret_cast<uint4(&)[Lanes<BT>::N]>(b[v]));
        } else {
#pragma unroll
            for (int q = 0; q < NX; ++q) x[v][q] = make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int q = 0; q < NB; ++q) b[v][q] = make_uint4(0, 0, 0, 0);
        }
    }
    // tau = x (delta) or x - base (checkpoint), binary32
    __device__ __forceinline__ void tau(int v, float (&t)[8]) const {
        raw_to_f32<XT>(x[v], t);
        if (CK) {
            float bb[8];
            raw_to_f32<BT>(reinterpret_cast<const uint4(&)[Lanes<BT>::N]>(b[v]), bb);
#pragma unroll
            for (int j = 0; j < 8; ++j) t[j] = __fsub_rn(t[j], bb[j]);
        }
    }
};

template <typename T>
__device__ __forceinline__ T warp_excl_scan(T v, T* total) {
    const int lane = threadIdx.x & 31;
    T x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        T y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
    }
    *total = __shfl_sync(0xFFFFFFFFu, x, 31);
    return x - v;
}

// tile id -> tensor (binary search over tile_base)
__device__ __forceinline__ int tensor_of_tile(const TensorDesc* tens, int n_tensors, long long tile) {
    int lo = 0, hi = n_tensors - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (tens[mid].tile_base <= tile) lo = mid; else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ void set_status(Header* h, int32_t code) {
    atomicCAS(&h->status, 0, code);
}

// ---------------------------------------------------------------------------
// block-wide helpers (blockDim.x a multiple of 32, <= 1024)
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

// Sum over the block; result valid in every thread.  `sm` needs 32 slots.
template <typename T>
__device__ __forceinline__ T block_sum(T v, T* sm) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) sm[warp] = v;
    __syncthreads();
    const int nw = (blockDim.x + 31) >> 5;
    T r = (lane < nw) ? sm[lane] : T(0);
    r = warp_sum(r);
    return r;
}

// Exclusive prefix over the block in thread order; *total receives the sum.
// `sm` needs 33 slots.
template <typename T>
__device__ __forceinline__ T block_excl_scan(T v, T* sm, T* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    T x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        T y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();
    if (lane == 31) sm[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const int nw = (blockDim.x + 31) >> 5;
        T w = (lane < nw) ? sm[lane] : T(0);
        T s = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            T y = __shfl_up_sync(0xFFFFFFFFu, s, o);
            if (lane >= o) s += y;
        }
        if (lane < nw) sm[lane] = s - w;   // exclusive warp offsets
        if (lane == nw - 1) sm[32] = s;
    }
    __syncthreads();
    T r = sm[warp] + x - v;
    *total = sm[32];
    return r;
}

// ---------------------------------------------------------------------------
// selection helpers shared by the select and fused passes
// ---------------------------------------------------------------------------
__device__ __forceinline__ long long k_of_density(double rho, long long n) {
    // floor(rho n + 1/2) with IEEE products and sums (no contraction)
    double kk = floor(__dadd_rn(__dmul_rn(rho, (double)n), 0.5));
    if (kk < 0.0) kk = 0.0;
    if (kk > (double)n) kk = (double)n;
    return (long long)kk;
}

// s + e += x exactly as a binary32 pair (Knuth's two-sum: the rounding
// error of s + x is carried in e)
__device__ __forceinline__ void two_sum_add(float& s, float& e, float x) {
    const float t = __fadd_rn(s, x);
    const float bp = __fsub_rn(t, s);
    const float err = __fadd_rn(__fsub_rn(s, __fsub_rn(t, bp)), __fsub_rn(x, bp));
    s = t;
    e = __fadd_rn(e, err);
}

__device__ __forceinline__ int bitlen32(uint32_t v) { return v ? 32 - __clz(v) : 0; }

__device__ __forceinline__ double sq(uint32_t key) {
    const double f = (double)__uint_as_float(key);
    return f * f;
}

// ---------------------------------------------------------------------------
// (expert, tile) item cursor: items are expert-major, tiles in tensor order
// ---------------------------------------------------------------------------
struct Cursor {
    long long it;        // current item
    long long run_end;   // first item after the current (expert, tensor) run
    long long g;         // tile
    int i, t;            // expert, tensor
};

__device__ __forceinline__ void cursor_at(const Plan& P, long long it, Cursor& c) {
    c.it = it;
    c.i = (int)(it / P.n_tiles);
    c.g = it - (long long)c.i * P.n_tiles;
    c.t = tensor_of_tile(P.tens, P.n_tensors, c.g);
    const TensorDesc& d = P.tens[c.t];
    c.run_end = (long long)c.i * P.n_tiles + d.tile_base + (d.numel + TILE - 1) / TILE;
}

__device__ __forceinline__ Unit* unit_of(const Plan& P, int i, const TensorDesc& d) {
    const int u = (P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit;
    return &P.units[(long long)i * P.n_units + u];
}

__device__ __forceinline__ Unit* count_unit(const Plan& P, const Cursor& c) {
    const TensorDesc& d = P.tens[c.t];
    if (!(d.flags & TF_TRIM)) return nullptr;
    Unit* U = unit_of(P, c.i, d);
    return (U->state == ST_BAND) ? U : nullptr;
}

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

// ---------------------------------------------------------------------------
// per-entry selection
// ---------------------------------------------------------------------------
struct SelParam { uint32_t t; long long cut; };

__device__ __forceinline__ bool kept(uint32_t key, long long pos, const SelParam& s) {
    return key > s.t || (key == s.t && pos < s.cut);
}

__device__ __forceinline__ void store8(void* p, long long e, long long n, const float (&v)[8], bool bf16) {
    if (bf16) {
        __nv_bfloat16* q = static_cast<__nv_bfloat16*>(p) + e;
        if (e + 8 <= n) {
            __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]);
            __nv_bfloat162 b = __floats2bfloat162_rn(v[2], v[3]);
            __nv_bfloat162 c = __floats2bfloat162_rn(v[4], v[5]);
            __nv_bfloat162 d = __floats2bfloat162_rn(v[6], v[7]);
            uint4 u;
            u.x = *reinterpret_cast<uint32_t*>(&a); u.y = *reinterpret_cast<uint32_t*>(&b);
            u.z = *reinterpret_cast<uint32_t*>(&c); u.w = *reinterpret_cast<uint32_t*>(&d);
            __stcs(reinterpret_cast<uint4*>(q), u);
        } else {
            for (int j = 0; j < 8; ++j)
                if (e + j < n) q[j] = __float2bfloat16_rn(v[j]);
        }
    } else {
        float* q = static_cast<float*>(p) + e;
        if (e + 8 <= n) {
            __stcs(reinterpret_cast<float4*>(q), make_float4(v[0], v[1], v[2], v[3]));
            __stcs(reinterpret_cast<float4*>(q) + 1, make_float4(v[4], v[5], v[6], v[7]));
        } else {
            for (int j = 0; j < 8; ++j)
                if (e + j < n) q[j] = v[j];
        }
    }
}

// the coefficient a unit has unless its retention system is degenerate:
// lambda for TIES; for ISO clip(Gamma / (Gamma + ridge)) rounds to
// clip(1, c_min, c_max) in binary32 whenever Gamma >= 2^25 ridge
__device__ __forceinline__ float k1_spec_coef(const Plan& P) {
    if (P.op == ISO_OP_ISO) return (float)fmin(fmax(1.0, P.c_min), P.c_max);
    return P.lambda;
}

// Two binary32 operations in one packed instruction (sm_100 and later): each
// half rounds to nearest like the scalar __fsub_rn / __fmul_rn / __fadd_rn,
// subnormals kept.
__device__ __forceinline__ void sub_rn2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
    asm("{\n\t.reg .b64 pa, pb, pd;\n\tmov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
        "sub.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
__device__ __forceinline__ void mul_rn2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
    asm("{\n\t.reg .b64 pa, pb, pd;\n\tmov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
        "mul.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
__device__ __forceinline__ void add_rn2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
    asm("{\n\t.reg .b64 pa, pb, pd;\n\tmov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
        "add.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(d0), "=f"(d1) : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}

// ---------------------------------------------------------------------------
// bulk copies into shared memory tracked by an mbarrier (sm_90 and later)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
// make the initialised barriers visible to the asynchronous proxy
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// one arrival that also announces `bytes` of transactions for the phase
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
// true once the phase with the given parity has completed; one probe, which
// may suspend the thread for at most MBAR_PROBE_NS nanoseconds (the thread is
// resumed early when the phase completes)
constexpr uint32_t MBAR_PROBE_NS = 1000;
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok) : "r"(bar), "r"(parity), "n"(MBAR_PROBE_NS) : "memory");
    return ok != 0;
}
// bytes (a multiple of 16) from global memory of this GPU to shared memory,
// both 16-byte aligned; completion is counted on the barrier's transactions
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// order this thread's earlier shared-memory accesses before its later
// bulk copies (asynchronous proxy) into the same memory
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// probes of one barrier phase before a wait gives up: at most about four
// seconds of suspension in all
constexpr int MBAR_SPIN_LIMIT = 1 << 22;

// Retention coefficients (Sec. 4.2; App. E, Retention coefficients): on the
// experts with Gamma_ii > 0, (Gamma + ridge I) c = diag(Gamma) by Gaussian
// elimination with partial pivoting in binary64, clipped to [c_min, c_max];
// an expert with Gamma_ii = 0 gets c = 0.  G is K x K row-major (K <= MAXK).
__device__ __forceinline__ void retention_solve(const double* G, int K, double ridge, double c_min,
                                                double c_max, double* c) {
    for (int i = 0; i < K; ++i) c[i] = 0.0;
    int idx[MAXK];
    int m = 0;
    for (int i = 0; i < K; ++i)
        if (G[i * K + i] > 0.0) idx[m++] = i;
    double A[MAXK * MAXK], rhs[MAXK], x[MAXK];
    for (int r = 0; r < m; ++r) {
        for (int q = 0; q < m; ++q) A[r * m + q] = G[idx[r] * K + idx[q]];
        A[r * m + r] = __dadd_rn(A[r * m + r], ridge);
        rhs[r] = G[idx[r] * K + idx[r]];
    }
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
        if (v < c_min) v = c_min;
        if (v > c_max) v = c_max;
        c[idx[r]] = v;
    }
}

__device__ __forceinline__ float out_of(float th0, float tau, float a) {
    const float upd = __fmul_rn(a, tau);
    return (upd == 0.0f) ? th0 : __fadd_rn(th0, upd);
}

}  // namespace iso
