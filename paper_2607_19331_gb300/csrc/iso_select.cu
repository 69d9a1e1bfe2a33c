// iso_select.cu -- exact TopKMask threshold per selection unit (TENSOR and
// GLOBAL scope).
//
// TopKMask(|tau|, rho) keeps the k = floor(rho n + 1/2) entries of largest
// |tau| (App. F, TIES trim); ties go to the lowest position.  The result of
// this file is, per unit, a threshold key t and a position cut such that
//     kept(p)  <=>  key(p) > t  ||  (key(p) == t && pos(p) < cut)
// which the streaming passes then apply as a pure per-entry predicate.
//
// Pipeline (all launches on the caller's stream, no waits between blocks):
//   k_sample   keys at evenly spaced chunks -> band [lo, hi] around rank k
//   k_count    one full read: #key > hi, #key == hi / == lo per tile, and the
//              interior keys lo < key < hi appended to the unit's segment
//   k_decide   locate rank k among the counters; a miss (or an overflowing
//              segment) switches the unit to a radix select over its data
//   k_radix_*  up to three 11-bit radix levels over the interior keys (or
//              over the whole unit on the fallback path)
//   k_tie      per-tile counts of keys == t where needed, and the sum of
//              squares of the kept entries (ISO, K = 1)
//   k_cut      the tile holding the need-th tie, then the exact position
#include "iso_internal.cuh"

namespace iso {

__device__ __forceinline__ long long k_of_density(double rho, long long n) {
    // floor(rho n + 1/2) with IEEE products and sums (no contraction)
    double kk = floor(__dadd_rn(__dmul_rn(rho, (double)n), 0.5));
    if (kk < 0.0) kk = 0.0;
    if (kk > (double)n) kk = (double)n;
    return (long long)kk;
}

__device__ __forceinline__ int bitlen32(uint32_t v) { return v ? 32 - __clz(v) : 0; }

// ---------------------------------------------------------------------------
// unit table
// ---------------------------------------------------------------------------
__global__ void k_init_units(Plan P, long long global_n) {
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= P.K * P.n_units) return;
    const int i = idx / P.n_units, u = idx % P.n_units;
    Unit& U = P.units[idx];
    U.expert = i;
    U.want_gamma = (P.op == ISO_OP_ISO && P.K == 1 && P.scope == ISO_SCOPE_TENSOR) ? 1 : 0;
    U.t = KEY_NONE;
    U.cut = 0;
    bool trimmed;
    if (P.scope == ISO_SCOPE_GLOBAL) {
        U.tensor = -1;
        U.n = global_n;
        U.tile_begin = 0;
        U.tile_end = P.n_tiles;
        U.cand_cap = P.tens[0].cand_cap;
        U.cand_off = P.tens[0].cand_off + (unsigned long long)i * U.cand_cap;
        trimmed = global_n > 0;
    } else {
        const TensorDesc& d = P.tens[u];
        U.tensor = u;
        U.n = d.numel;
        U.tile_begin = d.tile_base;
        U.tile_end = d.tile_base + (d.numel + TILE - 1) / TILE;
        U.cand_cap = d.cand_cap;
        U.cand_off = d.cand_off + (unsigned long long)i * d.cand_cap;
        trimmed = (d.flags & TF_TRIM) != 0;
    }
    if (!trimmed) {
        U.state = ST_OFF;
        U.k = -1;
        U.t = 0;          // key >= 0 always: every entry kept
        U.cut = CUT_ALL;
        return;
    }
    U.k = k_of_density(P.density, U.n);
    if (U.k == 0) {
        U.state = ST_NONE;
        return;
    }
    U.state = ST_SAMPLE;
}

// ---------------------------------------------------------------------------
// block-level radix select in shared memory
// ---------------------------------------------------------------------------

// Find, among nb bins taken from the top, the bin b with
// above(b) < rank <= above(b) + hist[b].  Result broadcast through `res`.
__device__ void block_find_from_top(const uint32_t* hist, int nb, long long rank,
                                    long long* sm_scan, int* res_bin, long long* res_above) {
    const int per = (nb + blockDim.x - 1) / blockDim.x;
    const int j0 = threadIdx.x * per;
    if (threadIdx.x == 0) { *res_bin = 0; *res_above = 0; }   // ordered by the scan's barriers
    long long local = 0;
    for (int j = j0; j < j0 + per && j < nb; ++j) local += hist[nb - 1 - j];
    long long total;
    long long excl = block_excl_scan(local, sm_scan, &total);
    if (excl < rank && rank <= excl + local) {
        long long acc = excl;
        for (int j = j0; j < j0 + per && j < nb; ++j) {
            uint32_t h = hist[nb - 1 - j];
            if (rank <= acc + h) { *res_bin = nb - 1 - j; *res_above = acc; break; }
            acc += h;
        }
    }
    __syncthreads();
}

// k-th largest (1-based rank) of the n keys in shared memory.
__device__ uint32_t block_kth_largest(const uint32_t* keys, int n, long long rank, uint32_t* hist,
                                      long long* sm_scan, int* sm_bin, long long* sm_above) {
    uint32_t prefix = 0;
    int pshift = 31;
    for (;;) {
        const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
        const int nb = 1 << (pshift - shift);
        for (int b = threadIdx.x; b < nb; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        for (int p = threadIdx.x; p < n; p += blockDim.x) {
            uint32_t v = keys[p];
            if ((v >> pshift) == prefix) atomicAdd(&hist[(v >> shift) & (nb - 1)], 1u);
        }
        __syncthreads();
        block_find_from_top(hist, nb, rank, sm_scan, sm_bin, sm_above);
        const int b = *sm_bin;
        rank -= *sm_above;
        prefix = (prefix << (pshift - shift)) | (uint32_t)b;
        __syncthreads();
        if (shift == 0) return prefix;
        pshift = shift;
    }
}

// ---------------------------------------------------------------------------
// sample -> band
// ---------------------------------------------------------------------------

// unit position -> (tensor, entry) for GLOBAL scope: last tensor with uoff <= pos
__device__ __forceinline__ int tensor_of_upos(const TensorDesc* tens, int n_tensors, long long pos) {
    int lo = 0, hi = n_tensors - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (tens[mid].uoff <= pos) lo = mid; else hi = mid - 1;
    }
    return lo;
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(SAMPLE_TPB) k_sample(Plan P) {
    extern __shared__ __align__(16) uint32_t s_keys[];
    uint32_t* s_hist = s_keys + SAMPLE_MAX;
    __shared__ long long s_scan[33];
    __shared__ int s_bin;
    __shared__ long long s_above;

    Unit& U = P.units[blockIdx.x];
    if (U.state != ST_SAMPLE) return;
    const int i = U.expert;
    const long long n = U.n;
    const int S = (int)(n < SAMPLE_MAX ? n : SAMPLE_MAX);
    const int nch = SAMPLE_MAX / SAMPLE_CHUNK;
    for (int q = threadIdx.x; q < S; q += blockDim.x) {
        long long pos;
        if (S == n) {
            pos = q;
        } else {
            const int c = q / SAMPLE_CHUNK, j = q % SAMPLE_CHUNK;
            pos = (long long)((double)(n - SAMPLE_CHUNK) * c / (nch - 1)) + j;
        }
        int t;
        long long e;
        if (P.scope == ISO_SCOPE_GLOBAL) {
            t = tensor_of_upos(P.tens, P.n_tensors, pos);
            e = pos - P.tens[t].uoff;
        } else {
            t = U.tensor;
            e = pos;
        }
        const float tau = TauSrc<XT, BT, CKPT>::load1(P.xptr[i * P.n_tensors + t], P.tens[t].base, e);
        s_keys[q] = key_of(tau);
    }
    __syncthreads();
    uint32_t lo, hi;
    if (S == n) {
        // the sample is the whole unit: the band is the exact threshold
        hi = block_kth_largest(s_keys, S, U.k, s_hist, s_scan, &s_bin, &s_above);
        lo = hi;
    } else {
        const double q = (double)U.k / (double)n;
        const double r = (double)U.k * (double)S / (double)n;
        const double delta = SAMPLE_Z * sqrt((double)S * q * (1.0 - q)) + 2.0;
        const long long ra = (long long)floor(r - delta);
        const long long rb = (long long)ceil(r + delta);
        hi = (ra >= 1) ? block_kth_largest(s_keys, S, ra, s_hist, s_scan, &s_bin, &s_above) : KEY_MAX;
        lo = (rb <= S) ? block_kth_largest(s_keys, S, rb, s_hist, s_scan, &s_bin, &s_above) : 0u;
    }
    if (threadIdx.x == 0) {
        U.lo = lo;
        U.hi = hi;
        U.state = ST_BAND;
    }
}

// ---------------------------------------------------------------------------
// count pass: one full read per unit
// ---------------------------------------------------------------------------
__device__ __forceinline__ Unit* unit_of_tile(const Plan& P, int i, const TensorDesc& d) {
    const int u = (P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit;
    return &P.units[(long long)i * P.n_units + u];
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(TPB) k_count(Plan P) {
    __shared__ unsigned long long s_red[33];
    __shared__ uint32_t s_scan[33];
    __shared__ double s_dred[33];
    __shared__ uint32_t s_slot;
    __shared__ int s_ok;

    const long long items = (long long)P.K * P.n_tiles;
    for (long long it = blockIdx.x; it < items; it += gridDim.x) {
        const int i = (int)(it / P.n_tiles);
        const long long g = it % P.n_tiles;
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        if (!(d.flags & TF_TRIM)) continue;
        Unit* U = unit_of_tile(P, i, d);
        if (U->state != ST_BAND) continue;
        const uint32_t lo = U->lo, hi = U->hi;
        const bool want_gamma = U->want_gamma != 0;
        const void* x = P.xptr[i * P.n_tensors + t];
        const long long e0 = (g - d.tile_base) * TILE;
        const long long n = d.numel;

        uint32_t keys[NVEC][VEC];
        uint32_t n_gt = 0, n_hi = 0, n_lo = 0, n_int = 0;
        bool bad = false;
        double gacc = 0.0;
#pragma unroll
        for (int v = 0; v < NVEC; ++v) {
            const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
            float tau[VEC];
            if (e < n) {
                TauSrc<XT, BT, CKPT>::load8(x, d.base, e, n, tau);
            } else {
#pragma unroll
                for (int j = 0; j < VEC; ++j) tau[j] = 0.0f;
            }
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const uint32_t kk = key_of(tau[j]);
                const bool valid = e + j < n;
                keys[v][j] = valid ? kk : 0xFFFFFFFFu;   // sentinel: not counted
                if (!valid) continue;
                bad |= kk >= KEY_INF;
                if (kk > hi) {
                    n_gt++;
                    if (want_gamma) gacc += (double)tau[j] * (double)tau[j];
                } else if (kk == hi) n_hi++;
                else if (kk == lo) n_lo++;
                else if (kk > lo) n_int++;
            }
        }
        if (bad) set_status(P.hdr, ISO_ERR_NONFINITE);
        unsigned long long packed = (unsigned long long)n_gt | ((unsigned long long)n_hi << 16) |
                                    ((unsigned long long)n_lo << 32) | ((unsigned long long)n_int << 48);
        uint32_t int_total;
        const uint32_t my_off = block_excl_scan(n_int, s_scan, &int_total);
        const unsigned long long tot = block_sum(packed, s_red);
        double gtot = 0.0;
        if (want_gamma) gtot = block_sum(gacc, s_dred);
        if (threadIdx.x == 0) {
            const uint32_t t_gt = (uint32_t)(tot & 0xFFFF), t_hi = (uint32_t)((tot >> 16) & 0xFFFF);
            const uint32_t t_lo = (uint32_t)((tot >> 32) & 0xFFFF);
            if (t_gt) atomicAdd(&U->c_gt, (unsigned long long)t_gt);
            if (t_hi) atomicAdd(&U->c_hi, (unsigned long long)t_hi);
            if (t_lo) atomicAdd(&U->c_lo, (unsigned long long)t_lo);
            if (want_gamma && gtot != 0.0) atomicAdd(&U->gamma_acc, gtot);
            unsigned long long slot = 0;
            if (int_total) slot = atomicAdd(&U->n_int, (unsigned long long)int_total);
            const int ok = (slot + int_total <= U->cand_cap) ? 1 : 0;
            TileRec r;
            r.start = (uint32_t)slot;
            r.count = ok ? int_total : 0u;
            r.eq_lo = t_lo;
            r.eq_hi = t_hi;
            P.trec[(long long)i * P.n_tiles + g] = r;
            s_slot = (uint32_t)slot;
            s_ok = ok;
        }
        __syncthreads();
        if (s_ok && n_int) {
            uint32_t* dst = P.cand + U->cand_off + s_slot + my_off;
            uint32_t w = 0;
#pragma unroll
            for (int v = 0; v < NVEC; ++v)
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    const uint32_t kk = keys[v][j];
                    if (kk != 0xFFFFFFFFu && kk < hi && kk > lo) dst[w++] = kk;
                }
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// decide: where is rank k relative to the band?
// ---------------------------------------------------------------------------
__global__ void k_decide(Plan P) {
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= P.K * P.n_units) return;
    Unit& U = P.units[idx];
    if (U.state != ST_BAND) return;
    const long long c_gt = (long long)U.c_gt, c_hi = (long long)U.c_hi;
    const long long c_lo = (long long)U.c_lo, n_int = (long long)U.n_int;
    long long r = U.k - c_gt;
    bool miss = false;
    if (r <= 0) {
        miss = true;
    } else if (r <= c_hi) {
        U.t = U.hi; U.count_above = c_gt; U.ties = c_hi; U.need = r; U.tie_src = TIE_EQ_HI;
        U.r_src = SRC_CAND;
        U.state = ST_TKNOWN;
    } else {
        r -= c_hi;
        if (r <= n_int) {
            if ((unsigned long long)n_int > U.cand_cap) {
                miss = true;
            } else {
                U.r_src = SRC_CAND;
                U.r_base = U.lo;
                U.r_pshift = bitlen32(U.hi - U.lo);
                U.r_prefix = 0;
                U.r_rank = r;
                U.r_above = c_gt + c_hi;
                U.state = ST_RADIX;
            }
        } else {
            r -= n_int;
            if (r <= c_lo) {
                U.t = U.lo; U.count_above = c_gt + c_hi + n_int; U.ties = c_lo; U.need = r;
                U.tie_src = TIE_EQ_LO;
                U.r_src = SRC_CAND;
                U.state = ST_TKNOWN;
            } else {
                miss = true;
            }
        }
    }
    if (miss) {
        // exact fallback: radix select over every entry of the unit
        U.fallback = 1;
        U.gamma_acc = 0.0;
        U.r_src = SRC_DATA;
        U.r_base = 0;
        U.r_pshift = 31;
        U.r_prefix = 0;
        U.r_rank = U.k;
        U.r_above = 0;
        U.state = ST_RADIX;
    }
    if (U.state == ST_RADIX) atomicAdd(&P.hdr->n_radix, 1);
    else atomicAdd(&P.hdr->n_tknown, 1);
}

// ---------------------------------------------------------------------------
// radix levels
// ---------------------------------------------------------------------------
template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(TPB) k_radix_hist(Plan P) {
    __shared__ uint32_t s_hist[RADIX_BINS];
    if (*(volatile int32_t*)&P.hdr->n_radix == 0) return;
    const long long items = (long long)P.K * P.n_tiles;
    const long long per = (items + gridDim.x - 1) / gridDim.x;
    const long long it0 = blockIdx.x * per;
    const long long it1 = (it0 + per < items) ? it0 + per : items;
    long long cur = -1;
    int cur_nb = 0;
    for (int b = threadIdx.x; b < RADIX_BINS; b += blockDim.x) s_hist[b] = 0;
    __syncthreads();
    for (long long it = it0; it < it1; ++it) {
        const int i = (int)(it / P.n_tiles);
        const long long g = it % P.n_tiles;
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        if (!(d.flags & TF_TRIM)) continue;
        Unit* U = unit_of_tile(P, i, d);
        if (U->state != ST_RADIX) continue;
        const long long ui = U - P.units;
        const int pshift = U->r_pshift;
        const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
        const int nb = 1 << (pshift - shift);
        if (ui != cur) {
            __syncthreads();
            if (cur >= 0)
                for (int b = threadIdx.x; b < cur_nb; b += blockDim.x)
                    if (s_hist[b]) { atomicAdd(&P.hist[cur * RADIX_BINS + b], s_hist[b]); s_hist[b] = 0; }
            __syncthreads();
            cur = ui;
            cur_nb = nb;
        }
        const uint32_t base = U->r_base, prefix = U->r_prefix;
        if (U->r_src == SRC_CAND) {
            const TileRec r = P.trec[(long long)i * P.n_tiles + g];
            const uint32_t* c = P.cand + U->cand_off + r.start;
            for (uint32_t j = threadIdx.x; j < r.count; j += blockDim.x) {
                const uint32_t v = c[j] - base;
                if ((v >> pshift) == prefix) atomicAdd(&s_hist[(v >> shift) & (nb - 1)], 1u);
            }
        } else {
            const void* x = P.xptr[i * P.n_tensors + t];
            const long long e0 = (g - d.tile_base) * TILE;
#pragma unroll
            for (int v = 0; v < NVEC; ++v) {
                const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
                if (e >= d.numel) continue;
                float tau[VEC];
                TauSrc<XT, BT, CKPT>::load8(x, d.base, e, d.numel, tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    if (e + j >= d.numel) continue;
                    const uint32_t kk = key_of(tau[j]);
                    if ((kk >> pshift) == prefix) atomicAdd(&s_hist[(kk >> shift) & (nb - 1)], 1u);
                }
            }
        }
    }
    __syncthreads();
    if (cur >= 0)
        for (int b = threadIdx.x; b < cur_nb; b += blockDim.x)
            if (s_hist[b]) atomicAdd(&P.hist[cur * RADIX_BINS + b], s_hist[b]);
}

__global__ void __launch_bounds__(TPB) k_radix_pick(Plan P) {
    __shared__ long long s_scan[33];
    __shared__ int s_bin;
    __shared__ long long s_above;
    Unit& U = P.units[blockIdx.x];
    if (U.state != ST_RADIX) return;
    uint32_t* h = P.hist + (long long)blockIdx.x * RADIX_BINS;
    const int pshift = U.r_pshift;
    const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
    const int nb = 1 << (pshift - shift);
    block_find_from_top(h, nb, U.r_rank, s_scan, &s_bin, &s_above);
    const int b = s_bin;
    const long long above = s_above;
    const uint32_t cnt = h[b];
    __syncthreads();
    for (int q = threadIdx.x; q < nb; q += blockDim.x) h[q] = 0;
    if (threadIdx.x == 0) {
        U.r_rank -= above;
        U.r_above += above;
        U.r_prefix = (U.r_prefix << (pshift - shift)) | (uint32_t)b;
        if (shift == 0) {
            U.t = U.r_base + U.r_prefix;
            U.count_above = U.r_above;
            U.ties = cnt;
            U.need = U.r_rank;
            U.tie_src = TIE_ARRAY;
            U.state = ST_TKNOWN;
            atomicSub(&P.hdr->n_radix, 1);
            atomicAdd(&P.hdr->n_tknown, 1);
        } else {
            U.r_pshift = shift;
        }
    }
}

// ---------------------------------------------------------------------------
// ties per tile and the sum of squares of the kept entries
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool tie_pass_needed(const Unit& U, bool* count, bool* gamma) {
    *count = (U.tie_src == TIE_ARRAY) && (U.need < U.ties);
    *gamma = U.want_gamma && (U.tie_src != TIE_EQ_HI);
    return *count || *gamma;
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(TPB) k_tie(Plan P) {
    __shared__ uint32_t s_red[33];
    __shared__ double s_dred[33];
    if (*(volatile int32_t*)&P.hdr->n_tknown == 0) return;
    const long long items = (long long)P.K * P.n_tiles;
    for (long long it = blockIdx.x; it < items; it += gridDim.x) {
        const int i = (int)(it / P.n_tiles);
        const long long g = it % P.n_tiles;
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        if (!(d.flags & TF_TRIM)) continue;
        Unit* U = unit_of_tile(P, i, d);
        if (U->state != ST_TKNOWN) continue;
        bool want_count, want_gamma;
        if (!tie_pass_needed(*U, &want_count, &want_gamma)) continue;
        const uint32_t tk = U->t;
        uint32_t cnt = 0;
        double gacc = 0.0;
        if (U->r_src == SRC_CAND) {
            const TileRec r = P.trec[(long long)i * P.n_tiles + g];
            const uint32_t* c = P.cand + U->cand_off + r.start;
            for (uint32_t j = threadIdx.x; j < r.count; j += blockDim.x) {
                const uint32_t kk = c[j];
                cnt += (kk == tk);
                if (want_gamma && kk > tk) {
                    const double f = (double)__uint_as_float(kk);
                    gacc += f * f;
                }
            }
        } else {
            const void* x = P.xptr[i * P.n_tensors + t];
            const long long e0 = (g - d.tile_base) * TILE;
#pragma unroll
            for (int v = 0; v < NVEC; ++v) {
                const long long e = e0 + v * (TPB * VEC) + threadIdx.x * VEC;
                if (e >= d.numel) continue;
                float tau[VEC];
                TauSrc<XT, BT, CKPT>::load8(x, d.base, e, d.numel, tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    if (e + j >= d.numel) continue;
                    const uint32_t kk = key_of(tau[j]);
                    cnt += (kk == tk);
                    if (want_gamma && kk > tk) gacc += (double)tau[j] * (double)tau[j];
                }
            }
        }
        if (want_count) {
            const uint32_t tot = block_sum(cnt, s_red);
            if (threadIdx.x == 0) P.tcnt[(long long)i * P.n_tiles + g] = tot;
        }
        if (want_gamma) {
            const double gt = block_sum(gacc, s_dred);
            if (threadIdx.x == 0 && gt != 0.0) atomicAdd(&U->gamma_acc2, gt);
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// cut: position of the need-th tie, stats, gamma
// ---------------------------------------------------------------------------
__device__ __forceinline__ void write_unit_stats(const Plan& P, int idx, const Unit& U) {
    if (!P.st_units) return;
    const int i = idx / P.n_units, u = idx % P.n_units;
    iso_unit_stats s;
    s.thresh_key = (U.state == ST_OFF) ? KEY_NONE : U.t;
    s.flags = U.fallback ? 1u : 0u;
    s.k = U.k;
    s.count_above = (U.state == ST_DONE) ? U.count_above : 0;
    s.ties_at_thresh = (U.state == ST_DONE) ? U.ties : 0;
    s.ties_taken = (U.state == ST_DONE) ? U.need : 0;
    P.st_units[(long long)i * P.st_units_stride + P.st_unit_base + u] = s;
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(TPB) k_cut(Plan P) {
    __shared__ long long s_scan[33];
    __shared__ uint32_t s_scan32[33];
    __shared__ long long s_tile;
    __shared__ long long s_rem;
    __shared__ long long s_pos;
    const int idx = blockIdx.x;
    Unit& U = P.units[idx];
    if (U.state == ST_OFF || U.state == ST_NONE) {
        if (threadIdx.x == 0) write_unit_stats(P, idx, U);
        return;
    }
    if (U.state != ST_TKNOWN) return;   // not reached for a well-formed plan
    const int i = U.expert;
    if (threadIdx.x == 0) { s_tile = -1; s_rem = 0; s_pos = -1; }   // ordered by the scan's barriers
    if (U.need < U.ties) {
        // 1. the tile that holds the need-th tie (tiles in unit order)
        const long long nt = U.tile_end - U.tile_begin;
        const long long per = (nt + blockDim.x - 1) / blockDim.x;
        const long long j0 = U.tile_begin + threadIdx.x * per;
        const long long j1 = (j0 + per < U.tile_end) ? j0 + per : U.tile_end;
        auto tile_ties = [&](long long g) -> long long {
            const long long q = (long long)i * P.n_tiles + g;
            if (U.tie_src == TIE_EQ_HI) return P.trec[q].eq_hi;
            if (U.tie_src == TIE_EQ_LO) return P.trec[q].eq_lo;
            return P.tcnt[q];
        };
        long long local = 0;
        for (long long g = j0; g < j1; ++g) local += tile_ties(g);
        long long total;
        const long long excl = block_excl_scan(local, s_scan, &total);
        if (excl < U.need && U.need <= excl + local) {
            long long acc = excl;
            for (long long g = j0; g < j1; ++g) {
                const long long c = tile_ties(g);
                if (U.need <= acc + c) { s_tile = g; s_rem = U.need - acc; break; }
                acc += c;
            }
        }
        __syncthreads();
        if (s_tile < U.tile_begin || s_tile >= U.tile_end) {
            // the tie counts do not reach `need`: inconsistent state, keep every tie
            if (threadIdx.x == 0) { set_status(P.hdr, ISO_ERR_CUDA); U.cut = CUT_ALL; }
            goto finish;
        }
        {
        // 2. inside that tile, the rem-th entry with key == t in index order
        const long long g = s_tile;
        const long long rem = s_rem;
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        const void* x = P.xptr[i * P.n_tensors + t];
        const long long e0 = (g - d.tile_base) * TILE;
        constexpr int PER = TILE / TPB;   // 32 consecutive entries per thread
        const long long eb = e0 + (long long)threadIdx.x * PER;
        uint32_t mine = 0;
        for (int j = 0; j < PER; j += VEC) {
            const long long e = eb + j;
            if (e >= d.numel) break;
            float tau[VEC];
            TauSrc<XT, BT, CKPT>::load8(x, d.base, e, d.numel, tau);
#pragma unroll
            for (int q = 0; q < VEC; ++q)
                if (e + q < d.numel && key_of(tau[q]) == U.t) mine++;
        }
        uint32_t tot32;
        const uint32_t before = block_excl_scan(mine, s_scan32, &tot32);
        if (before < rem && rem <= before + mine) {
            uint32_t acc = before;
            for (int j = 0; j < PER; ++j) {
                const long long e = eb + j;
                if (e >= d.numel) break;
                if (key_of(TauSrc<XT, BT, CKPT>::load1(x, d.base, e)) == U.t) {
                    if (++acc == rem) {
                        s_pos = ((P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0) + e;
                        break;
                    }
                }
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            if (s_pos < 0) { set_status(P.hdr, ISO_ERR_CUDA); U.cut = CUT_ALL; }
            else U.cut = s_pos + 1;
        }
        }
    } else if (threadIdx.x == 0) {
        U.cut = CUT_ALL;
    }
finish:
    if (threadIdx.x == 0) {
        if (U.want_gamma) {
            const double ft = (double)__uint_as_float(U.t);
            const double fh = (double)__uint_as_float(U.hi);
            double g;
            if (U.r_src == SRC_DATA) {
                g = U.gamma_acc2 + (double)U.need * ft * ft;
            } else if (U.tie_src == TIE_EQ_HI) {
                g = U.gamma_acc + (double)U.need * ft * ft;
            } else {
                g = U.gamma_acc + (double)U.c_hi * fh * fh + U.gamma_acc2 + (double)U.need * ft * ft;
            }
            U.gamma = g;
        }
        U.state = ST_DONE;
        write_unit_stats(P, idx, U);
    }
}

// ---------------------------------------------------------------------------
// instantiations
// ---------------------------------------------------------------------------
#define ISO_SELECT_INST(XT, BT, CK)                                            \
    template __global__ void k_sample<XT, BT, CK>(Plan);                      \
    template __global__ void k_count<XT, BT, CK>(Plan);                       \
    template __global__ void k_radix_hist<XT, BT, CK>(Plan);                  \
    template __global__ void k_tie<XT, BT, CK>(Plan);                         \
    template __global__ void k_cut<XT, BT, CK>(Plan);

ISO_SELECT_INST(__nv_bfloat16, __nv_bfloat16, false)
ISO_SELECT_INST(__nv_bfloat16, float, false)
ISO_SELECT_INST(float, __nv_bfloat16, false)
ISO_SELECT_INST(float, float, false)
ISO_SELECT_INST(__nv_bfloat16, __nv_bfloat16, true)
ISO_SELECT_INST(__nv_bfloat16, float, true)
ISO_SELECT_INST(float, __nv_bfloat16, true)
ISO_SELECT_INST(float, float, true)

}  // namespace iso
