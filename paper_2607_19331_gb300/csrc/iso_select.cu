// iso_select.cu -- exact TopKMask threshold per selection unit (TENSOR and
// GLOBAL scope).
//
// TopKMask(|tau|, rho) keeps the k = floor(rho n + 1/2) entries of largest
// |tau| (App. F, TIES trim); ties go to the lowest position.  The result of
// this file is, per unit, a threshold key t and a position cut such that
//     kept(p)  <=>  key(p) > t  ||  (key(p) == t && pos(p) < cut)
// which the streaming passes then apply as a pure per-entry predicate.
//
// Pipeline (all launches on the caller's stream; no block waits on another):
//   k_sample   keys at evenly spaced chunks -> band [lo, hi] around rank k
//   k_count    one full read: #key > hi, #key == hi / == lo per tile, and the
//              interior keys lo < key < hi appended to the unit's segment
//   k_decide   locate rank k among the counters; a miss (or an overflowing
//              segment) switches the unit to a radix select over its data
//   k_radix_*  up to three 11-bit radix levels over the interior keys (or
//              over the whole unit on the fallback path)
//   k_tie      per-tile counts of keys == t when the threshold is interior
//   k_cut      the tile holding the need-th tie, then the exact position
//
// Work layout: a tile is 1024 entries handled by one warp; every warp (or
// block) walks a contiguous range of (expert, tile) items, so the owning
// tensor and unit change rarely and are tracked incrementally.
#include "iso_kernels.cuh"

namespace iso {

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
        U.v_cap = d.v_cap;
        U.v_off = d.v_off + (unsigned long long)i * d.v_cap;
        U.brec_cap = d.brec_cap;
        U.brec_off = d.brec_off;
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
    U.state = (U.k == 0) ? ST_NONE : ST_SAMPLE;
}

// ---------------------------------------------------------------------------
// block-level radix select in shared memory
// ---------------------------------------------------------------------------

// Among nb bins taken from the top, the bin b with above(b) < rank <=
// above(b) + hist[b]; rank <= 0 or beyond the total gives bin 0.
__device__ void block_find_from_top(const uint32_t* hist, int nb, long long rank,
                                    long long* sm_scan, int* res_bin, long long* res_above) {
    const int per = (nb + blockDim.x - 1) / blockDim.x;
    const int j0 = threadIdx.x * per;
    if (threadIdx.x == 0) { *res_bin = 0; *res_above = 0; }   // ordered by the scan's barriers
    long long local = 0;
    for (int j = j0; j < j0 + per && j < nb; ++j) local += hist[nb - 1 - j];
    long long total;
    const long long excl = block_excl_scan(local, sm_scan, &total);
    if (excl < rank && rank <= excl + local) {
        long long acc = excl;
        for (int j = j0; j < j0 + per && j < nb; ++j) {
            const uint32_t h = hist[nb - 1 - j];
            if (rank <= acc + h) { *res_bin = nb - 1 - j; *res_above = acc; break; }
            acc += h;
        }
    }
    __syncthreads();
}

// The rank[r]-th largest (1-based, 1 <= rank[r] <= n) of n keys in shared
// memory for R <= SEL_R ranks at once.  The key is found one 8-bit digit at
// a time from the top; ranks whose prefixes agree share a histogram, so one
// pass over the keys per digit serves every rank (at most one histogram bin
// per key), and each histogram is scanned by one warp.  `hist` holds
// SEL_R * 256 zeroed counters on entry and is zero again on return.
constexpr int SEL_R = SAMPLE_SEL_R;
__device__ void block_select_ranks(const uint32_t* keys, int n, int R, const long long* rank,
                                   uint32_t* hist, uint32_t* out) {
    __shared__ uint32_t s_pref[SEL_R];
    __shared__ long long s_rem[SEL_R];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x < R) { s_pref[threadIdx.x] = 0; s_rem[threadIdx.x] = rank[threadIdx.x]; }
    __syncthreads();
#pragma unroll 1
    for (int lvl = 0; lvl < 4; ++lvl) {
        const int dsh = 24 - 8 * lvl;                    // the digit's shift
        // distinct prefixes in rank order (every thread alike)
        uint32_t gp[SEL_R];
        int grp[SEL_R];
        int ng = 0;
#pragma unroll
        for (int r = 0; r < SEL_R; ++r) {
            gp[r] = 0;
            grp[r] = -1;
        }
#pragma unroll
        for (int r = 0; r < SEL_R; ++r) {
            if (r < R) {
                const uint32_t pr = s_pref[r];
                int g = ng;
#pragma unroll
                for (int j = SEL_R - 1; j >= 0; --j)
                    if (j < ng && gp[j] == pr) g = j;
#pragma unroll
                for (int j = 0; j < SEL_R; ++j)
                    if (j == ng && g == ng) gp[j] = pr;
                if (g == ng) ++ng;
                grp[r] = g;
            }
        }
        // one histogram per distinct prefix; a thread's run of keys in one
        // bin adds once (the keys near the threshold crowd into a few bins)
        uint32_t run_slot = 0, run_cnt = 0;
        for (int q = threadIdx.x; q < n; q += blockDim.x) {
            const uint32_t v = keys[q];
            const uint32_t top = lvl == 0 ? 0u : v >> (dsh + 8);
            int g = -1;
#pragma unroll
            for (int j = SEL_R - 1; j >= 0; --j)
                if (j < ng && gp[j] == top) g = j;
            if (g < 0) continue;
            const uint32_t slot = (uint32_t)g * 256u + ((v >> dsh) & 255u);
            if (slot != run_slot) {
                if (run_cnt) atomicAdd(&hist[run_slot], run_cnt);
                run_slot = slot;
                run_cnt = 0;
            }
            ++run_cnt;
        }
        if (run_cnt) atomicAdd(&hist[run_slot], run_cnt);
        __syncthreads();
        // warp g scans histogram g from the top bin: lane L holds bins 255-8L .. 248-8L
        if (warp < ng) {
            uint32_t h[8];
            uint32_t* hg = hist + warp * 256;
            uint32_t sum = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) { h[j] = hg[255 - 8 * lane - j]; sum += h[j]; }
            uint32_t incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += y;
            }
            const long long excl = (long long)(incl - sum);
#pragma unroll
            for (int r = 0; r < SEL_R; ++r) {
                if (r >= R || grp[r] != warp) continue;
                const long long rr = s_rem[r];
                if (excl < rr && rr <= excl + (long long)sum) {
                    long long acc = excl;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        if (rr <= acc + (long long)h[j]) {
                            s_pref[r] = (s_pref[r] << 8) | (uint32_t)(255 - 8 * lane - j);
                            s_rem[r] = rr - acc;
                            break;
                        }
                        acc += h[j];
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) hg[255 - 8 * lane - j] = 0;
        }
        __syncthreads();
    }
    if (threadIdx.x < R) out[threadIdx.x] = s_pref[threadIdx.x];
    __syncthreads();
}

// ---------------------------------------------------------------------------
// sample -> band
// ---------------------------------------------------------------------------

// unit position -> tensor for GLOBAL scope: last tensor with uoff <= pos
__device__ __forceinline__ int tensor_of_upos(const TensorDesc* tens, int n_tensors, long long pos) {
    int lo = 0, hi = n_tensors - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (tens[mid].uoff <= pos) lo = mid; else hi = mid - 1;
    }
    return lo;
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(SAMPLE_TPB, 2) k_sample(Plan P) {
    extern __shared__ __align__(16) uint32_t s_keys[];
    uint32_t* s_hist = s_keys + SAMPLE_MAX;          // SEL_R * 256 counters
    __shared__ long long s_scan[33];

    Unit& U = P.units[blockIdx.x];
    if (U.state != ST_SAMPLE) return;
    const int i = U.expert;
    const long long n = U.n;
    const int S = (int)(n < SAMPLE_MAX ? n : SAMPLE_MAX);
    constexpr int nch = SAMPLE_MAX / SAMPLE_CHUNK;
    if (S < n && P.scope != ISO_SCOPE_GLOBAL) {
        // chunks of 256 contiguous entries at evenly spaced, 8-aligned starts:
        // one chunk per warp step, 8 entries per lane
        const int t = U.tensor;
        const void* x = P.xptr[i * P.n_tensors + t];
        const void* b = P.tens[t].base;
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
        // three chunks per warp at a time: their loads are in flight together
        constexpr int CB = 3;
        for (int c0 = warp; c0 < nch; c0 += CB * nw) {
            float tau[CB][VEC];
#pragma unroll
            for (int m = 0; m < CB; ++m) {
                const int c = c0 + m * nw;
                // (n - 256) c / 95, rounded down (exact: integer arithmetic)
                const long long start = (long long)(((unsigned long long)(n - SAMPLE_CHUNK) *
                                                     (unsigned long long)(c < nch ? c : 0)) /
                                                    (unsigned long long)(nch - 1)) & ~7LL;
                TauSrc<XT, BT, CKPT>::load8(x, b, start + lane * VEC, n, tau[m]);
            }
#pragma unroll
            for (int m = 0; m < CB; ++m) {
                const int c = c0 + m * nw;
                if (c < nch) {
#pragma unroll
                    for (int j = 0; j < VEC; ++j) s_keys[c * SAMPLE_CHUNK + lane * VEC + j] = key_of(tau[m][j]);
                }
            }
        }
    } else {
        for (int q = threadIdx.x; q < S; q += blockDim.x) {
            long long pos;
            if (S == n) {
                pos = q;
            } else {
                const int c = q / SAMPLE_CHUNK, j = q % SAMPLE_CHUNK;
                pos = (long long)(((unsigned long long)(n - SAMPLE_CHUNK) * (unsigned long long)c) /
                                  (unsigned long long)(nch - 1)) + j;
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
    }
    for (int q = threadIdx.x; q < SEL_R * 256; q += blockDim.x) s_hist[q] = 0;
    __syncthreads();
    uint32_t lo, hi;
    uint32_t that = 0;                       // fused pass: the estimate of the threshold
    const bool fused_t = P.fused && P.scope == ISO_SCOPE_TENSOR;
    __shared__ long long s_rk[SEL_R];
    __shared__ uint32_t s_kv[SEL_R];
    __shared__ int s_edge[2];
    if (S == n) {
        // the sample is the whole unit: the band is the exact threshold
        if (threadIdx.x == 0) s_rk[0] = U.k;
        __syncthreads();
        block_select_ranks(s_keys, S, 1, s_rk, s_hist, s_kv);
        hi = lo = that = s_kv[0];
    } else {
        // the band's sample ranks, by one thread (binary64 is slow on this
        // GPU), then every rank in one selection: the band edges and, for
        // the fused pass, the rank of k and halfway to either edge
        if (threadIdx.x == 0) {
            const double q = (double)U.k / (double)n;
            const double r = (double)U.k * (double)S / (double)n;
            const double delta = SAMPLE_Z * sqrt((double)S * q * (1.0 - q)) + 2.0;
            const long long ra = (long long)floor(r - delta), rb = (long long)ceil(r + delta);
            const long long rk = (long long)floor(r + 0.5), h = (long long)floor(delta / 2.0);
            auto clampr = [&](long long x) { return x < 1 ? 1LL : (x > S ? (long long)S : x); };
            s_rk[0] = clampr(ra);
            s_rk[1] = clampr(rb);
            s_rk[2] = clampr(rk - h);
            s_rk[3] = clampr(rk);
            s_rk[4] = clampr(rk + h);
            s_edge[0] = ra >= 1;
            s_edge[1] = rb <= S;
        }
        __syncthreads();
        block_select_ranks(s_keys, S, fused_t ? 5 : 2, s_rk, s_hist, s_kv);
        hi = s_edge[0] ? s_kv[0] : KEY_MAX;
        lo = s_edge[1] ? s_kv[1] : 0u;
        if (fused_t) {
            // t^: of the sampled keys at five ranks across the band (the band
            // edges, the rank of k and halfway between), the one that occurs
            // most often in the sample -- a run of ties wider than a fifth
            // of the band is always among them.  The corrections are then
            // small whichever side of that run rank k falls on.
            uint32_t pv[5];
            pv[0] = s_kv[0];
            pv[1] = s_kv[2];
            pv[2] = s_kv[3];
            pv[3] = s_kv[4];
            pv[4] = s_kv[1];
            unsigned cnt[5] = {0, 0, 0, 0, 0};
            for (int q = threadIdx.x; q < S; q += blockDim.x) {
                const uint32_t v = s_keys[q];
#pragma unroll
                for (int j = 0; j < 5; ++j) cnt[j] += (v == pv[j]);
            }
            __shared__ unsigned s_cnt[5];
            if (threadIdx.x < 5) s_cnt[threadIdx.x] = 0;
            __syncthreads();
#pragma unroll
            for (int j = 0; j < 5; ++j) {
                const unsigned w = __reduce_add_sync(0xFFFFFFFFu, cnt[j]);
                if ((threadIdx.x & 31) == 0 && w) atomicAdd(&s_cnt[j], w);
            }
            __syncthreads();
            int best = 2;
            for (int j = 0; j < 5; ++j)
                if (s_cnt[j] > s_cnt[best] || (s_cnt[j] == s_cnt[best] && j == 2)) best = j;
            that = pv[best];
            if (that > hi) that = hi;
            if (that < lo) that = lo;
            // run mode: the run of t^ covers the sample rank of k by half the
            // band on both sides (2.5 sample standard deviations), so the
            // threshold is t^ but for a small chance, which the counts catch
            // (then the unit is resolved exactly and re-applied): the band
            // collapses to t^ and the fused pass needs no band test
            if (pv[1] == that && pv[3] == that) { lo = that; hi = that; }
        }
    }
    // Fused K = 1 pass: the estimate t^ of the threshold (the sample's key at
    // the rank of k; bf16-derived task vectors hold long runs of ties there)
    // and of the position before which its ties are kept: exact here when
    // the sample is the whole unit, else interpolated from a larger count
    // sample by k_csample.
    long long chat = -1;
    if (fused_t) {
        __shared__ long long s_chat;
        if (threadIdx.x == 0) s_chat = n;
        __syncthreads();
        if (S == n) {
            // keys in position order: the need-th tie
            const uint32_t tk = that;
            const int per = (S + blockDim.x - 1) / blockDim.x;
            const int q0 = threadIdx.x * per;
            long long gt = 0, eq = 0;
            for (int q = q0; q < q0 + per && q < S; ++q) { gt += s_keys[q] > tk; eq += s_keys[q] == tk; }
            long long tot;
            const long long before = block_excl_scan(eq, s_scan, &tot);
            const long long cgt = block_sum(gt, s_scan);
            const long long need = U.k - cgt;
            if (before < need && need <= before + eq) {
                long long acc = before;
                for (int q = q0; q < q0 + per && q < S; ++q)
                    if (s_keys[q] == tk && ++acc == need) { s_chat = q + 1; break; }
            }
            __syncthreads();
        }
        chat = s_chat;
    }
    if (threadIdx.x == 0) {
        U.lo = lo;
        U.hi = hi;
        if (chat >= 0) { U.mode_t = 1; U.that = that; U.chat = chat; }
        U.state = ST_BAND;
    }
}

// Fused pass, units larger than the sample: the cut among the ties of t^
// estimated from a count sample of up to COUNT_CHUNKS chunks of 256 entries
// -- contiguous when they cover the unit (then the estimate is exact), else
// evenly spaced -- counting per chunk the keys equal to t^ and overall the
// keys above it.  CS_SPLIT blocks share a unit; the last of them to finish
// finds the chunk where the sampled ties reach the sampled need and
// interpolates inside it.
template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(CS_TPB, 4) k_csample(Plan P) {
    const int u = blockIdx.x / CS_SPLIT, part = blockIdx.x % CS_SPLIT;
    Unit& U = P.units[u];
    // uniform over the unit's blocks: all of them return here, or none
    if (U.state != ST_BAND || !U.mode_t || U.n <= SAMPLE_MAX) return;
    const long long n = U.n;
    const uint32_t tk = U.that;
    const long long nchunks = (n + SAMPLE_CHUNK - 1) / SAMPLE_CHUNK;
    const bool whole = nchunks <= COUNT_CHUNKS;
    const int CX = whole ? (int)nchunks : COUNT_CHUNKS;
    // (the divisor is a constant: no 64-bit division routine per chunk)
    auto chunk_start = [&](int c) -> long long {
        if (whole) return (long long)c * SAMPLE_CHUNK;
        return (long long)(((unsigned long long)(n - SAMPLE_CHUNK) * (unsigned long long)c) /
                           (unsigned long long)(COUNT_CHUNKS - 1)) & ~7LL;
    };
    uint32_t* ties = P.csamp + (size_t)u * COUNT_CHUNKS;
    const int t = U.tensor;
    const void* x = P.xptr[U.expert * P.n_tensors + t];
    const void* b = P.tens[t].base;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    constexpr int PER_PART = COUNT_CHUNKS / CS_SPLIT;
    const int c_lo = part * PER_PART, c_hi = min(CX, c_lo + PER_PART);
    // several chunks per warp at a time: their loads are in flight together
    constexpr int CB = sizeof(XT) == 2 ? 4 : 2;
    unsigned long long gt_w = 0;
    for (int c0 = c_lo + warp; c0 < c_hi; c0 += CB * nw) {
        float tau[CB][VEC];
        long long ec[CB];
#pragma unroll
        for (int m = 0; m < CB; ++m) {
            const int c = c0 + m * nw;
            ec[m] = (c < c_hi) ? chunk_start(c) + lane * VEC : n;
            TauSrc<XT, BT, CKPT>::load8(x, b, ec[m] < n ? ec[m] : 0, n, tau[m]);
        }
#pragma unroll
        for (int m = 0; m < CB; ++m) {
            const int c = c0 + m * nw;
            unsigned gt = 0, eq = 0;
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const uint32_t v = key_of(tau[m][j]);
                const bool in = ec[m] + j < n;
                gt += in && v > tk;
                eq += in && v == tk;
            }
            gt = __reduce_add_sync(0xFFFFFFFFu, gt);
            eq = __reduce_add_sync(0xFFFFFFFFu, eq);
            if (c < c_hi) {
                if (lane == 0) ties[c] = eq;
                gt_w += gt;
            }
        }
    }
    __shared__ unsigned long long s_gt;
    __shared__ int s_last;
    if (threadIdx.x == 0) s_gt = 0;
    __syncthreads();
    if (lane == 0 && gt_w) atomicAdd(&s_gt, gt_w);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (s_gt) atomicAdd(&U.cs_gt, s_gt);
        __threadfence();
        s_last = atomicAdd(&U.cs_done, 1u) == (unsigned)(CS_SPLIT - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // the unit's last block: the sampled need, then the chunk where the
    // sampled ties reach it (integer comparisons against ceil(need))
    __shared__ double s_need;
    __shared__ long long s_nc, s_chat;
    __shared__ long long s_scan[33];
    if (threadIdx.x == 0) {
        const long long SX = whole ? n : (long long)CX * SAMPLE_CHUNK;
        const unsigned long long cgt = atomicAdd(&U.cs_gt, 0ULL);
        const double need = (double)U.k * (double)SX / (double)n - (double)cgt;
        s_need = need;
        s_nc = need <= 0.0 ? 0 : (long long)ceil(need);
        s_chat = need <= 0.0 ? 0 : n;
    }
    __syncthreads();
    const long long nc = s_nc;
    constexpr int CPT = (COUNT_CHUNKS + CS_TPB - 1) / CS_TPB;   // chunks per thread
    const int cb = threadIdx.x * CPT;
    long long tcl[CPT];
    long long local = 0;
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        tcl[j] = (cb + j < CX) ? (long long)__ldcg(ties + cb + j) : 0;
        local += tcl[j];
    }
    long long tot;
    long long cum = block_excl_scan(local, s_scan, &tot);
    if (nc > 0) {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const int c = cb + j;
            if (tcl[j] > 0 && cum < nc && nc <= cum + tcl[j]) {
                const long long a0 = chunk_start(c);
                const long long bb = (c + 1 == CX) ? n : chunk_start(c + 1);
                const long long ch = a0 + (long long)((s_need - (double)cum) / (double)tcl[j] * (double)(bb - a0));
                s_chat = ch < 0 ? 0 : (ch > n ? n : ch);
            }
            cum += tcl[j];
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) U.chat = s_chat;
}

// ---------------------------------------------------------------------------
// count pass: one warp per tile, one contiguous item range per warp
// ---------------------------------------------------------------------------
// Per entry the pass does only what every entry needs: tau, its key, the
// count above the band and a band test.  Band keys (lo <= key <= hi, a few
// per cent of the entries) are staged in shared memory -- lane L's j-th at
// slot j*32 + L, conflict-free; every key is written and only a band key
// advances the lane's slot -- and then copied, per lane, to the unit's
// candidate segment.  The radix select and the tie counts work on that set.
//
// The warp's tiles stream through two register buffers: the next tile's loads
// are issued before the current tile is processed.  A non-finite tau has a key
// above every finite key, so it is either above hi, where it turns the lane's
// binary32 sum of tau^2 non-finite (then the tile is re-checked key by key),
// or a band key, checked when the band keys are copied; lo itself is a sampled
// key, so a non-finite lo is a band key of its own unit.

// consecutive items of one (expert, tensor) that the count pass visits (with
// round-robin items, one item)
struct CountRun {
    uint32_t it0, end;       // items [it0, end), end clipped to the warp's range
    uint32_t e0;             // tensor entry of item it0's first element
    uint32_t n;              // tensor entries
    uint32_t rec;            // index of item it0 in the per-(expert, tile) arrays
    uint32_t left0;          // this warp's items of the unit from it0 on
    const void* xp;
    const void* bp;
    Unit* U;
};

// the first counted item at or after item it (< end) in steps of `step`: the
// run of its (expert, tensor) with step 1, the item alone otherwise; false if
// there is none
__device__ __forceinline__ bool count_run_at(const Plan& P, uint32_t it, uint32_t end, uint32_t step, CountRun& r) {
    while (it < end) {
        Cursor c;
        cursor_at(P, it, c);
        const uint32_t re = min((uint32_t)c.run_end, end);
        Unit* U = count_unit(P, c);
        if (U) {
            const TensorDesc& d = P.tens[c.t];
            r.it0 = it;
            r.end = step == 1 ? re : it + 1;
            r.left0 = (re - it + step - 1) / step;
            r.e0 = (uint32_t)(c.g - d.tile_base) * TILE;
            r.n = (uint32_t)d.numel;
            r.rec = (uint32_t)((long long)c.i * P.n_tiles + c.g);
            r.xp = P.xptr[c.i * P.n_tensors + c.t];
            r.bp = d.base;
            r.U = U;
            return true;
        }
        it += (re - it + step - 1) / step * step;   // the warp's first item past the run
    }
    return false;
}

// EMIT: also write the compact candidates (Plan::ccv); a separate
// instantiation, so the plain counting pass keeps its registers.  The tile's
// binary32 task vector is kept in COUNT_EMIT_SMEM bytes of dynamic shared
// memory (32 rows of 33 words per warp, row w holding positions 32 w ..
// 32 w + 31), and after the count each lane turns one row into its mask word
// and writes the row's candidates in position order.
template <typename XT, typename BT, bool CK, bool EMIT>
__global__ void __launch_bounds__(TPB, COUNT_BLOCKS_PER_SM) k_count(Plan P) {
    __shared__ uint32_t s_band[WPB][TILE + 32];
    extern __shared__ float s_vst[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float* const vrow = s_vst + warp * (32 * 33);
    uint32_t* const sbl = s_band[warp] + lane;
    // item indices fit 32 bits (the host checks K * n_tiles < 2^31)
    const uint32_t W = gridDim.x * WPB;
    const uint32_t wid = blockIdx.x * WPB + warp;
    const uint32_t items = (uint32_t)(P.K * P.n_tiles);
    uint32_t beg, end, step;
    if (PASS_INTERLEAVE) {
        beg = wid;
        end = items;
        step = W;
    } else {
        const uint32_t per = (items + W - 1) / W;
        beg = wid * per;
        end = min(items, beg + per);
        step = 1;
    }
    if (beg >= end) return;
    const unsigned FULL = 0xFFFFFFFFu;

    CountRun r;
    if (!count_run_at(P, beg, end, step, r)) return;

    // per-unit accumulators (warp-uniform) and the candidate chunk
    Unit* au = nullptr;
    uint32_t a_gt = 0, a_int = 0, a_hi = 0, a_lo = 0;
    // per-lane sums of tau^2 (above hi; band keys above lo) as binary32
    // pairs: sum + error term, kept exact by two-sum, so no binary64
    // arithmetic runs per tile
    float s_gg = 0.0f, e_gg = 0.0f, s_gb = 0.0f, e_gb = 0.0f;
    uint32_t* cseg = nullptr;                     // the unit's candidate segment
    uint32_t ch_pos = 0, ch_left = 0, cap = 0;
    bool ovf = false;
    uint32_t lo = 0, hi = 0, span = 0;
    bool want_gamma = false;
    // compact candidates (P.ccv): the warp's chunk of the unit's value
    // segment; a tile needs at most TILE slots, taken before the tile
    float* vseg = nullptr;
    unsigned long long v_pos = 0;
    uint32_t v_left = 0;
    bool v_ovf = false;

    auto flush = [&]() {
        if (!au) return;
        const double gg = warp_sum((double)s_gg + (double)e_gg), gb = warp_sum((double)s_gb + (double)e_gb);
        if (lane == 0) {
            if (a_gt) atomicAdd(&au->c_gt, (unsigned long long)a_gt);
            if (a_int) atomicAdd(&au->n_int, (unsigned long long)a_int);
            if (a_hi) atomicAdd(&au->c_hi, (unsigned long long)a_hi);
            if (a_lo) atomicAdd(&au->c_lo, (unsigned long long)a_lo);
            if (want_gamma) {
                if (gg != 0.0) atomicAdd(&au->gamma_acc, gg);
                if (gb != 0.0) atomicAdd(&au->gamma_band, gb);
            }
            if (ovf) au->overflow = 1;
        }
        a_gt = a_int = a_hi = a_lo = 0;
        s_gg = e_gg = s_gb = e_gb = 0.0f;
    };

    // Count one tile held in registers (item it of run rr).  As each vector
    // step is converted to tau, its registers are refilled with the same step
    // of the next tile (item it2 of run r2), so a whole tile of loads is in
    // flight while this one is counted.
    RawTile<XT, BT, CK> rt;
    // the unused slots of the warp's chunk get KEY_NONE, so that a large
    // unit's pool can be read as one flat array (k_radix_hist)
    auto seal = [&]() {
        if (au && !ovf)
            for (uint32_t q = lane; q < ch_left; q += 32) cseg[ch_pos + q] = KEY_NONE;
        ch_left = 0;
    };

    auto count_tile = [&](const CountRun& rr, uint32_t it, bool more, const CountRun& r2, uint32_t it2) {
        if (rr.U != au) {
            seal();
            flush();
            au = rr.U;
            lo = au->lo;
            hi = au->hi;
            span = hi - lo;
            want_gamma = au->want_gamma != 0;
            cap = (uint32_t)au->cand_cap;
            cseg = P.cand + au->cand_off;
            ch_left = 0;
            ovf = false;
            vseg = P.vals + au->v_off;
            v_left = 0;
            v_ovf = false;
        }
        const uint32_t e0 = rr.e0 + (it - rr.it0) * TILE;
        const uint32_t rem = rr.n - e0;           // > 0
        const uint32_t rec = rr.rec + (it - rr.it0);
        const uint32_t ne0 = more ? r2.e0 + (it2 - r2.it0) * TILE : 0u;
        const uint32_t nrem = more ? r2.n - ne0 : 0u;
        if constexpr (EMIT) {
            if (v_left < TILE && !v_ovf) {
                unsigned long long start = 0;
                uint32_t req = 0;
                if (lane == 0) {
                    const uint32_t left = rr.left0 - (it - rr.it0);   // this warp's items of the unit still to count
                    req = (uint32_t)min((unsigned long long)VCHUNK, (unsigned long long)TILE * max(left, 1u));
                    start = atomicAdd(&au->v_alloc, (unsigned long long)req);
                }
                start = __shfl_sync(FULL, start, 0);
                req = __shfl_sync(FULL, req, 0);
                if (start + req > au->v_cap) v_ovf = true;
                else { v_pos = start; v_left = req; }
            }
        }
        // the step's binary32 values into the warp's rows (position
        // 256 v + 8 lane + j: row 8 v + lane / 4, column 8 (lane % 4) + j;
        // the 33-word rows keep both this and the row-per-lane reads free of
        // bank conflicts)
        auto stash = [&](int v, const float (&tau)[VEC]) {
            float* d = vrow + (8 * v + (lane >> 2)) * 33 + 8 * (lane & 3);
#pragma unroll
            for (int j = 0; j < VEC; ++j) d[j] = tau[j];
        };

        // pass 1: every entry
        uint32_t n_gt = 0;
        float f_gg = 0.0f;                         // tau^2 above hi (also the non-finite detector)
        uint32_t* sp = sbl;
        if (rem >= TILE) {
#pragma unroll
            for (int v = 0; v < WVEC; ++v) {
                float tau[VEC];
                rt.tau(v, tau);
                if (more) rt.load_step(v, r2.xp, r2.bp, ne0, nrem, lane);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    const uint32_t kk = key_of(tau[j]);
                    const bool gt = kk > hi;
                    n_gt += gt;
                    f_gg = gt ? __fmaf_rn(tau[j], tau[j], f_gg) : f_gg;
                    *sp = kk;
                    sp += (kk - lo <= span) ? 32 : 0;
                }
                if constexpr (EMIT) stash(v, tau);
            }
        } else {
#pragma unroll
            for (int v = 0; v < WVEC; ++v) {
                float tau[VEC];
                rt.tau(v, tau);
                if (more) rt.load_step(v, r2.xp, r2.bp, ne0, nrem, lane);
                const uint32_t o = (uint32_t)(v * (32 * VEC) + lane * VEC);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    if (o + j >= rem) continue;
                    const uint32_t kk = key_of(tau[j]);
                    const bool gt = kk > hi;
                    n_gt += gt;
                    f_gg = gt ? __fmaf_rn(tau[j], tau[j], f_gg) : f_gg;
                    *sp = kk;
                    sp += ((kk >= lo) & !gt) ? 32 : 0;
                }
                if constexpr (EMIT) stash(v, tau);
            }
        }
        const uint32_t nb = (uint32_t)(sp - sbl) >> 5;
        if (__any_sync(FULL, !(fabsf(f_gg) <= 3.402823466e38f))) {
            // a non-finite (or overflowing) sum: read the tile's keys again
            uint32_t kmax = 0;
            for (int v = 0; v < WVEC; ++v) {
                const uint32_t o = (uint32_t)(v * (32 * VEC) + lane * VEC);
                if (o >= rem) break;
                float tau[VEC];
                TauSrc<XT, BT, CK>::load8(rr.xp, rr.bp, (long long)e0 + o, (long long)rr.n, tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j)
                    if (o + j < rem) kmax = max(kmax, key_of(tau[j]));
            }
            if (__any_sync(FULL, kmax >= KEY_INF) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
        }
        if (want_gamma) two_sum_add(s_gg, e_gg, f_gg);
        __syncwarp();

        // pass 2: copy the staged band keys to the unit's candidate segment
        uint32_t t_int;
        const uint32_t off = warp_excl_scan(nb, &t_int);
        if (t_int && !ovf && t_int > ch_left) {
            // the rest of the current chunk is too short: seal it, take a new one
            for (uint32_t q = lane; q < ch_left; q += 32) cseg[ch_pos + q] = KEY_NONE;
            unsigned long long start = 0;
            uint32_t req = 0;
            if (lane == 0) {
                const uint32_t left = rr.left0 - (it - rr.it0);   // this warp's items of the unit still to count
                const unsigned long long want = (unsigned long long)t_int * (unsigned long long)left;
                req = (uint32_t)max((unsigned long long)t_int, min((unsigned long long)CHUNK_MAX, want));
                start = atomicAdd(&au->n_alloc, (unsigned long long)req);
            }
            start = __shfl_sync(FULL, start, 0);
            req = __shfl_sync(FULL, req, 0);
            if (start + req > cap) { ovf = true; ch_left = 0; }
            else { ch_pos = (uint32_t)start; ch_left = req; }
        }
        const bool store = t_int && !ovf;
        uint32_t n_hi = 0, n_lo = 0, kbad = 0;
        float f_band = 0.0f;                      // tau^2 over the band keys above lo
        {
            uint32_t* dst = cseg + ch_pos + off;
            for (uint32_t q = 0; q < nb; ++q) {
                const uint32_t kk = sbl[q * 32];
                if (store) dst[q] = kk;
                n_hi += (kk == hi);
                n_lo += (kk == lo) && (kk != hi);
                kbad |= (kk >= KEY_INF);
                if (want_gamma && kk != lo) { const float f = __uint_as_float(kk); f_band = __fmaf_rn(f, f, f_band); }
            }
        }
        if (__any_sync(FULL, kbad) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
        if (want_gamma) two_sum_add(s_gb, e_gb, f_band);
        const uint32_t t_gt = __reduce_add_sync(FULL, n_gt);
        const uint32_t t_hi = __reduce_add_sync(FULL, n_hi);
        const uint32_t t_lo = __reduce_add_sync(FULL, n_lo);
        if (lane == 0) {
            P.tcand[rec] = make_uint2(store ? ch_pos : 0u, store ? t_int : 0u);
            P.teq_lo[rec] = t_lo;
            P.teq_hi[rec] = t_hi;
            if (EMIT) P.tval[rec] = v_ovf ? KEY_NONE : (uint32_t)v_pos;
        }
        if constexpr (EMIT) {
            // lane l: row l (positions 32 l .. 32 l + 31) into mask word l and
            // its values with key >= lo, in position order
            __syncwarp();
            const float* row = vrow + lane * 33;
            uint32_t m = 0;
#pragma unroll
            for (int q = 0; q < 32; ++q)
                m |= (uint32_t)(key_of(row[q]) >= lo && (uint32_t)(32 * lane + q) < rem) << q;
            uint32_t tot;
            const uint32_t off = warp_excl_scan((uint32_t)__popc(m), &tot);
            if (!v_ovf) {
                float* dst = vseg + v_pos + off;
                uint32_t mm = m;
                while (mm) {
                    const int q = __ffs(mm) - 1;
                    mm &= mm - 1;
                    *dst++ = row[q];
                }
                v_pos += tot;
                v_left -= tot;
            }
            P.vmask[(size_t)rec * 32 + lane] = m;
            __syncwarp();
        }
        if (store) { ch_pos += t_int; ch_left -= t_int; }
        a_gt += t_gt; a_int += t_int; a_hi += t_hi; a_lo += t_lo;
        __syncwarp();
    };

    uint32_t it = r.it0;
    {
        const uint32_t e0 = r.e0;
#pragma unroll
        for (int v = 0; v < WVEC; ++v) rt.load_step(v, r.xp, r.bp, e0, r.n - e0, lane);
    }
    for (;;) {
        // the next item: the same run, or the next counted run
        uint32_t it2 = it + 1;
        CountRun r2 = r;
        bool more = true;
        if (it2 >= r.end) {
            more = count_run_at(P, step == 1 ? r.end : it + step, end, step, r2);
            it2 = r2.it0;
        }
        count_tile(r, it, more, r2, it2);
        if (!more) break;
        it = it2;
        r = r2;
    }
    seal();
    flush();
}

// ---------------------------------------------------------------------------
// decide: where is rank k relative to the band?
// ---------------------------------------------------------------------------
__global__ void k_decide(Plan P) {
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= P.K * P.n_units) return;
    Unit& U = P.units[idx];
    if (U.state != ST_BAND) return;
    // rank k counted from the top: c_gt keys lie above the band, then the
    // band's n_int keys: c_hi equal to hi, the interior, c_lo equal to lo
    const long long c_gt = (long long)U.c_gt, c_hi = (long long)U.c_hi, c_lo = (long long)U.c_lo;
    const long long nband = (long long)U.n_int;
    const long long r = U.k - c_gt;
    U.r_src = SRC_CAND;
    if (U.mode_t) {
        // fused pass: the band holds A candidates above t^, the E keys equal
        // to t^ (not candidates), and the candidates below t^
        const long long A = (long long)U.c_abv, E = (long long)U.c_eq;
        const long long tot = nband + E;
        if (r >= 1 && r <= tot && !U.overflow) {
            if (r > A && r <= A + E) {
                U.t = U.that; U.count_above = c_gt + A; U.ties = E; U.need = r - A; U.tie_src = TIE_EQ_HI;
                U.state = ST_TKNOWN;
            } else {
                U.r_base = U.lo;
                U.r_pshift = bitlen32(U.hi - U.lo);
                U.r_prefix = 0;
                U.r_rank = (r <= A) ? r : r - E;
                U.r_above = (r <= A) ? c_gt : c_gt + E;
                U.state = ST_RADIX;
            }
        } else {
            U.fallback = 1;
            U.r_src = SRC_DATA;
            U.r_base = 0;
            U.r_pshift = 31;
            U.r_prefix = 0;
            U.r_rank = U.k;
            U.r_above = 0;
            U.state = ST_RADIX;
        }
    } else if (r >= 1 && r <= nband && !U.overflow) {
        if (r <= c_hi) {
            U.t = U.hi; U.count_above = c_gt; U.ties = c_hi; U.need = r; U.tie_src = TIE_EQ_HI;
            U.state = ST_TKNOWN;
        } else if (r > nband - c_lo) {
            U.t = U.lo; U.count_above = c_gt + nband - c_lo; U.ties = c_lo; U.need = r - (nband - c_lo);
            U.tie_src = TIE_EQ_LO;
            U.state = ST_TKNOWN;
        } else {
            // an interior key: radix select over the band's keys
            U.r_base = U.lo;
            U.r_pshift = bitlen32(U.hi - U.lo);
            U.r_prefix = 0;
            U.r_rank = r;
            U.r_above = c_gt;
            U.state = ST_RADIX;
        }
    } else {
        // exact fallback: radix select over every entry of the unit
        U.fallback = 1;
        U.r_src = SRC_DATA;
        U.r_base = 0;
        U.r_pshift = 31;
        U.r_prefix = 0;
        U.r_rank = U.k;
        U.r_above = 0;
        U.state = ST_RADIX;
    }
    // the compact candidates hold every kept entry when the threshold lies
    // in the band (t >= lo) and the unit's value segment did not overflow
    U.v_ok = (P.ccv && !U.fallback && U.v_alloc <= U.v_cap) ? 1 : 0;
    if (U.state == ST_RADIX) atomicAdd(&P.hdr->n_radix, 1);
    else atomicAdd(&P.hdr->n_tknown, 1);
}

// ---------------------------------------------------------------------------
// radix levels: one block per contiguous item range, one warp per tile, a
// shared-memory histogram per (unit, run) flushed to the unit's global one.
// Equal bins inside a warp are merged with __match_any_sync (the band keys
// hold long runs of exact ties).  Each bin also keeps its smallest and
// largest key (the smallest as the maximum of complements, so zero-filled
// memory is the identity), which lets the pick stop at a single-key bin.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void hist_add(uint32_t* h, uint32_t* mxc, uint32_t* mx, int bin, uint32_t key,
                                         bool valid) {
    const unsigned active = __ballot_sync(0xFFFFFFFFu, valid);
    if (!valid) return;
    // lanes with equal bins form disjoint groups; each reduces over its own mask
    const unsigned grp = __match_any_sync(active, bin);
    const int leader = __ffs(grp) - 1;
    const uint32_t kmin = __reduce_min_sync(grp, key);
    const uint32_t kmax = __reduce_max_sync(grp, key);
    if ((int)(threadIdx.x & 31) == leader) {
        atomicAdd(&h[bin], (uint32_t)__popc(grp));
        atomicMax(&mxc[bin], ~kmin);
        atomicMax(&mx[bin], kmax);
    }
}

// A unit in radix select over a pool filled by k_count (not the fused pass,
// whose pool is not sealed) and large enough to scan as one flat array.
__device__ __forceinline__ bool radix_flat(const Plan& P, const Unit& U) {
    return P.scope == ISO_SCOPE_GLOBAL && U.state == ST_RADIX && U.r_src == SRC_CAND && !U.mode_t && !U.overflow &&
           U.n_alloc >= RADIX_FLAT_MIN;
}

// Large pools (radix_flat): every block takes a slice of the unit's pool
// (sealed slots hold KEY_NONE), read consecutively by each warp.  A band
// where a few keys hold most entries sends many keys to a few bins, so the
// counts are kept per warp (no two warps add to one counter), and instead of
// per-bin minima and maxima each bin records its first key and whether
// another key was seen: what the pick needs to tell a single-key bin.  RADIX_FLAT_SMEM bytes of dynamic shared
// memory: WPB count arrays, the first keys, the flags.
__global__ void __launch_bounds__(TPB) k_radix_flat(Plan P) {
    extern __shared__ uint32_t fsm[];
    if (*(volatile int32_t*)&P.hdr->n_radix == 0) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t* const wc = fsm + warp * RADIX_BINS;
    uint32_t* const bkey = fsm + WPB * RADIX_BINS;
    uint32_t* const mixed = bkey + RADIX_BINS;
    for (int b = threadIdx.x; b < (WPB + 2) * RADIX_BINS; b += blockDim.x)
        fsm[b] = (b >= WPB * RADIX_BINS && b < (WPB + 1) * RADIX_BINS) ? KEY_NONE : 0u;
    __syncthreads();
    const int KU = P.K * P.n_units;
    for (int u = 0; u < KU; ++u) {
        const Unit& U = P.units[u];
        if (!radix_flat(P, U)) continue;                  // the same for every thread
        const int pshift = U.r_pshift;
        const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
        const int nb = 1 << (pshift - shift);
        const uint32_t base = U.r_base, prefix = U.r_prefix;
        const uint32_t* cs = P.cand + U.cand_off;
        const long long n = (long long)U.n_alloc;
        // a warp takes FLAT_KEYS consecutive slots per step: four 16-byte
        // loads per lane issued together, then one count per key into the
        // warp's own array (lanes of one warp with equal bins are the only
        // conflicts), and the bin's first key compared with each key
        constexpr int FLAT_VEC = 4, FLAT_KEYS = 32 * 4 * FLAT_VEC;
        const bool vec = (reinterpret_cast<uintptr_t>(cs) & 15u) == 0;
        for (long long q0 = ((long long)blockIdx.x * WPB + warp) * FLAT_KEYS; q0 < n;
             q0 += (long long)gridDim.x * WPB * FLAT_KEYS) {
            uint32_t kk[4 * FLAT_VEC];
#pragma unroll
            for (int j = 0; j < FLAT_VEC; ++j) {
                const long long q = q0 + (long long)(j * 32 + lane) * 4;
                if (vec && q + 4 <= n) {
                    const uint4 w = *reinterpret_cast<const uint4*>(cs + q);
                    kk[4 * j] = w.x; kk[4 * j + 1] = w.y; kk[4 * j + 2] = w.z; kk[4 * j + 3] = w.w;
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i) kk[4 * j + i] = q + i < n ? cs[q + i] : KEY_NONE;
                }
            }
#pragma unroll
            for (int i = 0; i < 4 * FLAT_VEC; ++i) {
                const uint32_t v = kk[i] - base;
                if (kk[i] != KEY_NONE && (v >> pshift) == prefix) {
                    const int bin = (int)((v >> shift) & (uint32_t)(nb - 1));
                    atomicAdd(&wc[bin], 1u);
                    uint32_t bk = bkey[bin];
                    if (bk == KEY_NONE) {
                        const uint32_t old = atomicCAS(&bkey[bin], KEY_NONE, kk[i]);
                        bk = old == KEY_NONE ? kk[i] : old;
                    }
                    if (kk[i] != bk) mixed[bin] = 1u;
                }
            }
        }
        __syncthreads();
        // a single key k: (max, max of complements) = (k, ~k); several: both
        // all ones, so the pick's minimum (the complement) and maximum differ
        for (int b = threadIdx.x; b < nb; b += blockDim.x) {
            uint32_t c = 0;
#pragma unroll
            for (int w = 0; w < WPB; ++w) { c += fsm[w * RADIX_BINS + b]; fsm[w * RADIX_BINS + b] = 0; }
            if (c) {
                const bool mx = mixed[b] != 0;
                const uint32_t bk = bkey[b];
                atomicAdd(&P.hist[(long long)u * RADIX_BINS + b], c);
                atomicMax(&P.hmx[(long long)u * RADIX_BINS + b], mx ? 0xFFFFFFFFu : bk);
                atomicMax(&P.hmxc[(long long)u * RADIX_BINS + b], mx ? 0xFFFFFFFFu : ~bk);
            }
            bkey[b] = KEY_NONE;
            mixed[b] = 0;
        }
        __syncthreads();
    }
}

template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(TPB) k_radix_hist(Plan P) {
    __shared__ uint32_t s_hist[RADIX_BINS];
    __shared__ uint32_t s_mxc[RADIX_BINS];
    __shared__ uint32_t s_mx[RADIX_BINS];
    if (*(volatile int32_t*)&P.hdr->n_radix == 0) return;
    for (int b = threadIdx.x; b < RADIX_BINS; b += blockDim.x) { s_hist[b] = 0; s_mxc[b] = 0; s_mx[b] = 0; }
    __syncthreads();
    const long long items = (long long)P.K * P.n_tiles;
    const long long per = (items + gridDim.x - 1) / gridDim.x;
    const long long beg = blockIdx.x * per;
    const long long end = (beg + per < items) ? beg + per : items;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    long long it = beg;
    while (it < end) {
        Cursor c;
        cursor_at(P, it, c);
        const long long run_end = c.run_end < end ? c.run_end : end;
        const TensorDesc& d = P.tens[c.t];
        Unit* U = (d.flags & TF_TRIM) ? unit_of(P, c.i, d) : nullptr;
        if (!U || U->state != ST_RADIX || radix_flat(P, *U)) { it = run_end; continue; }
        const long long ui = U - P.units;
        const int pshift = U->r_pshift;
        const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
        const int nb = 1 << (pshift - shift);
        const uint32_t base = U->r_base, prefix = U->r_prefix;
        const long long ntile = run_end - it;
        if (U->r_src == SRC_CAND) {
            // one tile's candidate list per thread; runs of one bin (ties)
            // become one update
            const uint32_t* cs = P.cand + U->cand_off;
            for (long long q = threadIdx.x; q < ntile; q += blockDim.x) {
                const uint2 r = P.tcand[(long long)c.i * P.n_tiles + c.g + q];
                int cb = -1;
                uint32_t cn = 0, cmin = 0, cmax = 0;
                for (uint32_t j = 0; j < r.y; ++j) {
                    const uint32_t kk = cs[r.x + j];
                    const uint32_t v = kk - base;
                    if ((v >> pshift) != prefix) continue;
                    const int bin = (v >> shift) & (nb - 1);
                    if (bin != cb) {
                        if (cb >= 0) { atomicAdd(&s_hist[cb], cn); atomicMax(&s_mxc[cb], ~cmin); atomicMax(&s_mx[cb], cmax); }
                        cb = bin; cn = 0; cmin = kk; cmax = kk;
                    }
                    cn++;
                    cmin = min(cmin, kk);
                    cmax = max(cmax, kk);
                }
                if (cb >= 0) { atomicAdd(&s_hist[cb], cn); atomicMax(&s_mxc[cb], ~cmin); atomicMax(&s_mx[cb], cmax); }
            }
        } else {
            // full data, one tile per warp
            const void* x = P.xptr[c.i * P.n_tensors + c.t];
            for (long long q = warp; q < ntile; q += WPB) {
                RawTile<XT, BT, CK> rt;
                const long long e0 = (c.g + q - d.tile_base) * TILE;
                rt.load(x, d.base, e0, d.numel, lane);
#pragma unroll
                for (int v = 0; v < WVEC; ++v) {
                    float tau[VEC];
                    rt.tau(v, tau);
                    const long long e = e0 + v * (32 * VEC) + lane * VEC;
#pragma unroll
                    for (int j = 0; j < VEC; ++j) {
                        const uint32_t kk = key_of(tau[j]);
                        const bool ok = (e + j < d.numel) && (kk >> pshift) == prefix;
                        hist_add(s_hist, s_mxc, s_mx, (kk >> shift) & (nb - 1), kk, ok);
                    }
                }
            }
        }
        __syncthreads();
        for (int b = threadIdx.x; b < nb; b += blockDim.x) {
            if (s_hist[b]) {
                atomicAdd(&P.hist[ui * RADIX_BINS + b], s_hist[b]);
                atomicMax(&P.hmxc[ui * RADIX_BINS + b], s_mxc[b]);
                atomicMax(&P.hmx[ui * RADIX_BINS + b], s_mx[b]);
                s_hist[b] = 0;
                s_mxc[b] = 0;
                s_mx[b] = 0;
            }
        }
        __syncthreads();
        it = run_end;
    }
}

__global__ void __launch_bounds__(TPB) k_radix_pick(Plan P) {
    __shared__ long long s_scan[33];
    __shared__ int s_bin;
    __shared__ long long s_above;
    Unit& U = P.units[blockIdx.x];
    if (U.state != ST_RADIX) return;
    const long long hb = (long long)blockIdx.x * RADIX_BINS;
    uint32_t* h = P.hist + hb;
    const int pshift = U.r_pshift;
    const int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
    const int nb = 1 << (pshift - shift);
    block_find_from_top(h, nb, U.r_rank, s_scan, &s_bin, &s_above);
    const int b = s_bin;
    const long long above = s_above;
    const uint32_t cnt = h[b];
    const uint32_t kmin = ~P.hmxc[hb + b], kmax = P.hmx[hb + b];
    __syncthreads();
    for (int q = threadIdx.x; q < nb; q += blockDim.x) { h[q] = 0; P.hmxc[hb + q] = 0; P.hmx[hb + q] = 0; }
    if (threadIdx.x == 0) {
        U.r_rank -= above;
        U.r_above += above;
        if (shift == 0 || kmin == kmax) {
            // the bin is a single key: the threshold
            U.t = kmax;
            U.count_above = U.r_above;
            U.ties = cnt;
            U.need = U.r_rank;
            U.tie_src = TIE_ARRAY;
            U.state = ST_TKNOWN;
            atomicSub(&P.hdr->n_radix, 1);
            atomicAdd(&P.hdr->n_tknown, 1);
        } else {
            U.r_prefix = (U.r_prefix << (pshift - shift)) | (uint32_t)b;
            U.r_pshift = shift;
        }
    }
}

// ---------------------------------------------------------------------------
// per-tile counts of keys == t (partial ties), and for the K = 1 ISO
// coefficient the sum of tau^2 over the candidates above t
// ---------------------------------------------------------------------------
template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(TPB) k_tie(Plan P) {
    if (*(volatile int32_t*)&P.hdr->n_tknown == 0) return;
    const long long items = (long long)P.K * P.n_tiles;
    const long long per = (items + gridDim.x - 1) / gridDim.x;
    const long long beg = blockIdx.x * per;
    const long long end = (beg + per < items) ? beg + per : items;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    long long it = beg;
    while (it < end) {
        Cursor c;
        cursor_at(P, it, c);
        const long long run_end = c.run_end < end ? c.run_end : end;
        const TensorDesc& d = P.tens[c.t];
        Unit* U = (d.flags & TF_TRIM) ? unit_of(P, c.i, d) : nullptr;
        const bool arr = U && U->state == ST_TKNOWN && U->tie_src == TIE_ARRAY;
        const bool want_cnt = arr && U->need < U->ties;
        const bool want_g = arr && U->want_gamma;
        if (!want_cnt && !want_g) { it = run_end; continue; }
        const uint32_t tk = U->t;
        const long long ntile = run_end - it;
        uint32_t* tc = P.tcnt + (long long)c.i * P.n_tiles + c.g;
        double g_warp = 0.0;
        if (U->r_src == SRC_CAND) {
            // one tile's candidate list per thread
            const uint32_t* cs = P.cand + U->cand_off;
            for (long long q0 = 0; q0 < ntile; q0 += blockDim.x) {
                const long long q = q0 + threadIdx.x;
                uint32_t cnt = 0;
                float fg = 0.0f;
                if (q < ntile) {
                    const uint2 r = P.tcand[(long long)c.i * P.n_tiles + c.g + q];
                    for (uint32_t j = 0; j < r.y; ++j) {
                        const uint32_t kk = cs[r.x + j];
                        cnt += (kk == tk);
                        if (want_g && kk > tk) { const float f = __uint_as_float(kk); fg = __fmaf_rn(f, f, fg); }
                    }
                    if (want_cnt) tc[q] = cnt;
                }
                g_warp += (double)fg;
            }
        } else {
            const void* x = P.xptr[c.i * P.n_tensors + c.t];
            for (long long q = warp; q < ntile; q += WPB) {
                RawTile<XT, BT, CK> rt;
                const long long e0 = (c.g + q - d.tile_base) * TILE;
                rt.load(x, d.base, e0, d.numel, lane);
                uint32_t cnt = 0;
                float fg = 0.0f;
#pragma unroll
                for (int v = 0; v < WVEC; ++v) {
                    float tau[VEC];
                    rt.tau(v, tau);
                    const long long e = e0 + v * (32 * VEC) + lane * VEC;
#pragma unroll
                    for (int j = 0; j < VEC; ++j) {
                        const uint32_t kk = key_of(tau[j]);
                        const bool ok = e + j < d.numel;
                        cnt += (ok && kk == tk);
                        if (want_g && ok && kk > tk) fg = __fmaf_rn(tau[j], tau[j], fg);
                    }
                }
                cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
                if (want_cnt && lane == 0) tc[q] = cnt;
                g_warp += (double)fg;
            }
        }
        if (want_g) {
            g_warp = warp_sum(g_warp);
            if (lane == 0 && g_warp != 0.0) atomicAdd(&U->gamma_rad, g_warp);
        }
        it = run_end;
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
    s.flags = (U.fallback ? 1u : 0u) | (U.mode_t ? 2u : 0u) | (U.overflow ? 8u : 0u) | (U.v_ok ? 32u : 0u);
    s.k = U.k;
    s.count_above = (U.state == ST_DONE) ? U.count_above : 0;
    s.ties_at_thresh = (U.state == ST_DONE) ? U.ties : 0;
    s.ties_taken = (U.state == ST_DONE) ? U.need : 0;
    P.st_units[(long long)i * P.st_units_stride + P.st_unit_base + u] = s;
}

// The per-tile tie counts the cut of unit U scans.
__device__ __forceinline__ const uint32_t* cut_src(const Plan& P, const Unit& U) {
    return ((U.tie_src == TIE_EQ_HI) ? P.teq_hi : (U.tie_src == TIE_EQ_LO) ? P.teq_lo : P.tcnt) +
           (long long)U.expert * P.n_tiles;
}
__device__ __forceinline__ bool cut_split(const Plan& P, const Unit& U) {
    return P.scope == ISO_SCOPE_GLOBAL && U.state == ST_TKNOWN && U.need < U.ties &&
           U.tile_end - U.tile_begin >= CUT_SPLIT_MIN;
}

// For units with many tiles: the tie counts summed over RADIX_BINS chunks of
// consecutive tiles (chunk c holds tiles tile_begin + c * per ...), into the
// unit's histogram row (free once the radix select is over).  One warp per
// chunk, consecutive loads.
__global__ void __launch_bounds__(TPB) k_cut_part(Plan P) {
    const int lane = threadIdx.x & 31;
    const long long gw = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nw = ((long long)gridDim.x * blockDim.x) >> 5;
    const int KU = P.K * P.n_units;
    for (int u = 0; u < KU; ++u) {
        const Unit& U = P.units[u];
        if (!cut_split(P, U)) continue;
        const long long nt = U.tile_end - U.tile_begin;
        const long long per = (nt + RADIX_BINS - 1) / RADIX_BINS;
        const uint32_t* src = cut_src(P, U);
        for (long long c = gw; c < RADIX_BINS; c += nw) {
            const long long g0 = U.tile_begin + c * per;
            const long long g1 = min(U.tile_end, g0 + per);
            uint32_t sum = 0;                      // <= per * TILE < 2^32
            for (long long g = g0 + lane; g < g1; g += 32) sum += src[g];
            sum = __reduce_add_sync(0xFFFFFFFFu, sum);
            if (lane == 0) P.hist[(long long)u * RADIX_BINS + c] = sum;
        }
    }
}

template <typename XT, typename BT, bool CKPT>
__global__ void __launch_bounds__(CUT_TPB) k_cut(Plan P) {
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
        // 1. the tile that holds the need-th tie (tiles in unit order); a
        //    unit with many tiles first picks the chunk from k_cut_part's sums
        const uint32_t* src = cut_src(P, U);
        long long lo_t = U.tile_begin, hi_t = U.tile_end, need = U.need;
        if (cut_split(P, U)) {
            __shared__ long long s_c0, s_c1, s_before;
            const long long nt = U.tile_end - U.tile_begin;
            const long long per_c = (nt + RADIX_BINS - 1) / RADIX_BINS;
            const uint32_t* cs = P.hist + (long long)idx * RADIX_BINS;
            constexpr int CPT = RADIX_BINS / CUT_TPB;          // chunks per thread
            long long local = 0;
#pragma unroll
            for (int q = 0; q < CPT; ++q) local += cs[threadIdx.x * CPT + q];
            if (threadIdx.x == 0) { s_c0 = -1; s_c1 = -1; s_before = 0; }
            long long tot;
            const long long excl = block_excl_scan(local, s_scan, &tot);
            if (excl < need && need <= excl + local) {
                long long acc = excl;
                for (int q = 0; q < CPT; ++q) {
                    const long long c = threadIdx.x * CPT + q;
                    if (need <= acc + cs[c]) {
                        s_c0 = U.tile_begin + c * per_c;
                        s_c1 = min(U.tile_end, s_c0 + per_c);
                        s_before = acc;
                        break;
                    }
                    acc += cs[c];
                }
            }
            __syncthreads();
            if (s_c0 >= 0) { lo_t = s_c0; hi_t = s_c1; need -= s_before; }
        }
        const long long nt = hi_t - lo_t;
        const long long per = (nt + blockDim.x - 1) / blockDim.x;
        const long long j0 = lo_t + threadIdx.x * per;
        const long long j1 = (j0 + per < hi_t) ? j0 + per : hi_t;
        auto tile_ties = [&](long long g) -> long long { return src[g]; };
        long long local = 0;
        {
            // 16-byte loads where the chunk allows
            long long g = j0;
            for (; g < j1 && ((uintptr_t)(src + g) & 15); ++g) local += src[g];
            // eight 16-byte loads in flight at a time (a large unit gives a
            // thread a hundred tiles and more)
            for (; g + 32 <= j1; g += 32) {
                uint4 v[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) v[q] = *reinterpret_cast<const uint4*>(src + g + 4 * q);
#pragma unroll
                for (int q = 0; q < 8; ++q) local += (long long)v[q].x + v[q].y + v[q].z + v[q].w;
            }
            for (; g + 4 <= j1; g += 4) {
                const uint4 v = *reinterpret_cast<const uint4*>(src + g);
                local += (long long)v.x + v.y + v.z + v.w;
            }
            for (; g < j1; ++g) local += src[g];
        }
        long long total;
        const long long excl = block_excl_scan(local, s_scan, &total);
        if (excl < need && need <= excl + local) {
            long long acc = excl;
            for (long long g = j0; g < j1; ++g) {
                const long long cnt = tile_ties(g);
                if (need <= acc + cnt) { s_tile = g; s_rem = need - acc; break; }
                acc += cnt;
            }
        }
        __syncthreads();
        if (s_tile < U.tile_begin || s_tile >= U.tile_end) {
            // the tie counts do not reach `need`: inconsistent state, keep every tie
            if (threadIdx.x == 0) { set_status(P.hdr, ISO_ERR_CUDA); U.cut = CUT_ALL; }
        } else {
            // 2. inside that tile, the rem-th entry with key == t in index order:
            //    4 consecutive entries per thread, ordered block scan
            const long long g = s_tile;
            const long long rem = s_rem;
            const int t = tensor_of_tile(P.tens, P.n_tensors, g);
            const TensorDesc& d = P.tens[t];
            const void* x = P.xptr[i * P.n_tensors + t];
            constexpr int PER = TILE / CUT_TPB;
            const long long eb = (g - d.tile_base) * TILE + (long long)threadIdx.x * PER;
            uint32_t mine = 0;
            for (int j = 0; j < PER; ++j) {
                const long long e = eb + j;
                if (e < d.numel && key_of(TauSrc<XT, BT, CKPT>::load1(x, d.base, e)) == U.t) mine++;
            }
            uint32_t tot32;
            const uint32_t before = block_excl_scan(mine, s_scan32, &tot32);
            if (before < rem && rem <= before + mine) {
                uint32_t acc = before;
                for (int j = 0; j < PER; ++j) {
                    const long long e = eb + j;
                    if (e >= d.numel) break;
                    if (key_of(TauSrc<XT, BT, CKPT>::load1(x, d.base, e)) == U.t && ++acc == rem) {
                        s_pos = ((P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0) + e;
                        break;
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
    if (threadIdx.x == 0) {
        if (U.want_gamma) {
            // sum of tau^2 over the kept entries: above the band (count pass),
            // the band keys above t, and the kept ties
            const double ft2 = sq(U.t);
            double above;
            if (U.r_src == SRC_DATA) above = U.gamma_rad;              // every entry above t
            else if (U.mode_t) {
                // fused pass: gamma_band holds the candidates above t^
                if (U.tie_src == TIE_EQ_HI) above = U.gamma_acc + U.gamma_band;   // t == t^
                else above = U.gamma_acc + U.gamma_rad + (U.t < U.that ? (double)U.c_eq * sq(U.that) : 0.0);
            }
            else if (U.tie_src == TIE_EQ_HI) above = U.gamma_acc;      // nothing in the band above hi
            else if (U.tie_src == TIE_EQ_LO) above = U.gamma_acc + U.gamma_band;
            else above = U.gamma_acc + U.gamma_rad;                  // candidates above t
            U.gamma = above + (double)U.need * ft2;
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
    template __global__ void k_csample<XT, BT, CK>(Plan);                     \
    template __global__ void k_count<XT, BT, CK, false>(Plan);                \
    template __global__ void k_count<XT, BT, CK, true>(Plan);                 \
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
