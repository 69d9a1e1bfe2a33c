// iso_block.cu -- TopKMask with per-block thresholds (BLOCK scope).
//
// Each unit is one block_rows x block_cols tile of a row-major tensor, in
// row-major tile order; entries inside a tile keep the tensor's own index
// order, so "lowest index first" among equal |tau| is the tile's row-major
// order.  One CTA holds a whole unit on chip: it loads the unit's keys into
// shared memory, finds the k-th largest key by an 11/11/9-bit radix select,
// and resolves the ties by an ordered block scan.  The result (t, cut) feeds
// the same streaming apply pass as the other scopes.
#include "iso_kernels.cuh"

namespace iso {

__device__ __forceinline__ long long k_of_density_b(double rho, long long n) {
    double kk = floor(__dadd_rn(__dmul_rn(rho, (double)n), 0.5));
    if (kk < 0.0) kk = 0.0;
    if (kk > (double)n) kk = (double)n;
    return (long long)kk;
}

__device__ void block_find_from_top_b(const uint32_t* hist, int nb, long long rank,
                                      long long* sm_scan, int* res_bin, long long* res_above) {
    const int per = (nb + blockDim.x - 1) / blockDim.x;
    const int j0 = threadIdx.x * per;
    if (threadIdx.x == 0) { *res_bin = 0; *res_above = 0; }
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

// keys sit at q + q / 32: a thread walking its own contiguous range and a
// warp walking consecutive entries are both free of bank conflicts
__device__ __forceinline__ int kpad(int q) { return q + (q >> 5); }

template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(BLOCK_TPB, BLOCK_CTAS_PER_SM) k_block_select(Plan P) {
    extern __shared__ __align__(16) uint32_t s_keys[];      // kpad(BLOCK_MAX_ENTRIES)
    __shared__ uint32_t s_hist[RADIX_BINS];
    __shared__ long long s_scan[33];
    __shared__ uint32_t s_scan32[33];
    __shared__ double s_dred[33];
    __shared__ int s_bin;
    __shared__ long long s_above;
    __shared__ long long s_cutq;
    __shared__ uint32_t s_or;

    const int idx = blockIdx.x;
    const int i = idx / P.n_units, u = idx % P.n_units;
    // owning tensor: last tensor whose first unit is <= u and that has blocks
    int lo = 0, hi = P.n_tensors - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (P.tens[mid].unit <= u) lo = mid; else hi = mid - 1;
    }
    while (lo > 0 && P.tens[lo].nblocks == 0) --lo;
    const int t = lo;
    const TensorDesc& d = P.tens[t];
    Unit& U = P.units[idx];
    const int b = u - d.unit;
    const int br = b / d.bpr, bc = b % d.bpr;
    const long long r0 = (long long)br * P.block_rows, c0 = (long long)bc * P.block_cols;
    const long long h = min((long long)P.block_rows, d.rows - r0);
    const long long w = min((long long)P.block_cols, d.cols - c0);
    const int n = (int)(h * w);
    auto stats = [&](uint32_t tk, long long k, long long above, long long ties, long long need) {
        if (!P.st_units) return;
        iso_unit_stats s;
        s.thresh_key = tk; s.flags = 0; s.k = k; s.count_above = above;
        s.ties_at_thresh = ties; s.ties_taken = need;
        P.st_units[(long long)i * P.st_units_stride + P.st_unit_base + u] = s;
    };
    const void* x = P.xptr[i * P.n_tensors + t];
    const bool vec = (w % VEC == 0) && (d.cols % VEC == 0) && (c0 % VEC == 0);
    // fused K = 1 update (TIES / masked update): the block's outputs are
    // written here, theta_0 + lambda tau for the kept entries, theta_0 else
    const bool obf = sizeof(BT) == 2;
    auto apply_block = [&](uint32_t tk, long long cut, bool keep_all) {
        if (vec) {
            const int w8 = (int)(w / VEC);
            for (int q8 = threadIdx.x; q8 < n / VEC; q8 += blockDim.x) {
                const int rr = q8 / w8, cc = (q8 - rr * w8) * VEC;
                const long long e = (r0 + rr) * d.cols + c0 + cc;
                float th0[VEC], tau[VEC], o[VEC];
                load8_tail<BT>(d.base, e, d.numel, th0);
                TauSrc<XT, BT, CK>::load8(x, d.base, e, d.numel, tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    const uint32_t kk = key_of(tau[j]);
                    const bool kept = keep_all || kk > tk || (kk == tk && e + j < cut);
                    o[j] = kept ? out_of(th0[j], tau[j], P.lambda) : th0[j];
                }
                store8(d.out, e, d.numel, o, obf);
            }
        } else {
            for (int q = threadIdx.x; q < n; q += blockDim.x) {
                const int rr = q / (int)w, cc = q - rr * (int)w;
                const long long e = (r0 + rr) * d.cols + c0 + cc;
                const float th0 = Load8<BT>::one(d.base, e);
                const float tau = TauSrc<XT, BT, CK>::load1(x, d.base, e);
                const uint32_t kk = key_of(tau);
                const bool kept = keep_all || kk > tk || (kk == tk && e < cut);
                const float o = kept ? out_of(th0, tau, P.lambda) : th0;
                if (obf) static_cast<__nv_bfloat16*>(d.out)[e] = __float2bfloat16_rn(o);
                else static_cast<float*>(d.out)[e] = o;
            }
        }
    };
    if (!(d.flags & TF_TRIM)) {
        if (threadIdx.x == 0) {
            U.state = ST_OFF; U.k = -1; U.t = 0; U.cut = CUT_ALL;
            stats(KEY_NONE, -1, 0, 0, 0);
        }
        if (P.fuse_block) apply_block(0u, CUT_ALL, true);
        return;
    }
    // k in binary64 by one thread (binary64 is slow on this GPU), then shared
    __shared__ long long s_k;
    if (threadIdx.x == 0) s_k = k_of_density_b(P.density, n);
    __syncthreads();
    const long long k = s_k;
    if (k == 0) {
        if (threadIdx.x == 0) {
            U.state = ST_NONE; U.k = 0; U.t = KEY_NONE; U.cut = 0;
            stats(KEY_NONE, 0, 0, 0, 0);
        }
        if (P.fuse_block) apply_block(KEY_NONE, 0, false);
        return;
    }
    const bool want_gamma = (P.op == ISO_OP_ISO) && (P.K == 1);

    // Full block of BLOCK_TPB x BFE entries in rows of a multiple of BFE: each
    // thread holds BFE consecutive entries (block order) in registers -- their
    // keys and one word of signs, from which each tau is rebuilt exactly --
    // and the
    // threshold is found bit by bit from the top: t is the largest key value v
    // with #{key >= v} >= k, so a bit is kept when the block still counts k
    // keys at or above the prefix with that bit set.  No atomics, no bank
    // conflicts; one block sum per bit below the highest.
    constexpr int BFE = BLOCK_MAX_ENTRIES / BLOCK_TPB;
    if (n == BLOCK_TPB * BFE && w % BFE == 0 && (d.cols % VEC) == 0 && (c0 % VEC) == 0 &&
        blockDim.x == BLOCK_TPB) {
        const int tq = threadIdx.x * BFE;
        const int rr = tq / (int)w, cc = tq - rr * (int)w;
        const long long ea = (r0 + rr) * d.cols + c0 + cc;     // tensor position of the thread's first entry
        static_assert(BFE <= 32, "one sign word per thread");
        uint32_t key[BFE];
        uint32_t sgn = 0;
#pragma unroll
        for (int g = 0; g < BFE / VEC; ++g) {
            float t8[VEC];
            TauSrc<XT, BT, CK>::load8(x, d.base, ea + g * VEC, d.numel, t8);
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const uint32_t b = __float_as_uint(t8[j]);
                key[g * VEC + j] = b & 0x7FFFFFFFu;
                sgn |= (b >> 31) << (g * VEC + j);
            }
        }
        auto tau_of = [&](int j) -> float { return __uint_as_float(key[j] | (((sgn >> j) & 1u) << 31)); };
        uint32_t kmax = 0, kor = 0;
#pragma unroll
        for (int j = 0; j < BFE; ++j) { kmax = max(kmax, key[j]); kor |= key[j]; }
        if (kmax >= KEY_INF) set_status(P.hdr, ISO_ERR_NONFINITE);
        kor = __reduce_or_sync(0xFFFFFFFFu, kor);
        if (threadIdx.x == 0) s_or = 0;
        __syncthreads();
        if ((threadIdx.x & 31) == 0 && kor) atomicOr(&s_or, kor);
        __syncthreads();
        const int low = s_or ? __ffs(s_or) - 1 : 31;
        const int top = s_or ? 31 - __clz(s_or) : 0;
        // one barrier per bit: warp sums go to one of three counters; the
        // counter of the bit after next is cleared meanwhile (its last reads
        // were before this bit's barrier, its next adds come after the next one)
        __shared__ uint32_t s_cnt[3];
        if (threadIdx.x < 3) s_cnt[threadIdx.x] = 0;
        __syncthreads();
        uint32_t prefix = 0;
        int cur = 0;
        for (int bit = top; bit >= low; --bit) {
            const uint32_t cand = prefix | (1u << bit);
            uint32_t c = 0;
#pragma unroll
            for (int j = 0; j < BFE; ++j) c += key[j] >= cand;
            c = __reduce_add_sync(0xFFFFFFFFu, c);
            if ((threadIdx.x & 31) == 0 && c) atomicAdd(&s_cnt[cur], c);
            __syncthreads();
            if ((long long)s_cnt[cur] >= k) prefix = cand;
            const int nxt2 = (cur + 2) % 3;
            if (threadIdx.x == 0) s_cnt[nxt2] = 0;
            cur = (cur + 1) % 3;
        }
        const uint32_t tk = prefix;
        uint32_t above = 0, ties = 0;
#pragma unroll
        for (int j = 0; j < BFE; ++j) { above += key[j] > tk; ties += key[j] == tk; }
        uint32_t tot_ties;
        const uint32_t ties_before = block_excl_scan(ties, s_scan32, &tot_ties);
        const uint32_t tot_above = block_sum(above, s_scan32);
        const long long need = k - (long long)tot_above;
        if (threadIdx.x == 0) s_cutq = CUT_ALL;
        __syncthreads();
        if (need < (long long)tot_ties && (long long)ties_before < need && need <= (long long)(ties_before + ties)) {
            uint32_t acc = ties_before;
#pragma unroll
            for (int j = 0; j < BFE; ++j)
                if (key[j] == tk && (long long)(++acc) == need) s_cutq = ea + j + 1;
        }
        double g = 0.0;
        if (want_gamma) {
            // squares of the entries above t as binary32 two-sum pairs, then binary64 over the block
            float sg = 0.0f, eg = 0.0f;
#pragma unroll
            for (int j = 0; j < BFE; ++j) {
                const float f = __uint_as_float(key[j]);          // |tau|: the same square
                if (key[j] > tk) two_sum_add(sg, eg, __fmul_rn(f, f));
            }
            g = block_sum((double)sg + (double)eg, s_dred);
        }
        __syncthreads();
        const long long cut = s_cutq;
        if (threadIdx.x == 0) {
            U.n = n; U.k = k; U.t = tk; U.cut = cut;
            U.count_above = tot_above; U.ties = tot_ties; U.need = need;
            U.state = ST_DONE;
            if (want_gamma) {
                const double ft = (double)__uint_as_float(tk);
                atomicAdd(&P.gram[t], g + (double)need * ft * ft);
            }
            stats(tk, k, tot_above, tot_ties, need);
        }
        if (P.fuse_block) {
#pragma unroll
            for (int gq = 0; gq < BFE / VEC; ++gq) {
                const long long e = ea + gq * VEC;
                float th0[VEC], o[VEC];
                load8_tail<BT>(d.base, e, d.numel, th0);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    const uint32_t kk = key[gq * VEC + j];
                    const bool kept = kk > tk || (kk == tk && e + j < cut);
                    o[j] = kept ? out_of(th0[j], tau_of(gq * VEC + j), P.lambda) : th0[j];
                }
                store8(d.out, e, d.numel, o, obf);
            }
        }
        return;
    }
    // keys in block order (row-major inside the block)
    bool bad = false;
    uint32_t kor = 0;                        // OR of the keys: trailing zero bits need no radix level
    if (threadIdx.x == 0) s_or = 0;
    __syncthreads();
    if (vec) {
        const int w8 = (int)(w / VEC);
        for (int q8 = threadIdx.x; q8 < n / VEC; q8 += blockDim.x) {
            const int rr = q8 / w8, cc = (q8 - rr * w8) * VEC;
            const long long e = (r0 + rr) * d.cols + c0 + cc;
            float tau[VEC];
            TauSrc<XT, BT, CK>::load8(x, d.base, e, d.numel, tau);
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const uint32_t kk = key_of(tau[j]);
                bad |= kk >= KEY_INF;
                kor |= kk;
                s_keys[kpad(q8 * VEC + j)] = kk;
            }
        }
    } else {
        for (int q = threadIdx.x; q < n; q += blockDim.x) {
            const int rr = q / (int)w, cc = q - rr * (int)w;
            const long long e = (r0 + rr) * d.cols + c0 + cc;
            const uint32_t kk = key_of(TauSrc<XT, BT, CK>::load1(x, d.base, e));
            bad |= kk >= KEY_INF;
            kor |= kk;
            s_keys[kpad(q)] = kk;
        }
    }
    if (bad) set_status(P.hdr, ISO_ERR_NONFINITE);
    kor = __reduce_or_sync(0xFFFFFFFFu, kor);
    if ((threadIdx.x & 31) == 0 && kor) atomicOr(&s_or, kor);
    __syncthreads();
    // k-th largest key: radix levels down to the lowest bit any key has set
    // (bf16-valued task vectors leave the low 16 bits clear)
    const int low = s_or ? __ffs(s_or) - 1 : 31;
    uint32_t prefix = 0;
    long long rank = k;
    int pshift = 31;
    for (;;) {
        int shift = pshift > RADIX_BITS ? pshift - RADIX_BITS : 0;
        if (shift < low) shift = low;
        const int nb = 1 << (pshift - shift);
        for (int q = threadIdx.x; q < nb; q += blockDim.x) s_hist[q] = 0;
        __syncthreads();
        for (int q = threadIdx.x; q < n; q += blockDim.x) {
            const uint32_t v = s_keys[kpad(q)];
            if ((v >> pshift) == prefix) atomicAdd(&s_hist[(v >> shift) & (nb - 1)], 1u);
        }
        __syncthreads();
        block_find_from_top_b(s_hist, nb, rank, s_scan, &s_bin, &s_above);
        rank -= s_above;
        prefix = (prefix << (pshift - shift)) | (uint32_t)s_bin;
        __syncthreads();
        if (shift == low) break;
        pshift = shift;
    }
    const uint32_t tk = prefix << low;
    // counts above / at the threshold, and the squared norm of the kept entries
    const int per = (n + blockDim.x - 1) / blockDim.x;
    const int q0 = threadIdx.x * per;
    uint32_t above = 0, ties = 0;
    double gsum = 0.0;
    for (int q = q0; q < q0 + per && q < n; ++q) {
        const uint32_t v = s_keys[kpad(q)];
        above += v > tk;
        ties += v == tk;
        if (want_gamma && v > tk) {
            const double f = (double)__uint_as_float(v);
            gsum += f * f;
        }
    }
    uint32_t tot_ties;
    const uint32_t ties_before = block_excl_scan(ties, s_scan32, &tot_ties);
    const uint32_t tot_above = block_sum(above, s_scan32);
    const long long need = k - (long long)tot_above;
    if (threadIdx.x == 0) s_cutq = -1;
    __syncthreads();
    if (need < (long long)tot_ties) {
        if ((long long)ties_before < need && need <= (long long)(ties_before + ties)) {
            uint32_t acc = ties_before;
            for (int q = q0; q < q0 + per && q < n; ++q)
                if (s_keys[kpad(q)] == tk && (long long)(++acc) == need) { s_cutq = q; break; }
        }
    }
    __syncthreads();
    double g = 0.0;
    if (want_gamma) g = block_sum(gsum, s_dred);
    long long cut = CUT_ALL;
    if (s_cutq >= 0) {
        const long long rr = s_cutq / w, cc = s_cutq - rr * w;
        cut = (r0 + rr) * d.cols + c0 + cc + 1;
    }
    if (threadIdx.x == 0) {
        U.n = n; U.k = k; U.t = tk; U.cut = cut;
        U.count_above = tot_above; U.ties = tot_ties; U.need = need;
        U.state = ST_DONE;
        if (want_gamma) {
            const double ft = (double)__uint_as_float(tk);
            atomicAdd(&P.gram[t], g + (double)need * ft * ft);
        }
        stats(tk, k, tot_above, tot_ties, need);
    }
    if (P.fuse_block) apply_block(tk, cut, false);
}

#define ISO_BLOCK_INST(XT, BT, CK) template __global__ void k_block_select<XT, BT, CK>(Plan);
ISO_BLOCK_INST(__nv_bfloat16, __nv_bfloat16, false)
ISO_BLOCK_INST(__nv_bfloat16, float, false)
ISO_BLOCK_INST(float, __nv_bfloat16, false)
ISO_BLOCK_INST(float, float, false)
ISO_BLOCK_INST(__nv_bfloat16, __nv_bfloat16, true)
ISO_BLOCK_INST(__nv_bfloat16, float, true)
ISO_BLOCK_INST(float, __nv_bfloat16, true)
ISO_BLOCK_INST(float, float, true)

}  // namespace iso
