// iso_apply.cu -- the K = 1 update pass, the retention solve and the small
// passes around them.
//
//   k_apply  out = theta_0 + update for one expert, one read of theta_0 and
//            the expert and one write (App. F): every operator reduces to
//            update = a * m * tau with a per-tensor scale a
//              TA    a = lambda, no mask
//              TIES  a = lambda (one expert: the elected sign is its own)
//              ISO   2-D: a = c, the tensor's retention coefficient (Sec. 4.2)
//                    1-D: a = 1/K = 1, no mask                 (App. E, Algorithm 1)
//            An update of exactly zero leaves theta_0 untouched.
//            (K >= 2 and the Gram pass: iso_merge.cu)
//   k_solve  (Gamma + ridge I) c = diag Gamma on the non-zero experts, clip
//   k_mask   the mask itself as a packed bitmask
//   k_delta  tau = theta_i - theta_0 in binary32
//
// Arithmetic: binary32 with explicit round-to-nearest intrinsics (no
// contraction), experts summed in the fixed order i = 1..K.
#include "iso_kernels.cuh"

namespace iso {

// BLOCK scope: unit of entry e of tensor d
__device__ __forceinline__ int block_unit(const Plan& P, const TensorDesc& d, long long row, long long col) {
    return d.unit + (int)(row / P.block_rows) * d.bpr + (int)(col / P.block_cols);
}


// ---------------------------------------------------------------------------
// apply: one warp per tile, one contiguous tile range per warp
// ---------------------------------------------------------------------------
// the K experts' selection parameters and coefficients of one tensor
struct TensorParams {
    SelParam sp[MAXK];
    float cf[MAXK];
    const void* xs[MAXK];
    bool blk, iso2d, iso1d;
    long long pos_off;
};

__device__ __forceinline__ void tensor_params(const Plan& P, int t, int K, TensorParams& tp) {
    const TensorDesc& d = P.tens[t];
    const bool is1d = (d.flags & TF_1D) != 0;
    tp.iso2d = (P.op == ISO_OP_ISO) && !is1d;
    tp.iso1d = (P.op == ISO_OP_ISO) && is1d;
    tp.blk = (P.scope == ISO_SCOPE_BLOCK) && (d.flags & TF_TRIM);
    tp.pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
#pragma unroll
    for (int i = 0; i < MAXK; ++i) {
        if (i >= K) break;
        tp.xs[i] = P.xptr[i * P.n_tensors + t];
        tp.cf[i] = tp.iso2d ? (float)P.coef[(long long)t * K + i] : 0.0f;
        if (!tp.blk) {
            if (P.scope == ISO_SCOPE_GLOBAL && !(d.flags & TF_TRIM)) {
                // outside the one GLOBAL unit (a 1-D tensor TIES leaves
                // untrimmed): every entry kept, as an untrimmed tensor's own
                // unit record says in the other scopes
                tp.sp[i].t = 0;
                tp.sp[i].cut = CUT_ALL;
            } else {
                const Unit& U = P.units[(long long)i * P.n_units + ((P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit)];
                tp.sp[i].t = U.t;
                tp.sp[i].cut = U.cut;
            }
        }
    }
}

// K = 1: the per-tensor scale, whether the tensor is trimmed, and the packed
// threshold (t, ~cut) for tensor-local positions below 2^32
__device__ __forceinline__ void k1_params(const Plan& P, const TensorParams& tp, float* a, bool* mask,
                                          unsigned long long* thr) {
    if (P.op == ISO_OP_TA) { *a = P.lambda; *mask = false; }
    else if (tp.iso1d) { *a = 1.0f; *mask = false; }
    else if (tp.iso2d) { *a = tp.cf[0]; *mask = true; }
    else { *a = P.lambda; *mask = true; }
    // GLOBAL scope: the cut is a position in the concatenation; entry e of
    // this tensor sits at pos_off + e, so the tensor-local cut is cut - pos_off
    // clamped to [0, 2^32 - 1] (numel < 2^32 keeps every local position below)
    const long long cut = tp.sp[0].cut;
    const long long lc = (cut == CUT_ALL) ? cut : cut - tp.pos_off;
    const uint32_t c32 = (lc >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (lc <= 0 ? 0u : (uint32_t)lc);
    *thr = ((unsigned long long)tp.sp[0].t << 32) | (uint32_t)~c32;
}

// BLOCK scope: selection parameters of entry (row, col) for expert i
__device__ __forceinline__ SelParam block_param(const Plan& P, const TensorDesc& d, int i,
                                                long long row, long long col) {
    const Unit& U = P.units[(long long)i * P.n_units + block_unit(P, d, row, col)];
    SelParam s;
    s.t = U.t;
    s.cut = U.cut;
    return s;
}

template <typename XT, typename BT, bool CK, int KC>
__global__ void __launch_bounds__(TPB) k_apply(Plan P) {
    static_assert(KC == 1, "K >= 2 merges run in k_merge");
    const int K = 1;
    const int lane = threadIdx.x & 31;
    const long long W = (long long)gridDim.x * WPB;
    const long long wid = (long long)blockIdx.x * WPB + (threadIdx.x >> 5);
    // round-robin tiles (all warps sweep one window together) or one range per warp
    long long beg, end, step;
    if (PASS_INTERLEAVE) {
        beg = wid;
        end = P.n_tiles;
        step = W;
    } else {
        const long long per = (P.n_tiles + W - 1) / W;
        beg = wid * per;
        end = (beg + per < P.n_tiles) ? beg + per : P.n_tiles;
        step = 1;
    }
    if (beg >= end) return;
    const bool obf = sizeof(BT) == 2;
    int t = tensor_of_tile(P.tens, P.n_tensors, beg);
    long long t_end = P.tens[t].tile_base + (P.tens[t].numel + TILE - 1) / TILE;
    TensorParams tp;
    tensor_params(P, t, K, tp);

    {
        // K = 1: every operator reduces to theta_0 + a * (mask ? tau : 0) with a
        // per-tensor scale a (TA, TIES: lambda; ISO 2-D: c; ISO 1-D: 1/K = 1)
        // and the mask off for TA and ISO 1-D.  The whole tile sits in
        // registers while the next tile's loads are in flight.
        RawTile<XT, BT, true> cur, nxt;
        {
            const TensorDesc& d = P.tens[t];
            cur.load(tp.xs[0], d.base, (beg - d.tile_base) * TILE, d.numel, lane);
        }
        int nt = t;
        long long nt_end = t_end;
        float k1_a = 1.0f;
        bool k1_mask = true;
        unsigned long long k1_thr = 0;
        for (long long g = beg; g < end; g += step) {
            // prefetch the warp's next tile
            if (g + step < end) {
                while (g + step >= nt_end) {
                    ++nt;
                    nt_end = P.tens[nt].tile_base + (P.tens[nt].numel + TILE - 1) / TILE;
                }
                const TensorDesc& nd = P.tens[nt];
                nxt.load(P.xptr[nt], nd.base, (g + step - nd.tile_base) * TILE, nd.numel, lane);
            }
            if (g >= t_end || g == beg) {
                while (g >= t_end) { ++t; t_end = P.tens[t].tile_base + (P.tens[t].numel + TILE - 1) / TILE; }
                tensor_params(P, t, K, tp);
                k1_params(P, tp, &k1_a, &k1_mask, &k1_thr);
            }
            const TensorDesc& d = P.tens[t];
            const long long n = d.numel;
            const long long e0 = (g - d.tile_base) * TILE;
#pragma unroll
            for (int v = 0; v < WVEC; ++v) {
                const long long e = e0 + v * (32 * VEC) + lane * VEC;
                if (e >= n) continue;
                float th0[VEC], tau[VEC];
                raw_to_f32<BT>(reinterpret_cast<const uint4(&)[Lanes<BT>::N]>(cur.b[v]), th0);
                if (CK) {
                    cur.tau(v, tau);
                } else {
                    raw_to_f32<XT>(cur.x[v], tau);
                }
                float o[VEC];
                if (tp.blk) {
                    long long r = 0, cc = 0;
                    if (tp.blk) { r = e / d.cols; cc = e - r * d.cols; }
#pragma unroll
                    for (int j = 0; j < VEC; ++j) {
                        SelParam s = tp.sp[0];
                        if (tp.blk) {
                            s = block_param(P, d, 0, r, cc);
                            if (++cc == d.cols) { cc = 0; ++r; }
                        }
                        const bool sel = !k1_mask || kept(key_of(tau[j]), tp.pos_off + e + j, s);
                        const float upd = __fmul_rn(k1_a, sel ? tau[j] : 0.0f);
                        o[j] = (upd == 0.0f) ? th0[j] : __fadd_rn(th0[j], upd);
                    }
                } else {
                    // kept <=> (key, ~pos) > (t, ~cut) as one 64-bit comparison
                    const uint32_t p0 = ~(uint32_t)e;
#pragma unroll
                    for (int j = 0; j < VEC; ++j) {
                        const unsigned long long kp =
                            ((unsigned long long)key_of(tau[j]) << 32) | (uint32_t)(p0 - (uint32_t)j);
                        const bool sel = !k1_mask || kp > k1_thr;
                        const float upd = __fmul_rn(k1_a, sel ? tau[j] : 0.0f);
                        o[j] = (upd == 0.0f) ? th0[j] : __fadd_rn(th0[j], upd);
                    }
                }
                store8(d.out, e, n, o, obf);
            }
            cur = nxt;
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
        retention_solve(G, K, P.ridge, P.c_min, P.c_max, c);
    }
    for (int i = 0; i < K; ++i) P.coef[(long long)t * K + i] = c[i];
    if (P.repair) {
        // fused K = 1 pass: re-apply in full when the speculative outputs may be wrong
        const Unit& U = P.units[d.unit];
        int rep = 0;
        if ((d.flags & TF_TRIM) && U.state == ST_DONE) {
            const float a = active ? (float)c[0] : P.lambda;
            rep = (U.fallback || U.b_overflow || a != k1_spec_coef(P)) ? 1 : 0;
            if (rep && P.st_units)
                P.st_units[P.st_unit_base + d.unit].flags |= 4u | (U.b_overflow ? 16u : 0u);
        }
        P.repair[t] = rep;
    }
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
    const int lane = threadIdx.x & 31;
    const long long W = (long long)gridDim.x * WPB;
    for (long long g = (long long)blockIdx.x * WPB + (threadIdx.x >> 5); g < P.n_tiles; g += W) {
        const int t = tensor_of_tile(P.tens, P.n_tensors, g);
        const TensorDesc& d = P.tens[t];
        uint32_t* mw = mptr[t];
        if (!mw) continue;
        const long long n = d.numel;
        const long long e0 = (g - d.tile_base) * TILE;
        const bool blk = (P.scope == ISO_SCOPE_BLOCK);
        const long long pos_off = (P.scope == ISO_SCOPE_GLOBAL) ? d.uoff : 0;
        SelParam s0;
        s0.t = 0; s0.cut = 0;
        if (!blk) {
            const Unit& U = P.units[(P.scope == ISO_SCOPE_GLOBAL) ? 0 : d.unit];
            s0.t = U.t; s0.cut = U.cut;
        }
        for (int v = 0; v < WVEC; ++v) {
            const long long e = e0 + v * (32 * VEC) + lane * VEC;
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
                        s = block_param(P, d, 0, r, c);
                        if (++c == d.cols) { c = 0; ++r; }
                    }
                    if (kept(key_of(tau[j]), pos_off + e + j, s)) bits |= 1u << j;
                }
            }
            // four consecutive lanes hold 32 consecutive entries
            const int sub = lane & 3;
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

// The statistics of units that no tensor of a group trims (every tensor of
// the group is a 1-D tensor that the operator leaves untrimmed, or empty): no
// selection pass runs for such a group, so their records are written here,
// the same record the selection writes for an untrimmed unit.
__global__ void k_units_off(iso_unit_stats* st, long long stride, long long base, int n_units, int K) {
    const long long n = (long long)K * n_units;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long i = idx / n_units, u = idx % n_units;
        iso_unit_stats s;
        s.thresh_key = KEY_NONE;
        s.flags = 0;
        s.k = -1;
        s.count_above = 0;
        s.ties_at_thresh = 0;
        s.ties_taken = 0;
        st[i * stride + base + u] = s;
    }
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
    const int lane = threadIdx.x & 31;
    const long long n_tiles = A.tile_base[A.n];
    const long long W = (long long)gridDim.x * WPB;
    for (long long g = (long long)blockIdx.x * WPB + (threadIdx.x >> 5); g < n_tiles; g += W) {
        int t = 0;
        while (t + 1 < A.n && A.tile_base[t + 1] <= g) ++t;
        const long long n = A.numel[t];
        const long long e0 = (g - A.tile_base[t]) * TILE;
#pragma unroll
        for (int v = 0; v < WVEC; ++v) {
            const long long e = e0 + v * (32 * VEC) + lane * VEC;
            if (e >= n) continue;
            float a[VEC], b[VEC], o[VEC];
            load8_tail<AT>(A.a[t], e, n, a);
            load8_tail<BT>(A.b[t], e, n, b);
#pragma unroll
            for (int j = 0; j < VEC; ++j) o[j] = __fsub_rn(a[j], b[j]);
            store8(A.out[t], e, n, o, false);
        }
    }
}

// ---------------------------------------------------------------------------
// instantiations
// ---------------------------------------------------------------------------
#define ISO_APPLY_INST(XT, BT, CK)                                             \
    template __global__ void k_apply<XT, BT, CK, 1>(Plan);

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
