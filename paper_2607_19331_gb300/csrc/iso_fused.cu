// iso_fused.cu -- the K = 1 masked update in one pass over HBM.
//
// For one expert every operator reduces to
//     out = theta_0 + a * (kept ? tau : 0)                          (App. F; Sec. 4.2)
// with a per-tensor scale a: lambda for TIES, the retention coefficient c*
// for ISO (the K = 1 case of the retention system), 1 for ISO's 1-D average.
// The two-pass form reads the inputs twice: once to count (TopKMask needs the
// unit's k-th largest |tau| before any entry can be decided) and once to apply.
//
// Here a single pass does both.  With the sampled band [lo, hi] around rank k
// (k_sample) every entry above hi is kept and every entry below lo dropped
// whatever the exact threshold turns out to be; only band entries are
// undecided.  The pass therefore writes every output at once -- entries above
// hi with the coefficient a_spec the unit will have in every ordinary case,
// band entries as dropped -- and records each band entry (position and raw
// values).  Once the exact threshold and cut are known (the select chain) and
// the coefficient is exact, k_patch rewrites the band entries that are kept.
// A tensor whose band missed, whose records overflowed, or whose exact
// coefficient differs from a_spec is flagged and re-applied in full by
// k_apply, so the result is exact in every case.
#include "iso_kernels.cuh"

namespace iso {

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

#ifndef ISO_FUSED_BLOCKS_PER_SM
#define ISO_FUSED_BLOCKS_PER_SM 2
#endif
constexpr int FUSED_BLOCKS_PER_SM = ISO_FUSED_BLOCKS_PER_SM;

template <bool CK>
__global__ void __launch_bounds__(TPB, FUSED_BLOCKS_PER_SM) k_count_apply(Plan P) {
    // per warp: the tile's raw update and base values, and the offsets of its
    // band entries (lane L's j-th at j*32 + L)
    __shared__ __align__(16) uint16_t s_x[WPB][TILE];
    __shared__ __align__(16) uint16_t s_b[WPB][TILE];
    __shared__ uint16_t s_off[WPB][TILE + 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint16_t* sx = s_x[warp];
    uint16_t* sbs = s_b[warp];
    uint16_t* sol = s_off[warp] + lane;
    const uint32_t W = gridDim.x * WPB;
    const uint32_t wid = blockIdx.x * WPB + warp;
    const uint32_t items = (uint32_t)P.n_tiles;
    const uint32_t per = (items + W - 1) / W;
    const uint32_t beg = wid * per;
    const uint32_t end = min(items, beg + per);
    if (beg >= end) return;
    const unsigned FULL = 0xFFFFFFFFu;
    const float a_spec = k1_spec_coef(P);

    // per-unit accumulators and the two segments (interior keys, band records)
    Unit* au = nullptr;
    uint32_t a_gt = 0, a_int = 0;
    double d_gg = 0.0;
    uint32_t* cseg = nullptr;
    uint2* bseg = nullptr;
    uint32_t c_pos = 0, c_left = 0, c_cap = 0, b_pos = 0, b_left = 0, b_cap = 0;
    bool c_ovf = false, b_ovf = false;
    uint32_t lo = 0, hi = 0, span = 0;
    bool want_gamma = false;

    auto flush = [&]() {
        if (!au) return;
        const double gg = warp_sum(d_gg);
        if (lane == 0) {
            if (a_gt) atomicAdd(&au->c_gt, (unsigned long long)a_gt);
            if (a_int) atomicAdd(&au->n_int, (unsigned long long)a_int);
            if (want_gamma && gg != 0.0) atomicAdd(&au->gamma_acc, gg);
            if (c_ovf) au->overflow = 1;
            if (b_ovf) au->b_overflow = 1;
        }
        a_gt = a_int = 0;
        d_gg = 0.0;
    };

    // reserve n slots of a segment for one tile; returns false on overflow
    auto reserve = [&](unsigned long long* alloc, uint32_t need, uint32_t cap, uint32_t left_tiles,
                       uint32_t& pos, uint32_t& left) -> bool {
        unsigned long long start = 0;
        uint32_t req = 0;
        if (lane == 0) {
            const unsigned long long want = (unsigned long long)need * (unsigned long long)left_tiles;
            req = (uint32_t)max((unsigned long long)need, min((unsigned long long)CHUNK_MAX, want));
            start = atomicAdd(alloc, (unsigned long long)req);
        }
        start = __shfl_sync(FULL, start, 0);
        req = __shfl_sync(FULL, req, 0);
        if (start + req > cap) { left = 0; return false; }
        pos = (uint32_t)start;
        left = req;
        return true;
    };

    uint32_t run_end = beg, it0 = beg, g0 = 0, n = 0, tile_base = 0;
    const void* xp = nullptr;
    const void* bp = nullptr;
    void* op = nullptr;
    bool fuse = false, kept_all = false;
    float a_fix = 0.0f;
    uint32_t it = beg;
    while (it < end) {
        if (it >= run_end) {
            Cursor c;
            cursor_at(P, it, c);
            run_end = (uint32_t)c.run_end;
            const TensorDesc& d = P.tens[c.t];
            n = (uint32_t)d.numel;
            tile_base = (uint32_t)d.tile_base;
            xp = P.xptr[c.t];
            bp = d.base;
            op = d.out;
            it0 = it;
            g0 = (uint32_t)c.g;
            Unit* U = &P.units[d.unit];
            fuse = (d.flags & TF_TRIM) && U->state == ST_BAND;
            // a tensor whose selection is already final: untrimmed (all kept) or k = 0
            kept_all = !(d.flags & TF_TRIM);
            a_fix = (P.op == ISO_OP_ISO && (d.flags & TF_1D)) ? 1.0f : P.lambda;
            if (fuse && U != au) {
                flush();
                au = U;
                lo = U->lo;
                hi = U->hi;
                span = hi - lo;
                want_gamma = U->want_gamma != 0;
                c_cap = (uint32_t)U->cand_cap;
                cseg = P.cand + U->cand_off;
                b_cap = (uint32_t)U->brec_cap;
                bseg = P.brec + U->brec_off;
                c_left = b_left = 0;
                c_ovf = b_ovf = false;
            }
        }
        const uint32_t g = g0 + (it - it0);
        const uint32_t e0 = (g - tile_base) * TILE;
        RawTile<__nv_bfloat16, __nv_bfloat16, true> rt;
        rt.load(xp, bp, e0, n, lane);

        if (!fuse) {
            // final selection: plain map
#pragma unroll
            for (int v = 0; v < WVEC; ++v) {
                const uint32_t e = e0 + v * (32 * VEC) + lane * VEC;
                if (e >= n) continue;
                float th0[VEC], tau[VEC], o[VEC];
                raw_to_f32<__nv_bfloat16>(rt.b[v], th0);
                if (CK) rt.tau(v, tau); else raw_to_f32<__nv_bfloat16>(rt.x[v], tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j) o[j] = kept_all ? out_of(th0[j], tau[j], a_fix) : th0[j];
                store8(op, e, n, o, true);
            }
            ++it;
            continue;
        }

        // pass 1: every entry -- counts, band offsets, speculative outputs
        // (a ragged last tile reads zeros past the end: key 0 is never above
        // hi, and a band holding 0 is corrected below)
        uint32_t n_gt = 0, nb = 0, kmax = 0;
        float f_gg = 0.0f;
#pragma unroll
        for (int v = 0; v < WVEC; ++v) {
            const uint32_t e = e0 + v * (32 * VEC) + lane * VEC;
            *reinterpret_cast<uint4*>(sx + v * (32 * VEC) + lane * VEC) = rt.x[v][0];
            *reinterpret_cast<uint4*>(sbs + v * (32 * VEC) + lane * VEC) = rt.b[v][0];
            float th0[VEC], tau[VEC], o[VEC];
            raw_to_f32<__nv_bfloat16>(rt.b[v], th0);
            if (CK) rt.tau(v, tau); else raw_to_f32<__nv_bfloat16>(rt.x[v], tau);
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const uint32_t kk = key_of(tau[j]);
                const bool gt = kk > hi;
                kmax = max(kmax, kk);
                n_gt += gt;
                if (want_gamma && gt) f_gg = __fmaf_rn(tau[j], tau[j], f_gg);
                sol[nb * 32] = (uint16_t)(v * (32 * VEC) + lane * VEC + j);
                nb += (kk - lo <= span);
                o[j] = gt ? out_of(th0[j], tau[j], a_spec) : th0[j];
            }
            if (e < n) store8(op, e, n, o, true);
        }
        if (e0 + TILE > n && lo == 0) {
            // drop the zero-filled entries past the end from the band
            uint32_t keep = 0;
            for (uint32_t q = 0; q < nb; ++q) {
                const uint32_t off = sol[q * 32];
                if (e0 + off < n) sol[(keep++) * 32] = (uint16_t)off;
            }
            nb = keep;
        }
        if (__any_sync(FULL, kmax >= KEY_INF) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
        if (want_gamma) d_gg += (double)f_gg;
        __syncwarp();

        // pass 2: the band entries go to the unit's candidate segment (keys)
        // and to its band records (position and raw values)
        uint32_t nb_tot;
        const uint32_t nb_off = warp_excl_scan(nb, &nb_tot);
        const uint32_t left_tiles = min(run_end, end) - it;
        if (nb_tot && !c_ovf && nb_tot > c_left)
            c_ovf = !reserve(&au->n_alloc, nb_tot, c_cap, left_tiles, c_pos, c_left);
        if (nb_tot && !b_ovf && nb_tot > b_left)
            b_ovf = !reserve(&au->b_alloc, nb_tot, b_cap, left_tiles, b_pos, b_left);
        const bool c_store = nb_tot && !c_ovf;
        const bool b_store = nb_tot && !b_ovf;
        if (c_store || b_store) {
            uint32_t wi = c_pos + nb_off, wb = b_pos + nb_off;
            for (uint32_t q = 0; q < nb; ++q) {
                const uint32_t off = sol[q * 32];
                const uint32_t xr = sx[off], br = sbs[off];
                if (b_store) bseg[wb++] = make_uint2(e0 + off, (br << 16) | xr);
                if (c_store) {
                    const float xv = __uint_as_float(xr << 16), bv = __uint_as_float(br << 16);
                    cseg[wi++] = key_of(CK ? __fsub_rn(xv, bv) : xv);
                }
            }
        }
        const uint32_t t_gt = __reduce_add_sync(FULL, n_gt);
        if (lane == 0) {
            P.tcand[g] = make_uint2(c_store ? c_pos : 0u, c_store ? nb_tot : 0u);
            P.tband[g] = make_uint2(b_store ? b_pos : 0u, b_store ? nb_tot : 0u);
        }
        const uint32_t in_tot = nb_tot;
        if (c_store) { c_pos += in_tot; c_left -= in_tot; }
        if (b_store) { b_pos += nb_tot; b_left -= nb_tot; }
        a_gt += t_gt; a_int += in_tot;
        __syncwarp();
        ++it;
    }
    flush();
}

// Rewrites the kept band entries of every fused tensor that needs no repair.
template <bool CK>
__global__ void __launch_bounds__(TPB) k_patch(Plan P) {
    const int lane = threadIdx.x & 31;
    const uint32_t W = gridDim.x * WPB;
    const uint32_t wid = blockIdx.x * WPB + (threadIdx.x >> 5);
    const uint32_t items = (uint32_t)P.n_tiles;
    const uint32_t per = (items + W - 1) / W;
    const uint32_t beg = wid * per;
    const uint32_t end = min(items, beg + per);
    uint32_t it = beg, run_end = beg;
    const Unit* U = nullptr;
    const uint2* bseg = nullptr;
    __nv_bfloat16* op = nullptr;
    bool active = false;
    float a = 0.0f;
    uint32_t tk = 0;
    unsigned long long thr = 0;
    while (it < end) {
        if (it >= run_end) {
            const int t = tensor_of_tile(P.tens, P.n_tensors, it);
            const TensorDesc& d = P.tens[t];
            run_end = (uint32_t)(d.tile_base + (d.numel + TILE - 1) / TILE);
            U = &P.units[d.unit];
            active = (d.flags & TF_TRIM) && U->state == ST_DONE && !P.repair[t];
            if (!active) { it = run_end; continue; }
            bseg = P.brec + U->brec_off;
            op = static_cast<__nv_bfloat16*>(d.out);
            a = (P.op == ISO_OP_ISO) ? (float)P.coef[t] : P.lambda;
            tk = U->t;
            const long long cut = U->cut;
            const uint32_t c32 = (cut >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (uint32_t)cut;
            thr = ((unsigned long long)tk << 32) | (uint32_t)~c32;
        }
        const uint2 r = P.tband[it];
        for (uint32_t q = lane; q < r.y; q += 32) {
            const uint2 rec = bseg[r.x + q];
            const float xv = __uint_as_float(rec.y << 16);
            const float bv = __uint_as_float(rec.y & 0xFFFF0000u);
            const float tau = CK ? __fsub_rn(xv, bv) : xv;
            const unsigned long long kp = ((unsigned long long)key_of(tau) << 32) | (uint32_t)~rec.x;
            if (kp > thr) op[rec.x] = __float2bfloat16_rn(out_of(bv, tau, a));
        }
        ++it;
    }
}

// The exact apply for the fused tensors flagged by k_solve (normally none).
template <bool CK>
__global__ void __launch_bounds__(TPB) k_repair(Plan P) {
    const int lane = threadIdx.x & 31;
    const uint32_t W = gridDim.x * WPB;
    const uint32_t wid = blockIdx.x * WPB + (threadIdx.x >> 5);
    const uint32_t items = (uint32_t)P.n_tiles;
    const uint32_t per = (items + W - 1) / W;
    const uint32_t beg = wid * per;
    const uint32_t end = min(items, beg + per);
    uint32_t it = beg, run_end = beg, n = 0, tile_base = 0;
    const void* xp = nullptr;
    const void* bp = nullptr;
    void* op = nullptr;
    float a = 0.0f;
    unsigned long long thr = 0;
    while (it < end) {
        if (it >= run_end) {
            const int t = tensor_of_tile(P.tens, P.n_tensors, it);
            const TensorDesc& d = P.tens[t];
            run_end = (uint32_t)(d.tile_base + (d.numel + TILE - 1) / TILE);
            if (!P.repair[t]) { it = run_end; continue; }
            const Unit& U = P.units[d.unit];
            n = (uint32_t)d.numel;
            tile_base = (uint32_t)d.tile_base;
            xp = P.xptr[t];
            bp = d.base;
            op = d.out;
            a = (P.op == ISO_OP_ISO) ? (float)P.coef[t] : P.lambda;
            const long long cut = U.cut;
            const uint32_t c32 = (cut >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (uint32_t)cut;
            thr = ((unsigned long long)U.t << 32) | (uint32_t)~c32;
        }
        const uint32_t e0 = (it - tile_base) * TILE;
        RawTile<__nv_bfloat16, __nv_bfloat16, true> rt;
        rt.load(xp, bp, e0, n, lane);
#pragma unroll
        for (int v = 0; v < WVEC; ++v) {
            const uint32_t e = e0 + v * (32 * VEC) + lane * VEC;
            if (e >= n) continue;
            float th0[VEC], tau[VEC], o[VEC];
            raw_to_f32<__nv_bfloat16>(rt.b[v], th0);
            if (CK) rt.tau(v, tau); else raw_to_f32<__nv_bfloat16>(rt.x[v], tau);
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const unsigned long long kp = ((unsigned long long)key_of(tau[j]) << 32) | (uint32_t)~(e + j);
                o[j] = (kp > thr) ? out_of(th0[j], tau[j], a) : th0[j];
            }
            store8(op, e, n, o, true);
        }
        ++it;
    }
}

template __global__ void k_repair<true>(Plan);
template __global__ void k_repair<false>(Plan);
template __global__ void k_count_apply<true>(Plan);
template __global__ void k_count_apply<false>(Plan);
template __global__ void k_patch<true>(Plan);
template __global__ void k_patch<false>(Plan);

}  // namespace iso
