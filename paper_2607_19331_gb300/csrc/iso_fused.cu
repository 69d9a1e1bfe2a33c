// iso_fused.cu -- the K = 1 masked update in one pass over HBM.
//
// For one expert every operator reduces to
//     out = theta_0 + a * (kept ? tau : 0)                          (App. F; Sec. 4.2)
// with a per-tensor scale a: lambda for TIES, the retention coefficient c*
// for ISO (the K = 1 case of the retention system), 1 for ISO's 1-D average.
// The two-pass form reads the inputs twice: once to count (TopKMask needs the
// unit's k-th largest |tau| before any entry can be decided) and once to apply.
//
// Here a single pass counts and writes every output under a speculative
// selection taken from the sample (k_sample), and a small exact pass then
// corrects what the speculation can have got wrong:
//
//   run mode  (the sampled band is one key value t^, a run of exact ties, as
//             bf16-derived task vectors have): kept_spec = key > t^, or
//             key == t^ before the sampled cut position c^.  If the counts
//             confirm t = t^, only ties between c^ and the exact cut can be
//             wrong, and k_fix re-applies that position range exactly.
//   band mode (a band [lo, hi] of several key values): kept_spec = key > hi;
//             every band entry is recorded (position and raw values), and
//             k_patch writes the band entries that the exact cut keeps.
//
// The exact threshold and cut come from the same select chain as the two-pass
// form (k_decide, k_radix_*, k_tie, k_cut), fed by this pass's counters.  A
// unit whose speculation failed (threshold outside the band, overflowing
// records) or whose exact coefficient differs from the speculated one is
// re-applied in full by k_fix, so the result is exact in every case.
#include "iso_kernels.cuh"

namespace iso {

// One full tile of the fast form, read from the warp's stage in shared memory:
// out = theta_0 + (key > T ? a tau : -0) for every entry, counting the keys
// above hi and equal to t^ and, outside run mode, marking the band entries
// other than t^ (bit 8 v + j of tbm: entry v * 256 + 8 lane + j).
// RUN: the band is the single key t^ (no band entries besides its ties).
// A1: a == 1, so a tau == tau.
template <bool CK, bool RUN, bool A1>
__device__ __forceinline__ void fused_fast_tile(const unsigned char* sx, const unsigned char* sb,
                                                __nv_bfloat16* q, int lane, uint32_t T, uint32_t lo,
                                                uint32_t span, uint32_t hi, uint32_t th, float a,
                                                uint32_t& n_gt, uint32_t& n_eq, float& f_gg,
                                                uint32_t& tbm) {
#pragma unroll
    for (int v = 0; v < WVEC; ++v) {
        const uint32_t off = (uint32_t)(v * (32 * VEC) + lane * VEC);
        const uint4 xr = *reinterpret_cast<const uint4*>(sx + 2 * off);
        const uint4 br = *reinterpret_cast<const uint4*>(sb + 2 * off);
        const uint32_t xw[4] = {xr.x, xr.y, xr.z, xr.w};
        const uint32_t bw[4] = {br.x, br.y, br.z, br.w};
        uint32_t ow[4];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float b0 = __uint_as_float(bw[w] << 16), b1 = __uint_as_float(bw[w] & 0xFFFF0000u);
            float t0 = __uint_as_float(xw[w] << 16), t1 = __uint_as_float(xw[w] & 0xFFFF0000u);
            if (CK) sub_rn2(t0, t1, t0, t1, b0, b1);
            const uint32_t k0 = key_of(t0), k1 = key_of(t1);
            const bool kp0 = (int)k0 > (int)T, kp1 = (int)k1 > (int)T;
            const bool gt0 = k0 > hi, gt1 = k1 > hi;
            const bool eq0 = k0 == th, eq1 = k1 == th;
            n_gt += (uint32_t)gt0 + (uint32_t)gt1;
            n_eq += (uint32_t)eq0 + (uint32_t)eq1;
            if (gt0) f_gg = __fmaf_rn(t0, t0, f_gg);
            if (gt1) f_gg = __fmaf_rn(t1, t1, f_gg);
            if (!RUN) {
                if ((k0 - lo <= span) & !eq0) tbm |= 1u << (v * VEC + 2 * w);
                if ((k1 - lo <= span) & !eq1) tbm |= 1u << (v * VEC + 2 * w + 1);
            }
            float u0 = t0, u1 = t1;
            if (!A1) mul_rn2(u0, u1, a, a, t0, t1);
            float o0, o1;
            add_rn2(o0, o1, b0, b1, kp0 ? u0 : -0.0f, kp1 ? u1 : -0.0f);
            __nv_bfloat162 h = __floats2bfloat162_rn(o0, o1);
            ow[w] = *reinterpret_cast<uint32_t*>(&h);
        }
        __stcs(reinterpret_cast<uint4*>(q + off), make_uint4(ow[0], ow[1], ow[2], ow[3]));
    }
}

// The fused pass.  Each warp walks a contiguous range of tiles; a ring of
// FUSED_STAGES tile stages per warp in shared memory is filled by bulk copies
// (cp.async.bulk, completion counted on one mbarrier per stage) issued by the
// warp's lane 0 FUSED_STAGES - 1 tiles ahead of the tile being decided, so
// several tiles of both inputs are in flight per warp without registers.  A
// partial tile (a tensor's last) is not copied: its stage's barrier is
// arrived on without transactions and the tile is read from global memory.
template <bool CK>
__global__ void __launch_bounds__(TPB, FUSED_BLOCKS_PER_SM) k_count_apply(Plan P) {
    extern __shared__ __align__(128) unsigned char s_ring[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char* const ring = s_ring + (size_t)warp * FUSED_STAGES * FUSED_STAGE_BYTES;
    const uint32_t ring_s = smem_u32(ring);
    const uint32_t bar_s = smem_u32(s_ring + (size_t)WPB * FUSED_STAGES * FUSED_STAGE_BYTES) +
                           8u * (uint32_t)(warp * FUSED_STAGES);
    const uint32_t W = gridDim.x * WPB;
    const uint32_t wid = blockIdx.x * WPB + warp;
    const uint32_t items = (uint32_t)P.n_tiles;
    // the warp's tiles: g = beg, beg + step, ... below end -- interleaved over
    // the warps (all warps sweep one window of the tensors together) or one
    // contiguous range per warp
    uint32_t beg, end, step;
    if (FUSED_INTERLEAVE) {
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
    const float a_spec = k1_spec_coef(P);

    if (lane == 0) {
        for (int s = 0; s < FUSED_STAGES; ++s) mbar_init(bar_s + 8u * s, 1);
        mbar_fence_init();
    }
    __syncwarp();

    // the copy cursor: the tensor of the next tile whose copy is issued
    int ct = tensor_of_tile(P.tens, P.n_tensors, beg);
    uint32_t ct_end = (uint32_t)(P.tens[ct].tile_base + (P.tens[ct].numel + TILE - 1) / TILE);
    auto issue = [&](uint32_t g, int s) {
        while (g >= ct_end) {
            ++ct;
            ct_end = (uint32_t)(P.tens[ct].tile_base + (P.tens[ct].numel + TILE - 1) / TILE);
        }
        if (lane == 0) {
            const TensorDesc& d = P.tens[ct];
            const uint32_t e0 = (g - (uint32_t)d.tile_base) * TILE;
            const uint32_t bar = bar_s + 8u * s;
            if ((uint32_t)d.numel - e0 >= (uint32_t)TILE) {
                const uint32_t dst = ring_s + (uint32_t)s * FUSED_STAGE_BYTES;
                mbar_arrive_tx(bar, 2 * TILE * 2);
                bulk_g2s(dst, static_cast<const char*>(P.xptr[ct]) + (size_t)e0 * 2, TILE * 2, bar);
                bulk_g2s(dst + TILE * 2, static_cast<const char*>(d.base) + (size_t)e0 * 2, TILE * 2, bar);
            } else {
                mbar_arrive(bar);
            }
        }
    };

    // the current tensor and its unit
    int t = tensor_of_tile(P.tens, P.n_tensors, beg);
    uint32_t t_end = 0;                       // first tile after tensor t
    bool sel = false;                         // the tensor's unit is decided here
    bool keep_all = false;                    // otherwise: every entry kept (untrimmed) or none (k == 0)
    float a = 0.0f;                           // coefficient of the kept entries
    uint32_t lo = 0, hi = 0, th = 0, chat = 0;
    bool a_t_normal = false;                  // |a t^| is a normal binary32 number
    Unit* au = nullptr;
    uint32_t a_gt = 0, a_eq = 0, a_int = 0, a_abv = 0;
    float s_gg = 0.0f, e_gg = 0.0f, s_gb = 0.0f, e_gb = 0.0f;
    bool want_gamma = false;
    uint32_t* cseg = nullptr;
    uint2* bseg = nullptr;
    uint32_t c_pos = 0, c_left = 0, c_cap = 0, b_pos = 0, b_left = 0, b_cap = 0;
    bool c_ovf = false, b_ovf = false;

    auto flush = [&]() {
        if (!au) return;
        const double gg = warp_sum((double)s_gg + (double)e_gg), gb = warp_sum((double)s_gb + (double)e_gb);
        if (lane == 0) {
            if (a_gt) atomicAdd(&au->c_gt, (unsigned long long)a_gt);
            if (a_eq) atomicAdd(&au->c_eq, (unsigned long long)a_eq);
            if (a_int) atomicAdd(&au->n_int, (unsigned long long)a_int);
            if (a_abv) atomicAdd(&au->c_abv, (unsigned long long)a_abv);
            if (want_gamma) {
                if (gg != 0.0) atomicAdd(&au->gamma_acc, gg);
                if (gb != 0.0) atomicAdd(&au->gamma_band, gb);
            }
            if (c_ovf) au->overflow = 1;
            if (b_ovf) au->b_overflow = 1;
        }
        a_gt = a_eq = a_int = a_abv = 0;
        s_gg = e_gg = s_gb = e_gb = 0.0f;
    };

    auto enter_tensor = [&](int tt) {
        flush();
        au = nullptr;
        const TensorDesc& d = P.tens[tt];
        t_end = (uint32_t)(d.tile_base + (d.numel + TILE - 1) / TILE);
        const bool is1d = (d.flags & TF_1D) != 0;
        sel = false;
        if (!(d.flags & TF_TRIM)) {
            keep_all = true;
            a = (P.op == ISO_OP_ISO && is1d) ? 1.0f : P.lambda;
            return;
        }
        Unit* U = &P.units[d.unit];
        if (U->state != ST_BAND || !U->mode_t) {   // k == 0: nothing kept
            keep_all = false;
            a = 0.0f;
            return;
        }
        sel = true;
        au = U;
        a = a_spec;
        lo = U->lo;
        hi = U->hi;
        th = U->that;
        a_t_normal = fabsf(__fmul_rn(a, __uint_as_float(th))) >= 1.17549435e-38f;
        const long long ch = U->chat;
        chat = (uint32_t)(ch < 0 ? 0 : ch);
        want_gamma = U->want_gamma != 0;
        c_cap = (uint32_t)U->cand_cap;
        cseg = P.cand + U->cand_off;
        b_cap = (uint32_t)U->brec_cap;
        bseg = P.brec + U->brec_off;
        c_left = b_left = 0;
        c_ovf = b_ovf = false;
    };

    // reserve slots of a segment for one tile; false on overflow
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

    // the first tiles' copies
    for (int s = 0; s < FUSED_STAGES; ++s) {
        const unsigned long long gs = beg + (unsigned long long)s * step;
        if (gs < end) issue((uint32_t)gs, s);
    }

    enter_tensor(t);
    uint32_t phases = 0;                      // bit s: parity of stage s's next phase
    int s = 0;
    for (uint32_t g = beg; g < end; g += step) {
        {
            const uint32_t bar = bar_s + 8u * s;
            const uint32_t par = (phases >> s) & 1u;
            int spin = 0;
            while (!mbar_try_wait(bar, par)) {
                if (++spin >= MBAR_SPIN_LIMIT) {
                    // give up: report, then wait (bounded) for the copies this
                    // warp still has in flight before the block may exit
                    if (lane == 0) set_status(P.hdr, ISO_ERR_TIMEOUT);
                    const uint32_t pend = min((end - g + step - 1) / step, (uint32_t)FUSED_STAGES);
                    for (uint32_t j = 0; j < pend; ++j) {
                        const int sj = (s + (int)j) % FUSED_STAGES;
                        for (int r = 0; r < MBAR_SPIN_LIMIT; ++r)
                            if (mbar_try_wait(bar_s + 8u * sj, (phases >> sj) & 1u)) break;
                    }
                    return;
                }
            }
            phases ^= 1u << s;
        }
        if (g >= t_end) {
            while (g >= (uint32_t)(P.tens[t].tile_base + (P.tens[t].numel + TILE - 1) / TILE)) ++t;
            enter_tensor(t);
        }
        const TensorDesc& d = P.tens[t];
        __nv_bfloat16* const q16 = static_cast<__nv_bfloat16*>(d.out);
        const uint32_t n = (uint32_t)d.numel;
        const uint32_t e0 = (uint32_t)(g - d.tile_base) * TILE;
        const uint32_t rem = n - e0;
        const bool full = rem >= (uint32_t)TILE;
        const unsigned char* const sx = ring + (size_t)s * FUSED_STAGE_BYTES;
        const unsigned char* const sb = sx + TILE * 2;
        // a partial tile was not copied: it is read from global memory
        const unsigned short* const xs16 = full ? reinterpret_cast<const unsigned short*>(sx)
                                                : static_cast<const unsigned short*>(P.xptr[t]) + e0;
        const unsigned short* const bs16 = full ? reinterpret_cast<const unsigned short*>(sb)
                                                : static_cast<const unsigned short*>(d.base) + e0;

        // speculative selection: kept <=> key > t^, or key == t^ at a
        // position before chat.  In a whole tile on one side of chat that is
        // one comparison, key > T.  A tile of a tensor whose selection is
        // already final, a tile holding chat and a tensor's last tile (a few
        // per tensor) take a per-entry loop.  Band keys other than t^ are
        // rare: a per-lane bit marks them for the second step below.
        const uint32_t tile_hi = e0 + min(rem, (uint32_t)TILE);
        // the fast form writes theta_0 + (kept ? a tau : -0): exact (theta_0 bits
        // kept for an update of 0) because every kept |tau| is at least t^'s and
        // a times that stays a normal number
        const bool fast = sel && full && (tile_hi <= chat || e0 >= chat) && a_t_normal;
        uint32_t n_gt = 0, n_eq = 0;
        float f_gg = 0.0f;                     // tau^2 above hi (also the non-finite detector)
        uint32_t tbm = 0;                      // the lane's band entries of the tile
        bool slow_map = false;                 // tbm bit j: entry lane + 32 j (else v * 256 + 8 lane + j)
        if (fast) {
            const uint32_t T = (tile_hi <= chat) ? th - 1u : th;     // th >= 1 whenever ties are kept here
            const uint32_t span = hi - lo;     // band: key - lo <= span (unsigned), key != t^
            __nv_bfloat16* const qo = q16 + e0;
            const bool run = lo == hi, a1 = a == 1.0f;
            if (run) {
                if (a1) fused_fast_tile<CK, true, true>(sx, sb, qo, lane, T, lo, span, hi, th, a, n_gt, n_eq, f_gg, tbm);
                else    fused_fast_tile<CK, true, false>(sx, sb, qo, lane, T, lo, span, hi, th, a, n_gt, n_eq, f_gg, tbm);
            } else {
                if (a1) fused_fast_tile<CK, false, true>(sx, sb, qo, lane, T, lo, span, hi, th, a, n_gt, n_eq, f_gg, tbm);
                else    fused_fast_tile<CK, false, false>(sx, sb, qo, lane, T, lo, span, hi, th, a, n_gt, n_eq, f_gg, tbm);
            }
        } else if (!sel && full) {
            // a tensor whose selection is already final: every entry kept
            // (untrimmed) or none (k == 0)
#pragma unroll
            for (int v = 0; v < WVEC; ++v) {
                const uint32_t off = (uint32_t)(v * (32 * VEC) + lane * VEC);
                const uint4 xr = *reinterpret_cast<const uint4*>(sx + 2 * off);
                const uint4 br = *reinterpret_cast<const uint4*>(sb + 2 * off);
                float th0[VEC], tau[VEC], o[VEC];
                raw_to_f32<__nv_bfloat16>(reinterpret_cast<const uint4(&)[1]>(br), th0);
                raw_to_f32<__nv_bfloat16>(reinterpret_cast<const uint4(&)[1]>(xr), tau);
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                    const float tv = CK ? __fsub_rn(tau[j], th0[j]) : tau[j];
                    o[j] = keep_all ? out_of(th0[j], tv, a) : th0[j];
                }
                store8(q16, (long long)e0 + off, n, o, true);
            }
        } else {
            // entry by entry: lane L takes entries L + 32 j
            slow_map = true;
            const uint32_t cnt = min(rem, (uint32_t)TILE);
#pragma unroll 1
            for (uint32_t j = 0; j < 32; ++j) {
                const uint32_t o1 = (uint32_t)lane + 32u * j;
                if (o1 >= cnt) break;
                const uint32_t pos = e0 + o1;
                const uint32_t xr = xs16[o1], br = bs16[o1];
                const float bv = __uint_as_float(br << 16), xv = __uint_as_float(xr << 16);
                const float tv = CK ? __fsub_rn(xv, bv) : xv;
                float ov;
                if (!sel) {
                    ov = keep_all ? out_of(bv, tv, a) : bv;
                } else {
                    const uint32_t kk = key_of(tv);
                    const bool gt = kk > hi, eq = kk == th;
                    const bool kept = kk > th || (eq && pos < chat);
                    n_gt += gt;
                    n_eq += eq;
                    if (gt) f_gg = __fmaf_rn(tv, tv, f_gg);
                    if (kk >= lo && !gt && !eq) tbm |= 1u << j;
                    ov = kept ? out_of(bv, tv, a) : bv;
                }
                q16[pos] = __float2bfloat16_rn(ov);
            }
        }
        if (sel) {
            if (__any_sync(FULL, !(fabsf(f_gg) <= 3.402823466e38f))) {
                // a non-finite (or overflowing) sum: read the tile's keys again
                uint32_t kmax = 0;
                for (int v = 0; v < WVEC; ++v) {
                    const uint32_t o8 = (uint32_t)(v * (32 * VEC) + lane * VEC);
                    if (o8 >= rem) break;
                    float tau[VEC];
                    TauSrc<__nv_bfloat16, __nv_bfloat16, CK>::load8(P.xptr[t], d.base, (long long)e0 + o8, (long long)n, tau);
#pragma unroll
                    for (int j = 0; j < VEC; ++j)
                        if (o8 + j < rem) kmax = max(kmax, key_of(tau[j]));
                }
                if (__any_sync(FULL, kmax >= KEY_INF) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
            }
            if (want_gamma) two_sum_add(s_gg, e_gg, f_gg);
            const uint32_t t_gt = __reduce_add_sync(FULL, n_gt);
            const uint32_t t_eq = __reduce_add_sync(FULL, n_eq);
            a_gt += t_gt;
            a_eq += t_eq;

            // the marked band entries (keys other than t^, a fraction of a
            // per cent) go to the unit's candidate segment (keys) and its band
            // records (position and raw values), read again from the stage
            const uint32_t nb = __popc(tbm);
            uint32_t nb_tot;
            const uint32_t nb_off = warp_excl_scan(nb, &nb_tot);
            const uint32_t left_tiles = (min(t_end, end) - g + step - 1) / step;   // this warp's tiles left in the unit
            if (nb_tot && !c_ovf && nb_tot > c_left) c_ovf = !reserve(&au->n_alloc, nb_tot, c_cap, left_tiles, c_pos, c_left);
            if (nb_tot && !b_ovf && nb_tot > b_left) b_ovf = !reserve(&au->b_alloc, nb_tot, b_cap, left_tiles, b_pos, b_left);
            const bool c_store = nb_tot && !c_ovf;
            const bool b_store = nb_tot && !b_ovf;
            uint32_t n_abv = 0, kbad = 0;
            float f_band = 0.0f;               // tau^2 over the candidates above t^
            if (nb_tot) {
                uint32_t wi = c_pos + nb_off, wb = b_pos + nb_off;
                uint32_t m = tbm;
                while (m) {
                    const int b = __ffs(m) - 1;
                    m &= m - 1;
                    const uint32_t o1 = slow_map ? (uint32_t)lane + 32u * (uint32_t)b
                                                 : (uint32_t)((b >> 3) * (32 * VEC) + lane * VEC + (b & 7));
                    const uint32_t xr = xs16[o1], br = bs16[o1];
                    const float xv = __uint_as_float(xr << 16), bv = __uint_as_float(br << 16);
                    const float tv = CK ? __fsub_rn(xv, bv) : xv;
                    const uint32_t kk = key_of(tv);
                    if (b_store) bseg[wb++] = make_uint2(e0 + o1, (br << 16) | xr);
                    if (c_store) cseg[wi++] = kk;
                    const bool ab = kk > th;
                    n_abv += ab;
                    kbad |= (kk >= KEY_INF);
                    if (want_gamma && ab) f_band = __fmaf_rn(tv, tv, f_band);
                }
            }
            if (__any_sync(FULL, kbad) && lane == 0) set_status(P.hdr, ISO_ERR_NONFINITE);
            if (want_gamma) two_sum_add(s_gb, e_gb, f_band);
            const uint32_t t_abv = __reduce_add_sync(FULL, n_abv);
            if (lane == 0) {
                P.tcand[g] = make_uint2(c_store ? c_pos : 0u, c_store ? nb_tot : 0u);
                P.tband[g] = make_uint2(b_store ? b_pos : 0u, b_store ? nb_tot : 0u);
                P.teq_hi[g] = t_eq;             // teq_lo stays 0 (zeroed with the group's state)
            }
            if (c_store) { c_pos += nb_tot; c_left -= nb_tot; }
            if (b_store) { b_pos += nb_tot; b_left -= nb_tot; }
            a_int += nb_tot;
            a_abv += t_abv;
        }
        // the stage is free again: the copy of the tile FUSED_STAGES ahead
        __syncwarp();
        const unsigned long long gn = g + (unsigned long long)FUSED_STAGES * step;
        if (gn < end) {
            if (lane == 0) fence_proxy_async_smem();
            issue((uint32_t)gn, s);
        }
        s = (s + 1 == FUSED_STAGES) ? 0 : s + 1;
    }
    flush();
}

// The recorded band entries (keys other than t^): the fused pass kept those
// above t^; the exact selection decides each again, and an entry whose
// decision changed is rewritten.  Units re-applied by k_fix in full are
// skipped.
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
    const uint2* bseg = nullptr;
    __nv_bfloat16* op = nullptr;
    float a = 0.0f;
    uint32_t th = 0;
    unsigned long long thr = 0;
    while (it < end) {
        if (it >= run_end) {
            const int t = tensor_of_tile(P.tens, P.n_tensors, it);
            const TensorDesc& d = P.tens[t];
            run_end = (uint32_t)(d.tile_base + (d.numel + TILE - 1) / TILE);
            const Unit* U = &P.units[d.unit];
            const bool active = (d.flags & TF_TRIM) && U->state == ST_DONE && U->mode_t && !P.repair[t];
            if (!active) { it = run_end; continue; }
            bseg = P.brec + U->brec_off;
            op = static_cast<__nv_bfloat16*>(d.out);
            a = (P.op == ISO_OP_ISO) ? (float)P.coef[t] : P.lambda;
            th = U->that;
            const long long cut = U->cut;
            const uint32_t c32 = (cut >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (uint32_t)cut;
            thr = ((unsigned long long)U->t << 32) | (uint32_t)~c32;
        }
        // 32 tiles at a time, one per lane; a lane's records eight at a time,
        // their loads in flight together
        const uint32_t nt = min(32u, min(run_end, end) - it);
        const uint2 r = (lane < (int)nt) ? __ldg(&P.tband[it + lane]) : make_uint2(0u, 0u);
        for (uint32_t q0 = 0; q0 < r.y; q0 += 8) {
            uint2 rec[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                rec[u] = (q0 + u < r.y) ? __ldg(&bseg[r.x + q0 + u]) : make_uint2(0u, 0u);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (q0 + u >= r.y) break;
                const float xv = __uint_as_float(rec[u].y << 16);
                const float bv = __uint_as_float(rec[u].y & 0xFFFF0000u);
                const float tau = CK ? __fsub_rn(xv, bv) : xv;
                const uint32_t kk = key_of(tau);
                const bool kept = (((unsigned long long)kk << 32) | (uint32_t)~rec[u].x) > thr;
                if (kept != (kk > th)) op[rec[u].x] = __float2bfloat16_rn(kept ? out_of(bv, tau, a) : bv);
            }
        }
        it += nt;
    }
}

// The exact apply over a position range per tensor: the whole tensor for a
// unit flagged by k_solve (normally none); otherwise the keys equal to t^
// between the sampled cut chat and where the exact selection puts it (the
// exact cut when t == t^, the tensor's end when t < t^, its start when
// t > t^), the only entries the fused pass can have decided the wrong way
// besides the recorded band entries.
// The position range k_fix re-applies for each unit, and the prefix over
// units of its tile counts, so that k_fix can spread all ranges evenly over
// the GPU.  One block; the total goes to the header.
__global__ void __launch_bounds__(1024) k_fix_plan(Plan P) {
    __shared__ long long s_scan[33];
    long long base = 0;
    for (int t0 = 0; t0 < P.n_tensors; t0 += blockDim.x) {
        const int t = t0 + threadIdx.x;
        long long tiles = 0;
        if (t < P.n_tensors) {
            const TensorDesc& d = P.tens[t];
            Unit& U = P.units[d.unit];
            long long r0 = 0, r1 = 0;
            if ((d.flags & TF_TRIM) && U.state == ST_DONE && U.mode_t) {
                if (P.repair[t]) {
                    r0 = 0;
                    r1 = d.numel;
                } else {
                    const long long c = (U.t < U.that) ? d.numel
                                      : (U.t > U.that ? 0 : (U.cut > d.numel ? d.numel : U.cut));
                    r0 = min(c, U.chat);
                    r1 = max(c, U.chat);
                }
            }
            if (r1 > r0) tiles = (r1 + TILE - 1) / TILE - r0 / TILE;
            U.fix0 = r0;
            U.fix1 = r1;
        }
        long long tot;
        const long long off = block_excl_scan(tiles, s_scan, &tot);
        if (t < P.n_tensors) P.units[P.tens[t].unit].fix_off = base + off;
        base += tot;
        __syncthreads();
    }
    if (threadIdx.x == 0) P.hdr->fix_tiles = (int32_t)min(base, (long long)0x7FFFFFFF);
}

// Re-applies the exact selection on each unit's range (k_fix_plan): the whole
// tensor for a unit flagged by k_solve (normally none); otherwise the keys
// equal to t^ between the sampled cut chat and where the exact selection
// puts it (the exact cut when t == t^, the tensor's end when t < t^, its
// start when t > t^), the only entries the fused pass can have decided the
// wrong way besides the recorded band entries.  The ranges' tiles are split
// evenly over the warps.
// flattened fix tiles [off, off + nt) of tensor t start at tensor tile g_lo
struct FixRange {
    int t;
    long long off, nt, g_lo;
    __device__ __forceinline__ void load(const Plan& P, int tt) {
        t = tt;
        const Unit& U = P.units[P.tens[tt].unit];
        off = U.fix_off;
        g_lo = U.fix0 / TILE;
        nt = (U.fix1 > U.fix0) ? (U.fix1 + TILE - 1) / TILE - g_lo : 0;
    }
    // the range holding flattened tile f (>= off)
    __device__ __forceinline__ void seek(const Plan& P, long long f) {
        while (f >= off + nt) load(P, t + 1);
    }
    __device__ __forceinline__ uint32_t e0_of(long long f) const { return (uint32_t)(g_lo + (f - off)) * TILE; }
};

template <bool CK>
__global__ void __launch_bounds__(TPB) k_fix(Plan P) {
    const int lane = threadIdx.x & 31;
    const long long total = *(volatile int32_t*)&P.hdr->fix_tiles;
    const long long W = (long long)gridDim.x * WPB;
    const long long wid = (long long)blockIdx.x * WPB + (threadIdx.x >> 5);
    const long long per = (total + W - 1) / W;
    const long long fb = wid * per, fe = min(total, fb + per);
    if (fb >= fe) return;
    // the tensor holding flattened tile fb: last tensor with fix_off <= fb
    int t0 = 0;
    {
        int lo = 0, hi = P.n_tensors - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (P.units[P.tens[mid].unit].fix_off <= fb) lo = mid; else hi = mid - 1;
        }
        t0 = lo;
    }
    FixRange cur, nxt;          // the current tile's range, and the next tile's
    cur.load(P, t0);
    cur.seek(P, fb);
    nxt = cur;
    // the current range's parameters, reloaded when the range changes
    int pt = -1;
    long long r0 = 0, r1 = 0;
    bool all = false;
    uint32_t n = 0, th = 0;
    __nv_bfloat16* q = nullptr;
    float a = 0.0f;
    unsigned long long thr = 0;
    uint32_t e0 = cur.e0_of(fb);
    RawTile<__nv_bfloat16, __nv_bfloat16, true> rt;   // x in rt.x, theta_0 in rt.b
#pragma unroll
    for (int v = 0; v < WVEC; ++v)
        rt.load_step(v, P.xptr[cur.t], P.tens[cur.t].base, e0, (uint32_t)P.tens[cur.t].numel - e0, lane);
    for (long long f = fb; f < fe; ++f) {
        if (cur.t != pt) {
            pt = cur.t;
            const TensorDesc& d = P.tens[pt];
            const Unit& U = P.units[d.unit];
            r0 = U.fix0;
            r1 = U.fix1;
            all = P.repair[pt] != 0;
            n = (uint32_t)d.numel;
            th = U.that;
            q = static_cast<__nv_bfloat16*>(d.out);
            a = (P.op == ISO_OP_ISO) ? (float)P.coef[pt] : P.lambda;
            const long long cut = U.cut;
            const uint32_t c32 = (cut >= 0xFFFFFFFFLL) ? 0xFFFFFFFFu : (uint32_t)cut;
            thr = ((unsigned long long)U.t << 32) | (uint32_t)~c32;
        }
        // the next tile's loads replace each step as it is consumed
        const bool more = f + 1 < fe;
        uint32_t ne0 = 0, nrem = 0;
        const void* nxp = nullptr;
        const void* nbp = nullptr;
        if (more) {
            nxt.seek(P, f + 1);
            ne0 = nxt.e0_of(f + 1);
            nxp = P.xptr[nxt.t];
            nbp = P.tens[nxt.t].base;
            nrem = (uint32_t)P.tens[nxt.t].numel - ne0;
        }
#pragma unroll
        for (int v = 0; v < WVEC; ++v) {
            const uint32_t e = e0 + v * (32 * VEC) + lane * VEC;
            float th0[VEC], tau[VEC];
            raw_to_f32<__nv_bfloat16>(rt.b[v], th0);
            if (CK) rt.tau(v, tau); else raw_to_f32<__nv_bfloat16>(rt.x[v], tau);
            if (more) rt.load_step(v, nxp, nbp, ne0, nrem, lane);
            if (e >= n) continue;
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const long long pos = (long long)e + j;
                const uint32_t kk = key_of(tau[j]);
                if (pos >= n || pos < r0 || pos >= r1 || !(all || kk == th)) continue;
                const unsigned long long kp = ((unsigned long long)kk << 32) | (uint32_t)~(uint32_t)pos;
                q[pos] = __float2bfloat16_rn((kp > thr) ? out_of(th0[j], tau[j], a) : th0[j]);
            }
        }
        cur = nxt;
        e0 = ne0;
    }
}

template __global__ void k_fix<true>(Plan);
template __global__ void k_fix<false>(Plan);
template __global__ void k_count_apply<true>(Plan);
template __global__ void k_count_apply<false>(Plan);
template __global__ void k_patch<true>(Plan);
template __global__ void k_patch<false>(Plan);

}  // namespace iso
