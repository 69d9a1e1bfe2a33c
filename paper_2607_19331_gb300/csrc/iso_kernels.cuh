// iso_kernels.cuh -- kernel declarations (definitions and explicit
// instantiations live in iso_select.cu, iso_apply.cu, iso_merge.cu,
// iso_block.cu and iso_fused.cu).
#pragma once

#include "iso_internal.cuh"

namespace iso {



// the streaming passes over (expert, tile) items deal them round-robin over
// the warps (1) or give each warp one contiguous range (0).  Contiguous ranges
// measured faster for these passes on the 7B K = 8 merges (round-robin: every
// warp visits every unit, and the warps flush a unit's counters together);
// the fused K = 1 pass takes round-robin tiles (FUSED_INTERLEAVE)
#ifndef ISO_PASS_INTERLEAVE
#define ISO_PASS_INTERLEAVE 0
#endif
constexpr bool PASS_INTERLEAVE = ISO_PASS_INTERLEAVE != 0;

// select (TENSOR / GLOBAL scope)
constexpr int COUNT_BLOCKS_PER_SM = 2;      // k_count: resident blocks of TPB threads per SM
__global__ void k_init_units(Plan P, long long global_n);
template <typename XT, typename BT, bool CK> __global__ void k_sample(Plan P);
template <typename XT, typename BT, bool CK, bool EMIT> __global__ void k_count(Plan P);
__global__ void k_decide(Plan P);
template <typename XT, typename BT, bool CK> __global__ void k_radix_hist(Plan P);
__global__ void k_radix_pick(Plan P);
template <typename XT, typename BT, bool CK> __global__ void k_csample(Plan P);
template <typename XT, typename BT, bool CK> __global__ void k_tie(Plan P);
template <typename XT, typename BT, bool CK> __global__ void k_cut(Plan P);
__global__ void k_cut_part(Plan P);
__global__ void k_radix_flat(Plan P);

// select (BLOCK scope)
constexpr int BLOCK_TPB = 512;             // k_block_select: threads per unit (32 keys each on the fast path)
constexpr int BLOCK_CTAS_PER_SM = 2;       // two units in flight per SM
template <typename XT, typename BT, bool CK> __global__ void k_block_select(Plan P);

// fused K = 1 pass (bf16 base and update)
#ifndef ISO_FUSED_BLOCKS_PER_SM
#define ISO_FUSED_BLOCKS_PER_SM 2
#endif
#ifndef ISO_FUSED_STAGES
#define ISO_FUSED_STAGES 2
#endif
#ifndef ISO_FUSED_INTERLEAVE
#define ISO_FUSED_INTERLEAVE 1
#endif
constexpr int FUSED_BLOCKS_PER_SM = ISO_FUSED_BLOCKS_PER_SM;
constexpr bool FUSED_INTERLEAVE = ISO_FUSED_INTERLEAVE != 0;   // tiles dealt round-robin over the warps
constexpr int FUSED_STAGES = ISO_FUSED_STAGES;          // tile stages per warp in the copy ring
constexpr int FUSED_STAGE_BYTES = 2 * TILE * 2;         // one tile of the update and of theta_0 (bf16)
// dynamic shared memory: the warps' stage rings, then one 8-byte mbarrier per stage
constexpr int FUSED_SMEM = WPB * FUSED_STAGES * (FUSED_STAGE_BYTES + 8);
static_assert(FUSED_STAGES >= 2 && FUSED_STAGES <= 8, "stage ring");
template <bool CK> __global__ void k_count_apply(Plan P);
template <bool CK> __global__ void k_patch(Plan P);
__global__ void k_fix_plan(Plan P);
template <bool CK> __global__ void k_fix(Plan P);

// apply: K = 1 (iso_apply.cu); K >= 2 with a compile-time bound KC >= K on
// the expert count, and the Gram pass for any K (iso_merge.cu)
template <typename XT, typename BT, bool CK, int KC> __global__ void k_apply(Plan P);
// k_merge is compiled for TIES alone and for the other operators (ISO, whose
// 1-D tensors take the plain average, TA and RAM): TIES needs no coefficients
enum MergeOpFamily : int { OPF_TIES = 0, OPF_OTHER = 1 };
template <typename XT, typename BT, bool CK, int KC, int OPF> __global__ void k_merge(Plan P);
template <typename XT, typename BT, bool CK, int KC> __global__ void k_gramk(Plan P);
// k_merge: resident blocks of TPB threads per SM, two for every expert bound
// and family (eight experts read their step from the stage entry by entry)
constexpr int merge_blocks_per_sm(int KC, int OPF) { return 2; }
// k_merge's dynamic shared memory (its per-warp staging ring)
template <typename XT, typename BT, int KC, int OPF> int merge_smem_bytes();
template <typename XT, typename BT, int KC> int gram_smem_bytes();
constexpr int gram_blocks_per_sm(int KC) { return 2; }
template <typename XT, typename BT, bool CK, int KC, int OPF> __global__ void k_merge_c(Plan P);
template <typename XT, typename BT, bool CK, int KC> __global__ void k_gramk_c(Plan P);
// the compact kernels' dynamic shared memory (one stage per warp)
template <typename BT, int KC> int compact_smem_bytes();
__global__ void k_solve(Plan P, int gram_mode);
template <typename XT> __global__ void k_mask(Plan P, uint32_t* const* mptr);
__global__ void k_status(const Header* h, int32_t* out);
__global__ void k_units_off(iso_unit_stats* st, long long stride, long long base, int n_units, int K);

// upload of host-built tables through kernel parameters (no host staging
// buffer, capturable, ordered on the stream)
constexpr int UPLOAD_BYTES = 16384;
struct UploadChunk {
    unsigned long long dst;
    uint32_t nbytes;   // multiple of 16
    uint32_t pad;
    uint4 data[UPLOAD_BYTES / 16];
};
__global__ void k_upload(UploadChunk c);

// iso_delta: tensors passed by value in chunks
constexpr int DELTA_MAXT = 64;
struct DeltaArgs {
    int n;
    long long tile_base[DELTA_MAXT + 1];
    long long numel[DELTA_MAXT];
    const void* a[DELTA_MAXT];
    const void* b[DELTA_MAXT];
    float* out[DELTA_MAXT];
};
template <typename AT, typename BT> __global__ void k_delta(DeltaArgs A);

enum GramMode { GRAM_NONE = 0, GRAM_UNIT = 1, GRAM_ACCUM = 2 };

}  // namespace iso
