// iso_gemm.cu -- tcgen05 / TMEM / TMA GEMM for the frame-space merge (see
// iso_gemm.cuh for the structure).
#include "iso_gemm.cuh"
#include "iso_internal.cuh"

#include <mutex>

namespace iso {

namespace {

// Shared-memory matrix descriptor of one K-major operand tile in the
// 128-byte swizzle: rows of 128 bytes, 8-row (1024-byte) swizzle atoms
// stacked along M/N (stride 1024 bytes), one atom along K.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);          // start address
    d |= (uint64_t)1u << 16;                            // leading byte offset (unused here)
    d |= (uint64_t)((1024u >> 4) & 0x3FFFu) << 32;      // stride byte offset: one 8-row atom
    d |= (uint64_t)1u << 46;                            // descriptor version of sm_100
    d |= (uint64_t)2u << 61;                            // layout: 128-byte swizzle
    return d;
}

// Instruction descriptor of tcgen05.mma kind::tf32: fp32 accumulator, tf32
// A and B, both K-major, M = 128, N = 128.
constexpr uint32_t UMMA_IDESC = (1u << 4)               // D format: f32
                              | (2u << 7)               // A format: tf32
                              | (2u << 10)              // B format: tf32
                              | ((uint32_t)(GEMM_BN >> 3) << 17)
                              | ((uint32_t)(GEMM_BM >> 4) << 24);

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
                 " [%0], [%1, {%2, %3}], [%4];"
                 :: "r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar) : "memory");
}

__device__ __forceinline__ void umma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}"
                 :: "r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(UMMA_IDESC), "r"(accumulate) : "memory");
}

// arrive on `bar` once every tcgen05.mma this thread issued before has completed
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 :: "r"(bar) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's accumulator row
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 "
                 "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
                 "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
                   "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
                   "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
                   "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
                   "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

// bounded wait on one barrier phase; false once the limit is reached or
// another thread of the CTA gave up already
__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
    for (int spin = 0; spin < MBAR_SPIN_LIMIT; ++spin) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((spin & 1023) == 1023 && *abort_flag) return false;
    }
    *abort_flag = 1;
    return false;
}

}  // namespace

__global__ void __launch_bounds__(GEMM_THREADS, 1)
k_gemm_tf32(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, GemmArgs g) {
    if (g.skip && *reinterpret_cast<const volatile int32_t*>(g.skip)) return;
    extern __shared__ unsigned char gemm_smem_raw[];
    unsigned char* const smem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(gemm_smem_raw) + 1023) & ~(uintptr_t)1023);
    unsigned char* const sa = smem;                                        // [stage] A tiles
    unsigned char* const sb = smem + GEMM_STAGES * GEMM_TILE_BYTES;        // [stage] B tiles
    uint64_t* const bars = reinterpret_cast<uint64_t*>(smem + 2 * GEMM_STAGES * GEMM_TILE_BYTES);
    // bars[0, S): full (bytes landed), bars[S, 2S): empty (products done), bars[2S]: accumulator ready
    uint32_t* const tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * GEMM_STAGES + 1);
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * GEMM_BM, n0 = blockIdx.x * GEMM_BN;
    const uint32_t sa_s = smem_u32(sa), sb_s = smem_u32(sb), bar_s = smem_u32(bars);
    auto full_bar = [&](int s) { return bar_s + 8u * s; };
    auto empty_bar = [&](int s) { return bar_s + 8u * (GEMM_STAGES + s); };
    const uint32_t accum_bar = bar_s + 8u * (2 * GEMM_STAGES);

    if (threadIdx.x == 0) {
        for (int s = 0; s < GEMM_STAGES; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        mbar_init(accum_bar, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     :: "r"(smem_u32(tmem_slot)), "r"(GEMM_BN) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);
    const int KT = g.k_tiles;

    if (warp == 0 && lane == 0) {
        // producer: stage s is refilled once the products that read it are done
        int issued = 0;
        for (int kt = 0; kt < KT; ++kt) {
            const int s = kt % GEMM_STAGES;
            const uint32_t ph = (uint32_t)(kt / GEMM_STAGES) & 1u;
            if (!wait_phase(empty_bar(s), ph ^ 1u, abort_flag)) break;
            mbar_arrive_tx(full_bar(s), 2 * GEMM_TILE_BYTES);
            tma_load_2d(sa_s + s * GEMM_TILE_BYTES, &ta, g.a_k0 + kt * GEMM_BK, m0, full_bar(s));
            tma_load_2d(sb_s + s * GEMM_TILE_BYTES, &tb, g.b_k0 + kt * GEMM_BK, n0, full_bar(s));
            ++issued;
        }
        // every copy this thread issued has landed before the CTA may exit
        for (int kt = (issued > GEMM_STAGES ? issued - GEMM_STAGES : 0); kt < issued; ++kt) {
            const int s = kt % GEMM_STAGES;
            for (int spin = 0; spin < MBAR_SPIN_LIMIT; ++spin)
                if (mbar_try_wait(full_bar(s), (uint32_t)(kt / GEMM_STAGES) & 1u)) break;
        }
    } else if (warp == 1 && lane == 0) {
        // products: four K = 8 steps per 128-byte stage, the descriptor's start
        // address advanced by 32 bytes per step inside the swizzle atom
        for (int kt = 0; kt < KT; ++kt) {
            const int s = kt % GEMM_STAGES;
            const uint32_t ph = (uint32_t)(kt / GEMM_STAGES) & 1u;
            if (!wait_phase(full_bar(s), ph, abort_flag)) break;
            tc_fence_after();
            const uint32_t a0 = sa_s + s * GEMM_TILE_BYTES, b0 = sb_s + s * GEMM_TILE_BYTES;
#pragma unroll
            for (int kk = 0; kk < GEMM_BK / 8; ++kk)
                umma_tf32(tmem, sw128_desc(a0 + 32u * kk), sw128_desc(b0 + 32u * kk),
                          (kt > 0 || kk > 0) ? 1u : 0u);
            umma_commit(empty_bar(s));
        }
        // the accumulator barrier also tracks products issued before a give-up
        umma_commit(accum_bar);
    }
    __syncwarp();

    // epilogue: one accumulator row per thread, 32 columns per tensor-memory load
    const bool ok = wait_phase(accum_bar, 0u, abort_flag) && !*abort_flag;
    tc_fence_after();
    if (!ok) {
        if (threadIdx.x == 0 && g.status) atomicCAS(g.status, 0, (int32_t)ISO_ERR_TIMEOUT);
    } else {
        const int r = warp * 32 + lane;
        const long long row = (long long)m0 + r;
#pragma unroll 1
        for (int c = 0; c < GEMM_BN / 32; ++c) {
            float v[32];
            tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(c * 32), v);
            const int col0 = n0 + c * 32;
            if (g.mode == GEMM_STORE_F32) {
                float4* dst = reinterpret_cast<float4*>(g.C + row * g.ldc + col0);
#pragma unroll
                for (int j = 0; j < 8; ++j) dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
            } else if (g.mode == GEMM_ADAMW) {
                if (row < g.M) {
                    const AdamwArgs& a = g.adam;
#pragma unroll 4
                    for (int j = 0; j < 32; ++j) {
                        const int col = col0 + j;
                        if (col >= g.N) break;
                        const long long e = row * g.ldo + col;
                        const double gr = (double)v[j];
                        const double mm = a.beta1 * (double)a.m[e] + (1.0 - a.beta1) * gr;
                        const double vv = a.beta2 * (double)a.v[e] + (1.0 - a.beta2) * gr * gr;
                        a.m[e] = (float)mm;
                        a.v[e] = (float)vv;
                        a.dX[e] = -a.lr * a.wd * a.X[e] - (a.lr / a.bc1) * mm / (sqrt(vv / a.bc2) + a.eps);
                    }
                }
            } else if (row < g.M) {
                if (g.out_dtype == ISO_BF16) {
                    const unsigned short* w = static_cast<const unsigned short*>(g.w0) + row * g.ldo;
                    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(g.out) + row * g.ldo;
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col = col0 + j;
                        if (col < g.N) o[col] = __float2bfloat16_rn(__fadd_rn(__uint_as_float((uint32_t)w[col] << 16), v[j]));
                    }
                } else {
                    const float* w = static_cast<const float*>(g.w0) + row * g.ldo;
                    float* o = static_cast<float*>(g.out) + row * g.ldo;
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col = col0 + j;
                        if (col < g.N) o[col] = __fadd_rn(w[col], v[j]);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(tmem), "r"(GEMM_BN) : "memory");
    }
}

namespace {
using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiled encode_fn() {
    static std::once_flag once;
    static EncodeTiled fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    });
    return fn;
}
}  // namespace

int gemm_tensor_map(CUtensorMap* map, const float* base, long long rows, long long cols, long long ld) {
    EncodeTiled fn = encode_fn();
    if (!fn) return ISO_ERR_CUDA;
    if ((reinterpret_cast<uintptr_t>(base) & 15u) || (ld % 4) || (cols % GEMM_BK) || (rows % GEMM_BM))
        return ISO_ERR_ALIGN;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 4};
    const cuuint32_t box[2] = {(cuuint32_t)GEMM_BK, (cuuint32_t)GEMM_BM};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? ISO_OK : ISO_ERR_CUDA;
}

}  // namespace iso
