// iso_gemm.cuh -- the dense contraction of the frame-space merge on the
// fifth-generation tensor cores: C = A B^T for row-major fp32 operands read as
// tf32, with tcgen05.mma accumulating in tensor memory.
//
// One CTA of 128 threads computes one 128 x 128 tile of C:
//   warp 0, lane 0  loads the operand tiles (TMA, 128 rows x 32 fp32 = 128 B
//                   per row, 128-byte swizzle) into a GEMM_STAGES-deep ring,
//                   one mbarrier per stage counting the copied bytes;
//   warp 1, lane 0  issues four tcgen05.mma (K = 8 each) per stage into a
//                   128-lane x 128-column fp32 accumulator in tensor memory and
//                   frees the stage with tcgen05.commit;
//   all four warps  read the accumulator back with tcgen05.ld (warp w owns
//                   lanes 32 w .. 32 w + 31, one output row per thread) and
//                   store it (the epilogue).
// Every wait on a barrier is bounded; a wait that gives up records
// ISO_ERR_TIMEOUT, and the kernel still waits (bounded) for its own copies and
// products before it frees its tensor memory and returns.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace iso {

constexpr int GEMM_BM = 128;               // rows of A (and of C) per CTA
constexpr int GEMM_BN = 128;               // rows of B (columns of C) per CTA
constexpr int GEMM_BK = 32;                // contraction elements (fp32) per stage: 128 bytes
constexpr int GEMM_STAGES = 6;
constexpr int GEMM_TILE_BYTES = GEMM_BM * GEMM_BK * 4;                 // 16 KB per operand tile
constexpr int GEMM_SMEM = 1024 + GEMM_STAGES * 2 * GEMM_TILE_BYTES + 256;
constexpr int GEMM_THREADS = 128;

enum GemmEpilogue : int32_t {
    GEMM_STORE_F32 = 0,   // C[row * ldc + col] = acc (the tile is inside C's padded extents)
    GEMM_ADD_BASE = 1,    // out[row * ldo + col] = W0[row * ldo + col] + acc for row < M, col < N
    GEMM_ADAMW = 2        // acc is the gradient of the binary64 variable X (row < M, col < N, row
                          // stride ldo): AdamW moments updated in place, the step X_bar - X stored
};

// AdamW on a binary64 variable in the product's epilogue (decoupled weight
// decay, bias-corrected moments kept in binary32, arithmetic in binary64)
struct AdamwArgs {
    const double* X;      // the variable (read)
    float* m;             // first moment (in place)
    float* v;             // second moment (in place)
    double* dX;           // out: X_bar - X = -lr wd X - lr / bc1 * m / (sqrt(v / bc2) + eps)
    double lr, beta1, beta2, eps, wd, bc1, bc2;
};

struct GemmArgs {
    int32_t M, N;         // output extents (GEMM_ADD_BASE stores only inside them)
    int32_t k_tiles;      // contraction length / GEMM_BK
    int32_t a_k0, b_k0;   // first contraction column read from A's and B's arrays
    int32_t mode;         // GemmEpilogue
    float* C;
    long long ldc;
    void* out;            // GEMM_ADD_BASE: output and base (same dtype, iso_dtype out_dtype)
    const void* w0;
    long long ldo;
    int32_t out_dtype;
    int32_t pad;
    const int32_t* skip;  // optional: the whole grid returns at once while *skip != 0
    int32_t* status;      // header status word for ISO_ERR_TIMEOUT
    AdamwArgs adam;       // GEMM_ADAMW
};

__global__ void k_gemm_tf32(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                            GemmArgs g);

// Host side: a 2-D tensor map over a row-major fp32 array of `rows` x `cols`
// (cols a multiple of 4, rows and the row stride as given) with a 32 x 128
// box and the 128-byte swizzle the kernel's shared-memory descriptors expect.
int gemm_tensor_map(CUtensorMap* map, const float* base, long long rows, long long cols, long long ld);

// Launch accounting and per-kind device timing shared with the rest of the
// library (iso_api.cu): kind 0 = the tensor-core products, 1 = the other
// frame-merge and optimizer kernels, 2 = the range selection kernels
// (iso_range.cu).  prof_begin returns a slot (or -1 when profiling is
// off); prof_end records the end event and counts the launch.
int prof_begin(int frame_kind, cudaStream_t s);
void prof_end(int slot, cudaStream_t s);

#define ISO_TRY(x) do { int _r = (x); if (_r != ISO_OK) return _r; } while (0)

}  // namespace iso
