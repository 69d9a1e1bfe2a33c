// iso_range.cu -- the exact TopKMask of one selection unit whose entries are
// split over several GPUs (App. F, TIES trim under the global magnitude
// density): each GPU holds a contiguous range of the unit's positions, and
// the threshold is found by a radix descent over the magnitude keys whose
// per-digit histograms are summed over the GPUs (the host side of that
// exchange is paper_2607_19331_gb300/shard.py).  This file holds the two
// device pieces a GPU runs on its own range:
//
//   iso_range_hist  counts[b] = #{ e in [begin, end) : key_e >> pshift == prefix,
//                                  (key_e >> shift) & (nbins - 1) == b }
//                   (nbins = 1, pshift = shift = 0, prefix = t counts the keys equal to t)
//   iso_range_mask  bit e - begin set  <=>  key_e > t, or key_e == t and fewer than
//                   `take` keys equal to t lie in [begin, e)
//
// key_e = the binary32 bits of |tau_e| with the sign cleared; tau_e = x_e (a
// task vector) or x_e - base_e in binary32 (a checkpoint), as everywhere in
// the library.
#include "iso.h"
#include "iso_gemm.cuh"
#include "iso_internal.cuh"

#include <algorithm>

namespace iso {
namespace {

constexpr int RH_TPB = 256;
constexpr int RM_WARPS = 8;                 // warps per block of the mask kernels
constexpr int RM_TILE = 32 * 32;            // entries per warp tile: 32 words of 32 bits

template <typename XT, typename BT, bool CK>
__device__ __forceinline__ uint32_t range_key(const void* x, const void* base, long long e) {
    return key_of(TauSrc<XT, BT, CK>::load1(x, base, e));
}

// Per-block shared histogram over a grid-stride walk of the range, then one
// atomic add per bin and block.  Consecutive threads read consecutive
// entries.
template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(RH_TPB) k_range_hist(const void* x, const void* base, long long begin,
                                                       long long end, uint32_t prefix, int pshift, int shift,
                                                       int nbins, unsigned long long* counts) {
    extern __shared__ uint32_t sh[];
    for (int b = threadIdx.x; b < nbins; b += blockDim.x) sh[b] = 0;
    __syncthreads();
    const unsigned long long pre = prefix;
    for (long long e = begin + (long long)blockIdx.x * blockDim.x + threadIdx.x; e < end;
         e += (long long)gridDim.x * blockDim.x) {
        const unsigned long long k = range_key<XT, BT, CK>(x, base, e);
        if ((k >> pshift) == pre) atomicAdd(&sh[(k >> shift) & (unsigned long long)(nbins - 1)], 1u);
    }
    __syncthreads();
    for (int b = threadIdx.x; b < nbins; b += blockDim.x)
        if (sh[b]) atomicAdd(&counts[b], (unsigned long long)sh[b]);
}

// Keys equal to t per warp tile of RM_TILE positions (tile j covers
// positions begin + j RM_TILE ...).  Lane l reads position 32 w + l of word w,
// so a warp's loads are consecutive.
template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(RM_WARPS * 32) k_range_ties(const void* x, const void* base, long long begin,
                                                              long long end, uint32_t t, long long n_tiles,
                                                              long long* tile_ties) {
    const int lane = threadIdx.x & 31;
    for (long long j = (long long)blockIdx.x * RM_WARPS + (threadIdx.x >> 5); j < n_tiles;
         j += (long long)gridDim.x * RM_WARPS) {
        const long long p0 = begin + j * RM_TILE;
        int c = 0;
        for (int w = 0; w < 32; ++w) {
            const long long e = p0 + 32 * w + lane;
            const bool tie = e < end && range_key<XT, BT, CK>(x, base, e) == t;
            c += __popc(__ballot_sync(0xFFFFFFFFu, tie));
        }
        if (lane == 0) tile_ties[j] = c;
    }
}

// Exclusive prefix sum of the tile counts in place, one block of 1024
// threads (each takes a contiguous slice), so that tile_ties[j] becomes the
// keys equal to t before tile j.
__global__ void __launch_bounds__(1024) k_range_scan(long long* tile_ties, long long n_tiles) {
    __shared__ long long part[1024];
    const long long per = (n_tiles + blockDim.x - 1) / blockDim.x;
    const long long a = (long long)threadIdx.x * per, b = min(n_tiles, a + per);
    long long s = 0;
    for (long long j = a; j < b; ++j) s += tile_ties[j];
    part[threadIdx.x] = s;
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {
        const long long v = threadIdx.x >= (unsigned)o ? part[threadIdx.x - o] : 0;
        __syncthreads();
        part[threadIdx.x] += v;
        __syncthreads();
    }
    long long run = threadIdx.x ? part[threadIdx.x - 1] : 0;
    for (long long j = a; j < b; ++j) {
        const long long c = tile_ties[j];
        tile_ties[j] = run;
        run += c;
    }
}

// The mask words: word w of tile j is the ballot of its 32 positions; a key
// equal to t is kept while the keys equal to t before it (earlier tiles,
// earlier words of the tile, lower lanes of the word) are fewer than take.
template <typename XT, typename BT, bool CK>
__global__ void __launch_bounds__(RM_WARPS * 32) k_range_mask(const void* x, const void* base, long long begin,
                                                              long long end, uint32_t t, long long take,
                                                              long long n_tiles, const long long* tile_before,
                                                              uint32_t* mask) {
    const int lane = threadIdx.x & 31;
    const unsigned lt = (1u << lane) - 1u;
    const long long n_words = (end - begin + 31) / 32;
    for (long long j = (long long)blockIdx.x * RM_WARPS + (threadIdx.x >> 5); j < n_tiles;
         j += (long long)gridDim.x * RM_WARPS) {
        const long long p0 = begin + j * RM_TILE;
        long long before = tile_before[j];
        for (int w = 0; w < 32; ++w) {
            const long long e = p0 + 32 * w + lane;
            const uint32_t k = e < end ? range_key<XT, BT, CK>(x, base, e) : 0u;
            const bool tie = e < end && k == t;
            const unsigned tb = __ballot_sync(0xFFFFFFFFu, tie);
            const bool keep = e < end && (k > t || (tie && before + __popc(tb & lt) < take));
            const unsigned word = __ballot_sync(0xFFFFFFFFu, keep);
            const long long wi = j * 32 + w;
            if (lane == 0 && wi < n_words) mask[wi] = word;
            before += __popc(tb);
        }
    }
}

#define RG_LAUNCH(...) do { const int _slot = prof_begin(2, s); __VA_ARGS__; prof_end(_slot, s); \
                            if (cudaGetLastError() != cudaSuccess) return ISO_ERR_CUDA; } while (0)

template <bool B> struct BoolK { static constexpr bool value = B; };

template <typename F>
int dispatch_range(const iso_tensor& x, const iso_tensor* base, F&& f) {
    using Bf = __nv_bfloat16;
    const bool ck = base != nullptr;
    const int bdt = ck ? base->dtype : ISO_F32;
    if (x.dtype == ISO_BF16 && bdt == ISO_BF16) return ck ? f((Bf*)0, (Bf*)0, BoolK<true>()) : f((Bf*)0, (Bf*)0, BoolK<false>());
    if (x.dtype == ISO_BF16) return ck ? f((Bf*)0, (float*)0, BoolK<true>()) : f((Bf*)0, (float*)0, BoolK<false>());
    if (bdt == ISO_BF16) return ck ? f((float*)0, (Bf*)0, BoolK<true>()) : f((float*)0, (Bf*)0, BoolK<false>());
    return ck ? f((float*)0, (float*)0, BoolK<true>()) : f((float*)0, (float*)0, BoolK<false>());
}

bool ok_tensor(const iso_tensor& t) {
    if (t.rows < 0 || t.cols < 0 || t.rows >= (1LL << 32) || t.cols >= (1LL << 32)) return false;
    if (t.dtype != ISO_BF16 && t.dtype != ISO_F32) return false;
    const long long n = t.rows * t.cols;
    if (n >= (1LL << 40)) return false;
    if (n > 0 && (!t.data || (reinterpret_cast<uintptr_t>(t.data) & 15u))) return false;
    return true;
}

int check_range(const iso_tensor* x, const iso_tensor* base, int64_t begin, int64_t end) {
    if (!x) return ISO_ERR_ARG;
    if (!ok_tensor(*x) || (base && !ok_tensor(*base))) return ISO_ERR_ARG;
    if (base && (base->rows != x->rows || base->cols != x->cols)) return ISO_ERR_SHAPE;
    const long long n = x->rows * x->cols;
    if (begin < 0 || end < begin || end > n) return ISO_ERR_ARG;
    return ISO_OK;
}

int range_grid(long long n, int per_block) {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long want = (n + per_block - 1) / per_block;
    return (int)std::max(1LL, std::min(want, (long long)sms * 8));
}

}  // namespace
}  // namespace iso

using namespace iso;

extern "C" {

int32_t iso_range_hist(const iso_tensor* x, const iso_tensor* base, int64_t begin, int64_t end, uint32_t prefix,
                       int32_t pshift, int32_t shift, int32_t nbins, int64_t* counts, void* stream) {
    ISO_TRY(check_range(x, base, begin, end));
    if (!counts) return ISO_ERR_ARG;
    if (nbins < 1 || nbins > 4096 || (nbins & (nbins - 1))) return ISO_ERR_ARG;
    if (pshift < 0 || pshift > 32 || shift < 0 || shift > pshift) return ISO_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(counts, 0, sizeof(int64_t) * (size_t)nbins, s) != cudaSuccess) return ISO_ERR_CUDA;
    if (end == begin) return ISO_OK;
    const int grid = range_grid(end - begin, RH_TPB * 16);
    return dispatch_range(*x, base, [&](auto* xt, auto* bt, auto ck) -> int {
        using XT = std::remove_pointer_t<decltype(xt)>;
        using BT = std::remove_pointer_t<decltype(bt)>;
        constexpr bool CK = decltype(ck)::value;
        RG_LAUNCH((k_range_hist<XT, BT, CK><<<grid, RH_TPB, nbins * sizeof(uint32_t), s>>>(
            x->data, base ? base->data : nullptr, begin, end, prefix, pshift, shift, nbins,
            reinterpret_cast<unsigned long long*>(counts))));
        return ISO_OK;
    });
}

int32_t iso_range_mask_workspace_size(int64_t n, size_t* bytes) {
    if (!bytes || n < 0) return ISO_ERR_ARG;
    const long long tiles = (n + RM_TILE - 1) / RM_TILE;
    *bytes = (size_t)std::max(1LL, tiles) * sizeof(long long);
    return ISO_OK;
}

int32_t iso_range_mask(const iso_tensor* x, const iso_tensor* base, int64_t begin, int64_t end, uint32_t t,
                       int64_t take, uint32_t* mask_bits, void* workspace, size_t ws_bytes, void* stream) {
    ISO_TRY(check_range(x, base, begin, end));
    if (take < 0) return ISO_ERR_ARG;
    if (end == begin) return ISO_OK;
    if (!mask_bits || (reinterpret_cast<uintptr_t>(mask_bits) & 3u)) return ISO_ERR_ARG;
    size_t need = 0;
    iso_range_mask_workspace_size(end - begin, &need);
    if (!workspace || ws_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 7u)) return ISO_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const long long n_tiles = (end - begin + RM_TILE - 1) / RM_TILE;
    long long* tiles = static_cast<long long*>(workspace);
    const int grid = range_grid(n_tiles, RM_WARPS);
    return dispatch_range(*x, base, [&](auto* xt, auto* bt, auto ck) -> int {
        using XT = std::remove_pointer_t<decltype(xt)>;
        using BT = std::remove_pointer_t<decltype(bt)>;
        constexpr bool CK = decltype(ck)::value;
        const void* bp = base ? base->data : nullptr;
        RG_LAUNCH((k_range_ties<XT, BT, CK><<<grid, RM_WARPS * 32, 0, s>>>(x->data, bp, begin, end, t, n_tiles, tiles)));
        RG_LAUNCH((k_range_scan<<<1, 1024, 0, s>>>(tiles, n_tiles)));
        RG_LAUNCH((k_range_mask<XT, BT, CK><<<grid, RM_WARPS * 32, 0, s>>>(x->data, bp, begin, end, t, take, n_tiles,
                                                                          tiles, mask_bits)));
        return ISO_OK;
    });
}

}  // extern "C"
