// iso_api.cu -- host side of the C ABI declared in include/iso.h.
//
// Responsibilities: argument validation, the workspace layout, splitting a
// tensor list into groups that fit the caller's workspace, building the
// per-group tables (uploaded through kernel parameters), and the launch
// sequence.  No device memory is allocated here.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>
#include <type_traits>
#include <unordered_map>
#include <vector>

#include <cuda.h>

#include "iso_kernels.cuh"

namespace iso {
namespace {

constexpr int COUNT_GRID_PER_SM = COUNT_BLOCKS_PER_SM;
constexpr int FUSED_GRID_PER_SM = FUSED_BLOCKS_PER_SM;

// ---------------------------------------------------------------------------
// profiling and launch accounting
// ---------------------------------------------------------------------------
enum Kind {
    KD_UPLOAD, KD_INIT, KD_SAMPLE, KD_COUNT, KD_DECIDE, KD_RADIX_HIST, KD_RADIX_PICK, KD_TIE,
    KD_CUT, KD_BLOCK_SELECT, KD_GRAM, KD_SOLVE, KD_APPLY, KD_MASK, KD_DELTA, KD_STATUS, KD_MEMSET,
    KD_PATCH, KD_REPAIR, KD_FRAME_GEMM, KD_FRAME, KD_RANGE, KD_RADIX_FLAT, KD_CUT_PART, KD_COUNT_KINDS
};
const char* kKindNames[KD_COUNT_KINDS] = {
    "upload", "init_units", "sample", "count", "decide", "radix_hist", "radix_pick", "tie",
    "cut", "block_select", "gram", "solve", "apply", "mask", "delta", "status", "memset",
    "patch", "repair", "frame_gemm", "frame", "range", "radix_flat", "cut_part"};

std::atomic<uint64_t> g_launches{0};

struct Prof {
    bool on = false;
    static constexpr int CAP = 16384;
    std::vector<cudaEvent_t> ev;     // 2 per slot
    std::vector<int> kind;
    int used = 0;
} g_prof;
std::mutex g_prof_mu;

struct ProfScope {
    int slot = -1;
    cudaStream_t s;
    ProfScope(int kind, cudaStream_t st) : s(st) {
        if (!g_prof.on) return;
        std::lock_guard<std::mutex> lk(g_prof_mu);
        if (g_prof.used >= Prof::CAP) return;
        slot = g_prof.used;
        if ((int)g_prof.ev.size() < 2 * (slot + 1)) {
            cudaEvent_t a, b;
            if (cudaEventCreate(&a) != cudaSuccess) { slot = -1; return; }
            if (cudaEventCreate(&b) != cudaSuccess) { cudaEventDestroy(a); slot = -1; return; }
            g_prof.ev.push_back(a);
            g_prof.ev.push_back(b);
            g_prof.kind.push_back(kind);
        } else {
            g_prof.kind[slot] = kind;
        }
        g_prof.used++;
        cudaEventRecord(g_prof.ev[2 * slot], s);
    }
    ~ProfScope() {
        if (slot >= 0) cudaEventRecord(g_prof.ev[2 * slot + 1], s);
    }
};

// Launch a kernel; returns ISO_ERR_CUDA if the launch was rejected.
template <typename F>
int launch(int kind, cudaStream_t s, F&& f) {
    {
        ProfScope ps(kind, s);
        f();
    }
    if (kind != KD_MEMSET) g_launches.fetch_add(1, std::memory_order_relaxed);
    return (cudaGetLastError() == cudaSuccess) ? ISO_OK : ISO_ERR_CUDA;
}

#ifndef ISO_TRY
#define ISO_TRY(x) do { int _r = (x); if (_r != ISO_OK) return _r; } while (0)
#endif

// ---------------------------------------------------------------------------
// device properties (cached per device)
// ---------------------------------------------------------------------------
struct DevInfo { int sms = 0; bool smem_set = false; };
std::mutex g_dev_mu;
std::unordered_map<int, DevInfo> g_dev;

int dev_sms(int* sms) {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess) return ISO_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_dev_mu);
    DevInfo& di = g_dev[d];
    if (di.sms == 0) {
        if (cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, d) != cudaSuccess)
            return ISO_ERR_CUDA;
    }
    *sms = di.sms;
    return ISO_OK;
}

// Large dynamic shared memory must be opted into once per kernel and device.
template <typename K>
int smem_optin(K kernel, int bytes) {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess) return ISO_ERR_CUDA;
    static std::mutex mu;
    static std::unordered_map<long long, bool> done;
    const long long key = ((long long)d << 48) ^ (long long)(uintptr_t)(const void*)kernel;
    std::lock_guard<std::mutex> lk(mu);
    if (done.count(key)) return ISO_OK;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
        return ISO_ERR_CUDA;
    done[key] = true;
    return ISO_OK;
}

// A grid of exactly the blocks that are resident at once (one wave), for
// latency-bound kernels that split their work evenly over the warps.
template <typename K>
int resident_grid(K kernel, int tpb, int smem, int sms, int* grid) {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess) return ISO_ERR_CUDA;
    static std::mutex mu;
    static std::unordered_map<long long, int> per_sm;
    const long long key = ((long long)d << 48) ^ (long long)(uintptr_t)(const void*)kernel;
    std::lock_guard<std::mutex> lk(mu);
    auto it = per_sm.find(key);
    if (it == per_sm.end()) {
        int b = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, tpb, smem) != cudaSuccess) return ISO_ERR_CUDA;
        it = per_sm.emplace(key, b < 1 ? 1 : b).first;
    }
    *grid = sms * it->second;
    return ISO_OK;
}

// ---------------------------------------------------------------------------
// validation
// ---------------------------------------------------------------------------
bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// rows * cols; only called on descriptors that check_tensor accepted, whose
// extents are each below 2^32 and whose product is below 2^32
long long numel_of(const iso_tensor& t) { return t.rows * t.cols; }

int check_tensor(const iso_tensor& t) {
    if (t.rows < 0 || t.cols < 0) return ISO_ERR_SHAPE;
    if (t.dtype != ISO_BF16 && t.dtype != ISO_F32) return ISO_ERR_DTYPE;
    if (t.is_1d != 0 && t.is_1d != 1) return ISO_ERR_ARG;
    // each extent below 2^32 before the product is formed, so rows * cols
    // cannot overflow 64 bits
    if (t.rows >= (1LL << 32) || t.cols >= (1LL << 32)) return ISO_ERR_UNSUPPORTED;
    const long long n = numel_of(t);
    if (n >= (1LL << 32)) return ISO_ERR_UNSUPPORTED;
    if (n > 0 && t.data == nullptr) return ISO_ERR_ARG;
    if (n > 0 && !aligned16(t.data)) return ISO_ERR_ALIGN;
    return ISO_OK;
}

bool same_shape(const iso_tensor& a, const iso_tensor& b) { return a.rows == b.rows && a.cols == b.cols; }

int check_topk(const iso_topk_cfg& c) {
    if (!(c.density >= 0.0 && c.density <= 1.0)) return ISO_ERR_ARG;
    if (c.scope < ISO_SCOPE_TENSOR || c.scope > ISO_SCOPE_GLOBAL) return ISO_ERR_ARG;
    if (c.reserved != 0) return ISO_ERR_ARG;
    if (c.scope == ISO_SCOPE_BLOCK) {
        if (c.block_rows < 1 || c.block_rows > 256) return ISO_ERR_ARG;
        if (c.block_cols < 8 || c.block_cols > 256 || (c.block_cols % 8) != 0) return ISO_ERR_ARG;
        if ((long long)c.block_rows * c.block_cols > BLOCK_MAX_ENTRIES) return ISO_ERR_UNSUPPORTED;
    }
    return ISO_OK;
}

int check_merge_cfg(const iso_merge_cfg& c) {
    if (c.op < ISO_OP_TA || c.op > ISO_OP_RAM) return ISO_ERR_ARG;
    if (c.mask_1d != 0 && c.mask_1d != 1) return ISO_ERR_ARG;
    if (!std::isfinite(c.lambda)) return ISO_ERR_ARG;
    if (!std::isfinite(c.eps_act) || c.eps_act < 0.0f) return ISO_ERR_ARG;
    if (!std::isfinite(c.ridge) || c.ridge < 0.0) return ISO_ERR_ARG;
    if (!std::isfinite(c.c_min) || !std::isfinite(c.c_max) || c.c_min > c.c_max) return ISO_ERR_ARG;
    if (c.op != ISO_OP_TA && c.op != ISO_OP_RAM) return check_topk(c.topk);
    return ISO_OK;
}

// ---------------------------------------------------------------------------
// a call, described once
// ---------------------------------------------------------------------------
struct Call {
    const iso_tensor* base = nullptr;     // [n] theta_0 (nullptr for mask-only calls)
    const iso_tensor* x = nullptr;        // [K * n] experts / task vectors
    const iso_tensor* out = nullptr;      // [n] or nullptr
    uint32_t* const* masks = nullptr;     // mask-only calls
    int n = 0, K = 1;
    bool ckpt = false;
    int op = ISO_OP_TIES;
    bool mask_only = false;
    bool mask_1d = true;
    float lambda = 1.0f;
    float eps_act = 0.0f;                 // RAM threshold, +0 for a zero
    double ridge = 1e-12, c_min = 0.0, c_max = 1.5;
    iso_topk_cfg topk{};
    bool trims = true;                    // some tensor is trimmed
    std::vector<char> trim;               // per tensor
    int xdt = ISO_F32, bdt = ISO_F32;
    bool ccv = false;                     // compact candidates (set by run_call when they fit)
};

bool tensor_trimmed(const Call& c, int t) { return c.trim[t] != 0; }

long long tiles_of(long long n) { return (n + TILE - 1) / TILE; }

long long blocks_of(const iso_tensor& t, const iso_topk_cfg& c) {
    if (t.rows == 0 || t.cols == 0) return 0;
    return ((t.rows + c.block_rows - 1) / c.block_rows) * ((t.cols + c.block_cols - 1) / c.block_cols);
}

// candidate capacity of one unit of n entries at density rho
unsigned long long cand_cap_of(long long n, double rho, bool quantized) {
    if (n <= SAMPLE_MAX) return (unsigned long long)n;   // exact band: its ties
    double kk = std::floor(rho * (double)n + 0.5);
    kk = std::min(std::max(kk, 0.0), (double)n);
    const double q = kk / (double)n;
    const double S = SAMPLE_MAX;
    const double band = 2.0 * (SAMPLE_Z * std::sqrt(S * q * (1.0 - q)) + 2.0) / S;
    // interior keys of the band (twice its expected width), plus what the
    // warps' candidate chunks may leave unused at the end of their ranges
    const double waste = (double)CHUNK_MAX * (std::ceil((double)n / (TILE * 64.0)) + 2.0);
    // the band's keys: its rank width (twice the expected size) and room for
    // runs of exact ties at its edges, which bfloat16-derived task vectors have
    // (few significant bits) and binary32 ones essentially do not
    const double ties = quantized ? 0.08 : 0.004;
    const double cap = 8192.0 + std::ceil((2.0 * band + ties) * (double)n) + waste;
    return (unsigned long long)std::min(cap, (double)n);
}

// Value slots of one unit's compact candidates (keys >= lo, about the kept
// fraction plus the band): the band's rank width twice over, room for ties at
// its low edge, and the chunk ends the count pass's warps may leave unused
// (at most VCHUNK per warp that reaches the unit; per = the count pass's
// items per warp on the largest GPU this is sized for).  Never more than the
// tile-padded entries plus one tile per such warp.
constexpr long long CCV_WARPS = 160LL * COUNT_BLOCKS_PER_SM * WPB;
unsigned long long v_cap_of(long long n, double rho, bool quantized, long long per) {
    const long long tiles = (n + TILE - 1) / TILE;
    const long long warps = tiles / std::max(1LL, per) + 2;
    double q = std::floor(rho * (double)n + 0.5) / std::max(1.0, (double)n);
    q = std::min(std::max(q, 0.0), 1.0);
    const double S = SAMPLE_MAX;
    const double band = n <= SAMPLE_MAX ? 0.0 : 2.0 * (SAMPLE_Z * std::sqrt(S * q * (1.0 - q)) + 2.0) / S;
    const double ties = quantized ? 0.08 : 0.004;
    const double est = 8192.0 + std::ceil((q + 2.0 * band + ties) * (double)n) + (double)VCHUNK * (double)warps;
    const double most = (double)tiles * TILE + (double)TILE * (double)warps;
    return (unsigned long long)std::min(std::min(est, most), 4294967040.0);
}

std::atomic<int> g_ccv{0};
// K >= 2 TIES / ISO merges at per-tensor scope and moderate density: the
// count pass writes the candidates, the Gram and merge passes read them
bool ccv_eligible(const Call& c) {
    return g_ccv.load(std::memory_order_relaxed) && c.K >= 2 && !c.mask_only && c.trims &&
           (c.op == ISO_OP_TIES || c.op == ISO_OP_ISO) && c.topk.scope == ISO_SCOPE_TENSOR &&
           c.topk.density <= 0.3;
}

// band-record capacity of one unit for the fused K = 1 pass: the band's rank
// width (twice its expected size) plus room for exact ties at its edges
unsigned long long brec_cap_of(long long n, double rho) {
    if (n <= SAMPLE_MAX) return (unsigned long long)n;
    double kk = std::floor(rho * (double)n + 0.5);
    kk = std::min(std::max(kk, 0.0), (double)n);
    const double q = kk / (double)n;
    const double S = SAMPLE_MAX;
    const double band = 2.0 * (SAMPLE_Z * std::sqrt(S * q * (1.0 - q)) + 2.0) / S;
    const double waste = (double)CHUNK_MAX * (std::ceil((double)n / (TILE * 64.0)) + 2.0);
    const double cap = 8192.0 + std::ceil((2.0 * band + 0.08) * (double)n) + waste;
    return (unsigned long long)std::min(cap, (double)n);
}

std::atomic<int> g_two_pass{0};
// The K = 1 update takes the fused single pass (bf16 base and update,
// per-tensor units) unless iso_force_two_pass selected the two-pass form.
// Its corrections re-read theta_0 after the outputs are written, so an output
// that aliases theta_0 (an in-place update) takes the two-pass form.
bool fused_path(const Call& c) {
    if (g_two_pass.load(std::memory_order_relaxed) || c.K != 1 || c.mask_only || c.op == ISO_OP_TA ||
        c.topk.scope != ISO_SCOPE_TENSOR || c.xdt != ISO_BF16 || c.bdt != ISO_BF16 || !c.trims)
        return false;
    // (workspace sizing passes no outputs: it sizes for the fused pass)
    for (int t = 0; c.out && t < c.n; ++t) {
        const char* b = static_cast<const char*>(c.base[t].data);
        const char* o = static_cast<const char*>(c.out[t].data);
        const long long bytes = numel_of(c.base[t]) * 2;
        if (b && o && b < o + bytes && o < b + bytes) return false;
    }
    return true;
}

size_t al256(size_t v) { return (v + 255) & ~(size_t)255; }

struct Layout {
    size_t hdr, units, tcand, teq_lo, teq_hi, tcnt, hist, hmxc, hmx, gram, coef, zero_end;
    size_t tens, xptr, mptr, table_end;
    size_t tband, repair, csamp, cand, brec, vmask, tval, vals, total;
    unsigned long long brec_total = 0;
    long long n_tiles = 0;
    int n_units = 0;
    unsigned long long cand_total = 0;
    unsigned long long v_total = 0;       // compact-candidate value slots
    long long v_per = 1;                  // count-pass items per warp (compact-candidate sizing)
    long long global_n = 0;
};

// Layout of the workspace for tensors [t0, t1).
Layout layout_of(const Call& c, int t0, int t1) {
    Layout L;
    const int T = t1 - t0;
    const int K = c.K;
    const int scope = c.topk.scope;
    long long tiles = 0, units = 0, gn = 0;
    unsigned long long cand = 0;
    for (int t = t0; t < t1; ++t) {
        const iso_tensor& d = c.x[t];
        const long long n = numel_of(d);
        tiles += tiles_of(n);
        if (scope == ISO_SCOPE_BLOCK) units += blocks_of(d, c.topk);
        if (tensor_trimmed(c, t)) {
            gn += n;
            if (scope == ISO_SCOPE_TENSOR) cand += (unsigned long long)K * cand_cap_of(n, c.topk.density, c.xdt == ISO_BF16);
        }
    }
    if (scope == ISO_SCOPE_TENSOR) units = T;
    if (scope == ISO_SCOPE_GLOBAL) {
        units = 1;
        cand = (unsigned long long)K * cand_cap_of(gn, c.topk.density, c.xdt == ISO_BF16);
    }
    const bool select = c.trims;
    const bool fused = fused_path(c);
    if (fused)
        for (int t = t0; t < t1; ++t)
            if (tensor_trimmed(c, t)) L.brec_total += brec_cap_of(numel_of(c.x[t]), c.topk.density);
    L.n_tiles = tiles;
    L.n_units = (int)units;
    L.cand_total = select ? cand : 0;
    if (c.ccv) {
        L.v_per = ((long long)K * tiles + CCV_WARPS - 1) / CCV_WARPS;
        for (int t = t0; t < t1; ++t)
            if (tensor_trimmed(c, t))
                L.v_total += (unsigned long long)K * v_cap_of(numel_of(c.x[t]), c.topk.density, c.xdt == ISO_BF16, L.v_per);
    }
    L.global_n = gn;
    size_t o = 0;
    L.hdr = o;   o = al256(o + sizeof(Header));
    L.units = o; o = al256(o + (size_t)K * units * sizeof(Unit));
    const size_t trec = (select && scope != ISO_SCOPE_BLOCK) ? (size_t)K * tiles : 0;
    L.tcand = o;  o = al256(o + trec * 8);
    L.teq_lo = o; o = al256(o + trec * 4);
    L.teq_hi = o; o = al256(o + trec * 4);
    L.tcnt = o;   o = al256(o + trec * 4);
    L.hist = o;  o = al256(o + (select && scope != ISO_SCOPE_BLOCK ? (size_t)K * units * RADIX_BINS * 4 : 0));
    L.hmxc = o;  o = al256(o + (select && scope != ISO_SCOPE_BLOCK ? (size_t)K * units * RADIX_BINS * 4 : 0));
    L.hmx = o;   o = al256(o + (select && scope != ISO_SCOPE_BLOCK ? (size_t)K * units * RADIX_BINS * 4 : 0));
    L.gram = o;  o = al256(o + (size_t)T * K * K * 8);
    L.coef = o;  o = al256(o + (size_t)T * K * 8);
    L.zero_end = o;
    L.tens = o;  o = al256(o + (size_t)T * sizeof(TensorDesc));
    L.xptr = o;  o = al256(o + (size_t)K * T * sizeof(void*));
    L.mptr = o;  o = al256(o + (size_t)T * sizeof(void*));
    L.table_end = o;
    L.tband = o;  o = al256(o + (fused ? (size_t)tiles * 8 : 0));
    L.repair = o; o = al256(o + (fused ? (size_t)T * 4 : 0));
    L.csamp = o;  o = al256(o + (fused ? (size_t)K * units * COUNT_CHUNKS * 4 : 0));
    L.cand = o;   o = al256(o + (size_t)L.cand_total * 4);
    L.brec = o;   o = al256(o + (size_t)L.brec_total * 8);
    L.vmask = o;  o = al256(o + (c.ccv ? (size_t)K * tiles * 128 : 0));
    L.tval = o;   o = al256(o + (c.ccv ? (size_t)K * tiles * 4 : 0));
    L.vals = o;   o = al256(o + (size_t)L.v_total * 4);
    L.total = o;
    return L;
}

// Split [0, n) into groups whose layout fits `ws` bytes (or one group when
// the scope spans every tensor).
int plan_groups(const Call& c, size_t ws, std::vector<int>* bounds) {
    bounds->clear();
    bounds->push_back(0);
    if (c.n == 0) return ISO_OK;
    if (c.topk.scope == ISO_SCOPE_GLOBAL && c.trims) {
        if (layout_of(c, 0, c.n).total > ws) return ISO_ERR_WORKSPACE;
        bounds->push_back(c.n);
        return ISO_OK;
    }
    int t0 = 0;
    while (t0 < c.n) {
        if (layout_of(c, t0, t0 + 1).total > ws) return ISO_ERR_WORKSPACE;
        // grow the group while it fits (doubling, then bisection)
        int good = t0 + 1, step = 1;
        while (good < c.n) {
            const int cand = std::min(c.n, good + step);
            if (layout_of(c, t0, cand).total <= ws) { good = cand; step *= 2; }
            else if (step == 1) break;
            else step = 1;
        }
        bounds->push_back(good);
        t0 = good;
    }
    return ISO_OK;
}

// ---------------------------------------------------------------------------
// dtype dispatch: F is a generic lambda taking (XT*, BT*, bool_constant<CK>)
// ---------------------------------------------------------------------------
template <bool V> struct BoolC { static constexpr bool value = V; };

template <typename F>
int dispatch_src(int xdt, int bdt, bool ckpt, F&& f) {
    using B = __nv_bfloat16;
    if (xdt == ISO_BF16 && bdt == ISO_BF16) return ckpt ? f((B*)0, (B*)0, BoolC<true>()) : f((B*)0, (B*)0, BoolC<false>());
    if (xdt == ISO_BF16 && bdt == ISO_F32) return ckpt ? f((B*)0, (float*)0, BoolC<true>()) : f((B*)0, (float*)0, BoolC<false>());
    if (xdt == ISO_F32 && bdt == ISO_BF16) return ckpt ? f((float*)0, (B*)0, BoolC<true>()) : f((float*)0, (B*)0, BoolC<false>());
    return ckpt ? f((float*)0, (float*)0, BoolC<true>()) : f((float*)0, (float*)0, BoolC<false>());
}

int upload(cudaStream_t s, char* dst_dev, const std::vector<char>& blob) {
    size_t off = 0;
    while (off < blob.size()) {
        UploadChunk ch;
        const size_t nb = std::min((size_t)UPLOAD_BYTES, blob.size() - off);
        ch.dst = (unsigned long long)(uintptr_t)(dst_dev + off);
        ch.nbytes = (uint32_t)((nb + 15) & ~(size_t)15);
        ch.pad = 0;
        std::memset(ch.data, 0, sizeof(ch.data));
        std::memcpy(ch.data, blob.data() + off, nb);
        ISO_TRY(launch(KD_UPLOAD, s, [&] { k_upload<<<1, 256, 0, s>>>(ch); }));
        off += nb;
    }
    return ISO_OK;
}

// ---------------------------------------------------------------------------
// one group
// ---------------------------------------------------------------------------
int run_group(const Call& c, int t0, int t1, char* ws, cudaStream_t s, const iso_merge_stats* st,
              long long units_stride, int unit_base_global) {
    const Layout L = layout_of(c, t0, t1);
    const int T = t1 - t0;
    const int K = c.K;
    int sms = 0;
    ISO_TRY(dev_sms(&sms));

    // tables
    std::vector<char> blob(L.table_end - L.tens, 0);
    TensorDesc* tens = reinterpret_cast<TensorDesc*>(blob.data());
    const void** xptr = reinterpret_cast<const void**>(blob.data() + (L.xptr - L.tens));
    uint32_t** mptr = reinterpret_cast<uint32_t**>(blob.data() + (L.mptr - L.tens));
    long long tile = 0, uoff = 0;
    int unit = 0;
    unsigned long long cand = 0, brec = 0, vslots = 0;
    const bool fused = fused_path(c);
    for (int q = 0; q < T; ++q) {
        const int t = t0 + q;
        const iso_tensor& xt = c.x[t];
        TensorDesc& d = tens[q];
        d.base = c.base ? c.base[t].data : nullptr;
        d.out = c.out ? c.out[t].data : nullptr;
        d.numel = numel_of(xt);
        d.rows = xt.rows;
        d.cols = xt.cols;
        d.tile_base = tile;
        tile += tiles_of(d.numel);
        d.flags = (xt.is_1d ? TF_1D : 0) | (tensor_trimmed(c, t) ? TF_TRIM : 0);
        d.uoff = uoff;
        if (tensor_trimmed(c, t)) uoff += d.numel;
        if (c.topk.scope == ISO_SCOPE_BLOCK) {
            d.unit = unit;
            d.bpr = (int)((xt.cols + c.topk.block_cols - 1) / c.topk.block_cols);
            d.nblocks = (int)blocks_of(xt, c.topk);
            unit += d.nblocks;
        } else {
            d.unit = (c.topk.scope == ISO_SCOPE_GLOBAL) ? 0 : q;
            d.bpr = 0;
            d.nblocks = 0;
        }
        if (c.topk.scope == ISO_SCOPE_TENSOR) {
            const unsigned long long cap =
                tensor_trimmed(c, t) ? cand_cap_of(d.numel, c.topk.density, c.xdt == ISO_BF16) : 0;
            d.cand_off = cand;
            d.cand_cap = cap;
            cand += (unsigned long long)K * cap;
        } else {
            d.cand_off = 0;
            d.cand_cap = (c.topk.scope == ISO_SCOPE_GLOBAL)
                             ? cand_cap_of(L.global_n, c.topk.density, c.xdt == ISO_BF16) : 0;
        }
        d.brec_off = brec;
        d.brec_cap = (fused && tensor_trimmed(c, t)) ? brec_cap_of(d.numel, c.topk.density) : 0;
        brec += d.brec_cap;
        d.v_off = vslots;
        d.v_cap = (c.ccv && tensor_trimmed(c, t)) ? v_cap_of(d.numel, c.topk.density, c.xdt == ISO_BF16, L.v_per) : 0;
        vslots += (unsigned long long)K * d.v_cap;
        for (int i = 0; i < K; ++i) xptr[i * T + q] = c.x[(size_t)i * c.n + t].data;
        mptr[q] = c.masks ? c.masks[t] : nullptr;
    }

    Plan P;
    std::memset(&P, 0, sizeof(P));
    P.hdr = reinterpret_cast<Header*>(ws + L.hdr);
    P.tens = reinterpret_cast<TensorDesc*>(ws + L.tens);
    P.xptr = reinterpret_cast<const void**>(ws + L.xptr);
    P.units = reinterpret_cast<Unit*>(ws + L.units);
    P.tcand = reinterpret_cast<uint2*>(ws + L.tcand);
    P.teq_lo = reinterpret_cast<uint32_t*>(ws + L.teq_lo);
    P.teq_hi = reinterpret_cast<uint32_t*>(ws + L.teq_hi);
    P.tcnt = reinterpret_cast<uint32_t*>(ws + L.tcnt);
    P.hist = reinterpret_cast<uint32_t*>(ws + L.hist);
    P.hmxc = reinterpret_cast<uint32_t*>(ws + L.hmxc);
    P.hmx = reinterpret_cast<uint32_t*>(ws + L.hmx);
    P.cand = reinterpret_cast<uint32_t*>(ws + L.cand);
    P.brec = reinterpret_cast<uint2*>(ws + L.brec);
    P.tband = reinterpret_cast<uint2*>(ws + L.tband);
    P.repair = fused ? reinterpret_cast<int32_t*>(ws + L.repair) : nullptr;
    P.csamp = fused ? reinterpret_cast<uint32_t*>(ws + L.csamp) : nullptr;
    P.gram = reinterpret_cast<double*>(ws + L.gram);
    P.coef = reinterpret_cast<double*>(ws + L.coef);
    P.ccv = c.ccv ? 1 : 0;
    P.vmask = c.ccv ? reinterpret_cast<uint32_t*>(ws + L.vmask) : nullptr;
    P.tval = c.ccv ? reinterpret_cast<uint32_t*>(ws + L.tval) : nullptr;
    P.vals = c.ccv ? reinterpret_cast<float*>(ws + L.vals) : nullptr;
    P.n_tensors = T;
    P.K = K;
    P.n_units = L.n_units;
    P.scope = c.topk.scope;
    P.n_tiles = L.n_tiles;
    P.xdt = c.xdt;
    P.bdt = c.bdt;
    P.ckpt = c.ckpt ? 1 : 0;
    P.op = c.mask_only ? ISO_OP_TIES : c.op;
    P.fused = fused ? 1 : 0;
    // BLOCK scope, one expert, TIES: the block kernel writes the outputs itself
    const bool fuse_block = c.trims && !c.mask_only && K == 1 && c.topk.scope == ISO_SCOPE_BLOCK &&
                            c.op == ISO_OP_TIES;
    P.fuse_block = fuse_block ? 1 : 0;
    P.block_rows = c.topk.block_rows;
    P.block_cols = c.topk.block_cols;
    P.lambda = c.lambda;
    P.eps_act = c.eps_act;
    P.density = c.topk.density;
    P.ridge = c.ridge;
    P.c_min = c.c_min;
    P.c_max = c.c_max;
    P.st_units = st ? st->units : nullptr;
    P.st_units_stride = units_stride;
    P.st_unit_base = unit_base_global;
    P.st_tensor_base = t0;
    P.st_gram = st ? st->gram : nullptr;
    P.st_coef = st ? st->coef : nullptr;

    // zero the per-group state (the status word at offset 0 persists across groups)
    ISO_TRY(launch(KD_MEMSET, s, [&] { cudaMemsetAsync(ws + 4, 0, L.zero_end - 4, s); }));
    ISO_TRY(upload(s, ws + L.tens, blob));

    const int pgrid = sms * 4;
    const bool select = c.trims && (c.mask_only || c.op != ISO_OP_TA);
    if ((long long)K * L.n_tiles >= (1LL << 31)) return ISO_ERR_UNSUPPORTED;   // 32-bit item indices
    int gram_mode = GRAM_NONE;
    if (!c.mask_only && c.op == ISO_OP_ISO) {
        if (K == 1 && c.topk.scope == ISO_SCOPE_TENSOR) gram_mode = GRAM_UNIT;
        else gram_mode = GRAM_ACCUM;
    }
    const bool need_gram_pass = gram_mode == GRAM_ACCUM && !(K == 1 && c.topk.scope == ISO_SCOPE_BLOCK);
    const int KU = K * L.n_units;

    int rc = ISO_OK;
    if (!select && !c.mask_only && (c.op == ISO_OP_TIES || c.op == ISO_OP_ISO) && P.st_units && KU > 0)
        ISO_TRY(launch(KD_INIT, s, [&] {
            k_units_off<<<(KU + 255) / 256, 256, 0, s>>>(P.st_units, P.st_units_stride, P.st_unit_base, L.n_units, K);
        }));
    if (select && c.topk.scope != ISO_SCOPE_BLOCK) {
        ISO_TRY(launch(KD_INIT, s, [&] { k_init_units<<<(KU + 255) / 256, 256, 0, s>>>(P, L.global_n); }));
        rc = dispatch_src(c.xdt, c.bdt, c.ckpt, [&](auto* xt, auto* bt, auto ck) -> int {
            using XT = std::remove_pointer_t<decltype(xt)>;
            using BT = std::remove_pointer_t<decltype(bt)>;
            constexpr bool CK = decltype(ck)::value;
            const int smem = (SAMPLE_MAX + SAMPLE_SEL_R * 256) * 4;
            ISO_TRY(smem_optin(k_sample<XT, BT, CK>, smem));
            ISO_TRY(launch(KD_SAMPLE, s, [&] { k_sample<XT, BT, CK><<<KU, SAMPLE_TPB, smem, s>>>(P); }));
            if (fused)
                ISO_TRY(launch(KD_SAMPLE, s, [&] { k_csample<XT, BT, CK><<<KU * CS_SPLIT, CS_TPB, 0, s>>>(P); }));
            if (fused) {
                if (CK) {
                    ISO_TRY(smem_optin(k_count_apply<true>, FUSED_SMEM));
                    ISO_TRY(launch(KD_COUNT, s, [&] { k_count_apply<true><<<sms * FUSED_GRID_PER_SM, TPB, FUSED_SMEM, s>>>(P); }));
                } else {
                    ISO_TRY(smem_optin(k_count_apply<false>, FUSED_SMEM));
                    ISO_TRY(launch(KD_COUNT, s, [&] { k_count_apply<false><<<sms * FUSED_GRID_PER_SM, TPB, FUSED_SMEM, s>>>(P); }));
                }
            } else {
                if (c.ccv) {
                    ISO_TRY(smem_optin(k_count<XT, BT, CK, true>, COUNT_EMIT_SMEM));
                    ISO_TRY(launch(KD_COUNT, s, [&] {
                        k_count<XT, BT, CK, true><<<sms * COUNT_GRID_PER_SM, TPB, COUNT_EMIT_SMEM, s>>>(P);
                    }));
                }
                else
                    ISO_TRY(launch(KD_COUNT, s, [&] { k_count<XT, BT, CK, false><<<sms * COUNT_GRID_PER_SM, TPB, 0, s>>>(P); }));
            }
            ISO_TRY(launch(KD_DECIDE, s, [&] { k_decide<<<(KU + 255) / 256, 256, 0, s>>>(P); }));
            if (c.topk.scope == ISO_SCOPE_GLOBAL) ISO_TRY(smem_optin(k_radix_flat, RADIX_FLAT_SMEM));
            for (int level = 0; level < 3; ++level) {
                if (c.topk.scope == ISO_SCOPE_GLOBAL)
                    ISO_TRY(launch(KD_RADIX_FLAT, s, [&] { k_radix_flat<<<sms * 2, TPB, RADIX_FLAT_SMEM, s>>>(P); }));
                ISO_TRY(launch(KD_RADIX_HIST, s, [&] { k_radix_hist<XT, BT, CK><<<pgrid, TPB, 0, s>>>(P); }));
                ISO_TRY(launch(KD_RADIX_PICK, s, [&] { k_radix_pick<<<KU, TPB, 0, s>>>(P); }));
            }
            ISO_TRY(launch(KD_TIE, s, [&] { k_tie<XT, BT, CK><<<pgrid, TPB, 0, s>>>(P); }));
            if (c.topk.scope == ISO_SCOPE_GLOBAL)
                ISO_TRY(launch(KD_CUT_PART, s, [&] { k_cut_part<<<pgrid, TPB, 0, s>>>(P); }));
            ISO_TRY(launch(KD_CUT, s, [&] { k_cut<XT, BT, CK><<<KU, CUT_TPB, 0, s>>>(P); }));
            return ISO_OK;
        });
        ISO_TRY(rc);
    } else if (select) {
        rc = dispatch_src(c.xdt, c.bdt, c.ckpt, [&](auto* xt, auto* bt, auto ck) -> int {
            using XT = std::remove_pointer_t<decltype(xt)>;
            using BT = std::remove_pointer_t<decltype(bt)>;
            constexpr bool CK = decltype(ck)::value;
            const int smem = BLOCK_KEYS_WORDS * 4;
            ISO_TRY(smem_optin(k_block_select<XT, BT, CK>, smem));
            if (KU > 0)
                ISO_TRY(launch(KD_BLOCK_SELECT, s, [&] { k_block_select<XT, BT, CK><<<KU, BLOCK_TPB, smem, s>>>(P); }));
            return ISO_OK;
        });
        ISO_TRY(rc);
    }

    if (c.mask_only) {
        uint32_t* const* mdev = reinterpret_cast<uint32_t* const*>(ws + L.mptr);
        if (c.xdt == ISO_BF16)
            ISO_TRY(launch(KD_MASK, s, [&] { k_mask<__nv_bfloat16><<<pgrid, TPB, 0, s>>>(P, mdev); }));
        else
            ISO_TRY(launch(KD_MASK, s, [&] { k_mask<float><<<pgrid, TPB, 0, s>>>(P, mdev); }));
        return ISO_OK;
    }

    if (fused) {
        // exact coefficients and repair flags, then the kept band entries, then
        // the full exact apply of any flagged tensor
        ISO_TRY(launch(KD_SOLVE, s, [&] { k_solve<<<(T + 127) / 128, 128, 0, s>>>(P, gram_mode); }));
        ISO_TRY(launch(KD_REPAIR, s, [&] { k_fix_plan<<<1, 1024, 0, s>>>(P); }));
        int ggrid = 0, fgrid = 0;
        if (c.ckpt) {
            ISO_TRY(resident_grid(k_patch<true>, TPB, 0, sms, &ggrid));
            ISO_TRY(resident_grid(k_fix<true>, TPB, 0, sms, &fgrid));
            ISO_TRY(launch(KD_PATCH, s, [&] { k_patch<true><<<ggrid, TPB, 0, s>>>(P); }));
            ISO_TRY(launch(KD_REPAIR, s, [&] { k_fix<true><<<fgrid, TPB, 0, s>>>(P); }));
        } else {
            ISO_TRY(resident_grid(k_patch<false>, TPB, 0, sms, &ggrid));
            ISO_TRY(resident_grid(k_fix<false>, TPB, 0, sms, &fgrid));
            ISO_TRY(launch(KD_PATCH, s, [&] { k_patch<false><<<ggrid, TPB, 0, s>>>(P); }));
            ISO_TRY(launch(KD_REPAIR, s, [&] { k_fix<false><<<fgrid, TPB, 0, s>>>(P); }));
        }
        return ISO_OK;
    }

    rc = dispatch_src(c.xdt, c.bdt, c.ckpt, [&](auto* xt, auto* bt, auto ck) -> int {
        using XT = std::remove_pointer_t<decltype(xt)>;
        using BT = std::remove_pointer_t<decltype(bt)>;
        constexpr bool CK = decltype(ck)::value;

        if (gram_mode != GRAM_NONE) {
            if (need_gram_pass) {
                auto gram = [&](auto kc) {
                    constexpr int KC = decltype(kc)::value;
                    if constexpr (KC >= 2) {
                        if (c.ccv) {
                            const int cs = compact_smem_bytes<BT, KC>();
                            ISO_TRY(smem_optin(k_gramk_c<XT, BT, CK, KC>, cs));
                            return launch(KD_GRAM, s, [&] { k_gramk_c<XT, BT, CK, KC><<<sms * 2, TPB, cs, s>>>(P); });
                        }
                    }
                    const int ggrid = sms * gram_blocks_per_sm(KC);
                    const int smem = gram_smem_bytes<XT, BT, KC>();
                    ISO_TRY(smem_optin(k_gramk<XT, BT, CK, KC>, smem));
                    return launch(KD_GRAM, s, [&] { k_gramk<XT, BT, CK, KC><<<ggrid, TPB, smem, s>>>(P); });
                };
                if (K == 1) ISO_TRY(gram(std::integral_constant<int, 1>{}));
                else if (K == 2) ISO_TRY(gram(std::integral_constant<int, 2>{}));
                else if (K <= 4) ISO_TRY(gram(std::integral_constant<int, 4>{}));
                else ISO_TRY(gram(std::integral_constant<int, 8>{}));
            }
            ISO_TRY(launch(KD_SOLVE, s, [&] { k_solve<<<(T + 127) / 128, 128, 0, s>>>(P, gram_mode); }));
        }
        auto merge = [&](auto kc) {
            constexpr int KC = decltype(kc)::value;
            if (c.ccv) {
                const int cs = compact_smem_bytes<BT, KC>();
                if (c.op == ISO_OP_TIES) {
                    ISO_TRY(smem_optin(k_merge_c<XT, BT, CK, KC, OPF_TIES>, cs));
                    return launch(KD_APPLY, s, [&] { k_merge_c<XT, BT, CK, KC, OPF_TIES><<<sms * 2, TPB, cs, s>>>(P); });
                }
                ISO_TRY(smem_optin(k_merge_c<XT, BT, CK, KC, OPF_OTHER>, cs));
                return launch(KD_APPLY, s, [&] { k_merge_c<XT, BT, CK, KC, OPF_OTHER><<<sms * 2, TPB, cs, s>>>(P); });
            }
            if (c.op == ISO_OP_TIES) {
                const int smem = merge_smem_bytes<XT, BT, KC, OPF_TIES>();
                const int mgrid = sms * merge_blocks_per_sm(KC, OPF_TIES);
                ISO_TRY(smem_optin(k_merge<XT, BT, CK, KC, OPF_TIES>, smem));
                return launch(KD_APPLY, s, [&] { k_merge<XT, BT, CK, KC, OPF_TIES><<<mgrid, TPB, smem, s>>>(P); });
            }
            const int smem = merge_smem_bytes<XT, BT, KC, OPF_OTHER>();
            const int mgrid = sms * merge_blocks_per_sm(KC, OPF_OTHER);
            ISO_TRY(smem_optin(k_merge<XT, BT, CK, KC, OPF_OTHER>, smem));
            return launch(KD_APPLY, s, [&] { k_merge<XT, BT, CK, KC, OPF_OTHER><<<mgrid, TPB, smem, s>>>(P); });
        };
        if (K == 1 && fuse_block) return ISO_OK;
        // RAM with one expert: the merge pass (its activity test lives there)
        if (K == 1 && c.op == ISO_OP_RAM) ISO_TRY(merge(std::integral_constant<int, 2>{}));
        else if (K == 1) ISO_TRY(launch(KD_APPLY, s, [&] { k_apply<XT, BT, CK, 1><<<pgrid, TPB, 0, s>>>(P); }));
        else if (K == 2) ISO_TRY(merge(std::integral_constant<int, 2>{}));
        else if (K <= 4) ISO_TRY(merge(std::integral_constant<int, 4>{}));
        else ISO_TRY(merge(std::integral_constant<int, 8>{}));
        return ISO_OK;
    });
    return rc;
}

// ---------------------------------------------------------------------------
// shared driver for update / merge / mask
// ---------------------------------------------------------------------------
int units_per_expert(const iso_tensor* tens, int n, const iso_topk_cfg& c, long long* out) {
    long long u = 0;
    if (c.scope == ISO_SCOPE_TENSOR) u = n;
    else if (c.scope == ISO_SCOPE_GLOBAL) u = 1;
    else for (int t = 0; t < n; ++t) u += blocks_of(tens[t], c);
    *out = u;
    return ISO_OK;
}

int run_call(Call& c, void* workspace, size_t ws_bytes, const iso_merge_stats* st, cudaStream_t s) {
    if (c.n > 0) {
        if (!workspace) return ISO_ERR_WORKSPACE;
        if (((uintptr_t)workspace & 255u) != 0) return ISO_ERR_WORKSPACE;
    }
    std::vector<int> bounds;
    // compact candidates when every tensor group can hold them, else the
    // full passes
    c.ccv = ccv_eligible(c);
    if (c.ccv && plan_groups(c, ws_bytes, &bounds) != ISO_OK) c.ccv = false;
    ISO_TRY(plan_groups(c, ws_bytes, &bounds));
    char* ws = static_cast<char*>(workspace);
    if (c.n > 0) ISO_TRY(launch(KD_MEMSET, s, [&] { cudaMemsetAsync(ws, 0, 4, s); }));
    long long stride = 0;
    units_per_expert(c.x, c.n, c.topk, &stride);
    int unit_base = 0;
    for (size_t g = 0; g + 1 < bounds.size(); ++g) {
        const int t0 = bounds[g], t1 = bounds[g + 1];
        ISO_TRY(run_group(c, t0, t1, ws, s, st, stride, unit_base));
        if (c.topk.scope == ISO_SCOPE_BLOCK)
            for (int t = t0; t < t1; ++t) unit_base += (int)blocks_of(c.x[t], c.topk);
        else if (c.topk.scope == ISO_SCOPE_TENSOR)
            unit_base += t1 - t0;
    }
    if (st && st->status) {
        if (c.n > 0)
            ISO_TRY(launch(KD_STATUS, s, [&] { k_status<<<1, 32, 0, s>>>(reinterpret_cast<const Header*>(ws), st->status); }));
        else
            ISO_TRY(launch(KD_MEMSET, s, [&] { cudaMemsetAsync(st->status, 0, 4, s); }));
    }
    return ISO_OK;
}

// out[t] may coincide with theta_0[t] exactly (an in-place update) and must
// share no byte with any other tensor of the call: another base tensor, any
// expert or another output.  The passes read inputs after outputs have been
// written (the fused pass's corrections, the K >= 2 staging), so a partial or
// cross-tensor overlap would give wrong results without an error.
int check_out_overlap(const iso_tensor* theta_0, const iso_tensor* experts, int K,
                      const iso_tensor* out, int n) {
    struct Span { uintptr_t a, b; int kind, t; };   // kind 0: output, 1: base, 2: expert
    std::vector<Span> v;
    v.reserve((size_t)n * (K + 2));
    auto add = [&](const iso_tensor& d, int kind, int t) {
        const long long bytes = numel_of(d) * (d.dtype == ISO_BF16 ? 2 : 4);
        if (bytes > 0) v.push_back({(uintptr_t)d.data, (uintptr_t)d.data + (uintptr_t)bytes, kind, t});
    };
    for (int t = 0; t < n; ++t) {
        add(out[t], 0, t);
        add(theta_0[t], 1, t);
        for (int i = 0; i < K; ++i) add(experts[(size_t)i * n + t], 2, t);
    }
    std::sort(v.begin(), v.end(), [](const Span& x, const Span& y) { return x.a < y.a; });
    for (size_t p = 0; p < v.size(); ++p) {
        for (size_t q = p + 1; q < v.size() && v[q].a < v[p].b; ++q) {
            const Span& x = v[p];
            const Span& y = v[q];
            if (x.kind != 0 && y.kind != 0) continue;            // inputs may share memory
            const Span& o = x.kind == 0 ? x : y;
            const Span& w = x.kind == 0 ? y : x;
            if (w.kind == 1 && w.t == o.t && w.a == o.a && w.b == o.b) continue;   // in place
            return ISO_ERR_ARG;
        }
    }
    return ISO_OK;
}

void set_trim(Call& c, const iso_tensor* tens) {
    c.trim.assign(c.n, 0);
    c.trims = false;
    for (int t = 0; t < c.n; ++t) {
        bool tr;
        if (c.mask_only) tr = true;
        else if (c.op == ISO_OP_TA || c.op == ISO_OP_RAM) tr = false;
        else if (c.op == ISO_OP_TIES) tr = c.mask_1d || !tens[t].is_1d;
        else tr = !tens[t].is_1d;
        c.trim[t] = tr ? 1 : 0;
        c.trims |= tr && numel_of(tens[t]) > 0;
    }
}

int build_merge_call(Call& c, const iso_tensor* theta_0, const iso_tensor* experts, int K,
                     int experts_are_deltas, const iso_tensor* out, int n, const iso_merge_cfg* cfg) {
    if (n < 0 || K < 1) return ISO_ERR_ARG;
    if (K > ISO_MAX_EXPERTS) return ISO_ERR_UNSUPPORTED;
    if (!cfg) return ISO_ERR_ARG;
    if (n > 0 && (!theta_0 || !experts || !out)) return ISO_ERR_ARG;
    if (experts_are_deltas != 0 && experts_are_deltas != 1) return ISO_ERR_ARG;
    ISO_TRY(check_merge_cfg(*cfg));
    for (int t = 0; t < n; ++t) {
        ISO_TRY(check_tensor(theta_0[t]));
        ISO_TRY(check_tensor(out[t]));
        if (!same_shape(theta_0[t], out[t])) return ISO_ERR_SHAPE;
        if (out[t].dtype != theta_0[t].dtype) return ISO_ERR_DTYPE;
        if (theta_0[t].dtype != theta_0[0].dtype) return ISO_ERR_DTYPE;
        if (out[t].is_1d != theta_0[t].is_1d) return ISO_ERR_SHAPE;
        for (int i = 0; i < K; ++i) {
            const iso_tensor& x = experts[(size_t)i * n + t];
            ISO_TRY(check_tensor(x));
            if (!same_shape(x, theta_0[t])) return ISO_ERR_SHAPE;
            if (x.dtype != experts[0].dtype) return ISO_ERR_DTYPE;
        }
    }
    ISO_TRY(check_out_overlap(theta_0, experts, K, out, n));
    c.base = theta_0;
    c.x = experts;
    c.out = out;
    c.n = n;
    c.K = K;
    c.ckpt = experts_are_deltas == 0;
    c.op = cfg->op;
    c.mask_1d = cfg->mask_1d != 0;
    c.lambda = cfg->lambda;
    c.eps_act = (cfg->eps_act == 0.0f) ? 0.0f : cfg->eps_act;   // -0 -> +0: |tau| > 0 keeps zeros out
    c.ridge = cfg->ridge;
    c.c_min = cfg->c_min;
    c.c_max = cfg->c_max;
    c.topk = cfg->topk;
    if (c.op == ISO_OP_TA || c.op == ISO_OP_RAM) { c.topk.scope = ISO_SCOPE_TENSOR; c.topk.density = 1.0; }
    c.xdt = n > 0 ? experts[0].dtype : ISO_F32;
    c.bdt = n > 0 ? theta_0[0].dtype : ISO_F32;
    set_trim(c, theta_0);
    return ISO_OK;
}

}  // namespace

// Launch accounting and profiling for the kernels of other translation units
// (0: the tensor-core product, 1: the frame-space merge and optimizer, 2: the
// range selection of iso_range.cu).
int prof_begin(int frame_kind, cudaStream_t s) {
    if (!g_prof.on) return -1;
    const int kind = frame_kind == 0 ? KD_FRAME_GEMM : frame_kind == 1 ? KD_FRAME : KD_RANGE;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (g_prof.used >= Prof::CAP) return -1;
    const int slot = g_prof.used;
    if ((int)g_prof.ev.size() < 2 * (slot + 1)) {
        cudaEvent_t a, b;
        if (cudaEventCreate(&a) != cudaSuccess) return -1;
        if (cudaEventCreate(&b) != cudaSuccess) { cudaEventDestroy(a); return -1; }
        g_prof.ev.push_back(a);
        g_prof.ev.push_back(b);
        g_prof.kind.push_back(kind);
    } else {
        g_prof.kind[slot] = kind;
    }
    g_prof.used++;
    cudaEventRecord(g_prof.ev[2 * slot], s);
    return slot;
}
void prof_end(int slot, cudaStream_t s) {
    if (slot >= 0) cudaEventRecord(g_prof.ev[2 * slot + 1], s);
    g_launches.fetch_add(1, std::memory_order_relaxed);
}
}  // namespace iso

// ===========================================================================
// C ABI
// ===========================================================================
using namespace iso;

extern "C" {

int32_t iso_num_units(const iso_tensor* tensors, int32_t n_tensors, const iso_topk_cfg* topk,
                      int64_t* n_units) {
    if (!topk || !n_units || n_tensors < 0 || (n_tensors > 0 && !tensors)) return ISO_ERR_ARG;
    ISO_TRY(check_topk(*topk));
    for (int t = 0; t < n_tensors; ++t)
        if (tensors[t].rows < 0 || tensors[t].cols < 0) return ISO_ERR_SHAPE;
    long long u = 0;
    units_per_expert(tensors, n_tensors, *topk, &u);
    *n_units = u;
    return ISO_OK;
}

int32_t iso_workspace_size(const iso_tensor* tensors, int32_t n_tensors, int32_t K,
                           const iso_merge_cfg* cfg, size_t* bytes_min, size_t* bytes_full) {
    if (!cfg || n_tensors < 0 || (n_tensors > 0 && !tensors) || K < 1) return ISO_ERR_ARG;
    if (K > ISO_MAX_EXPERTS) return ISO_ERR_UNSUPPORTED;
    ISO_TRY(check_merge_cfg(*cfg));
    for (int t = 0; t < n_tensors; ++t) {
        if (tensors[t].rows < 0 || tensors[t].cols < 0) return ISO_ERR_SHAPE;
        if (numel_of(tensors[t]) >= (1LL << 32)) return ISO_ERR_UNSUPPORTED;
    }
    Call c;
    std::vector<iso_tensor> xs((size_t)K * n_tensors);
    for (int i = 0; i < K; ++i)
        for (int t = 0; t < n_tensors; ++t) xs[(size_t)i * n_tensors + t] = tensors[t];
    c.x = xs.data();
    c.n = n_tensors;
    c.K = K;
    c.op = cfg->op;
    c.mask_1d = cfg->mask_1d != 0;
    c.topk = cfg->topk;
    if (c.op == ISO_OP_TA || c.op == ISO_OP_RAM) { c.topk.scope = ISO_SCOPE_TENSOR; c.topk.density = 1.0; }
    // experts are taken to share the base's dtype: for other combinations the
    // size reported is an upper bound
    c.xdt = c.bdt = n_tensors ? tensors[0].dtype : ISO_F32;
    set_trim(c, tensors);
    // the smallest workspace runs the full passes; the full size holds the
    // compact candidates where the call takes them
    size_t mn = 256;
    c.ccv = ccv_eligible(c);
    size_t full = n_tensors ? layout_of(c, 0, n_tensors).total : 256;
    c.ccv = false;
    if (c.topk.scope == ISO_SCOPE_GLOBAL && c.trims) mn = full;
    else for (int t = 0; t < n_tensors; ++t) mn = std::max(mn, layout_of(c, t, t + 1).total);
    if (bytes_min) *bytes_min = mn;
    if (bytes_full) *bytes_full = std::max(full, mn);
    return ISO_OK;
}

int32_t iso_delta(const iso_tensor* theta_i, const iso_tensor* theta_0, const iso_tensor* tau,
                  int32_t n_tensors, void* stream) {
    if (n_tensors < 0) return ISO_ERR_ARG;
    if (n_tensors == 0) return ISO_OK;
    if (!theta_i || !theta_0 || !tau) return ISO_ERR_ARG;
    for (int t = 0; t < n_tensors; ++t) {
        ISO_TRY(check_tensor(theta_i[t]));
        ISO_TRY(check_tensor(theta_0[t]));
        ISO_TRY(check_tensor(tau[t]));
        if (!same_shape(theta_i[t], theta_0[t]) || !same_shape(tau[t], theta_0[t])) return ISO_ERR_SHAPE;
        if (tau[t].dtype != ISO_F32) return ISO_ERR_DTYPE;
        if (theta_i[t].dtype != theta_i[0].dtype || theta_0[t].dtype != theta_0[0].dtype) return ISO_ERR_DTYPE;
        if (numel_of(tau[t]) > 0 && (tau[t].data == theta_i[t].data || tau[t].data == theta_0[t].data))
            return ISO_ERR_ARG;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int sms = 0;
    ISO_TRY(dev_sms(&sms));
    for (int t0 = 0; t0 < n_tensors; t0 += DELTA_MAXT) {
        DeltaArgs A;
        std::memset(&A, 0, sizeof(A));
        A.n = std::min(DELTA_MAXT, n_tensors - t0);
        long long tile = 0;
        for (int q = 0; q < A.n; ++q) {
            const int t = t0 + q;
            A.tile_base[q] = tile;
            A.numel[q] = numel_of(theta_0[t]);
            tile += tiles_of(A.numel[q]);
            A.a[q] = theta_i[t].data;
            A.b[q] = theta_0[t].data;
            A.out[q] = static_cast<float*>(tau[t].data);
        }
        A.tile_base[A.n] = tile;
        if (tile == 0) continue;
        const int grid = (int)std::min<long long>(tile, (long long)sms * 4);
        const int adt = theta_i[0].dtype, bdt = theta_0[0].dtype;
        using B = __nv_bfloat16;
        if (adt == ISO_BF16 && bdt == ISO_BF16) ISO_TRY(launch(KD_DELTA, s, [&] { k_delta<B, B><<<grid, TPB, 0, s>>>(A); }));
        else if (adt == ISO_BF16) ISO_TRY(launch(KD_DELTA, s, [&] { k_delta<B, float><<<grid, TPB, 0, s>>>(A); }));
        else if (bdt == ISO_BF16) ISO_TRY(launch(KD_DELTA, s, [&] { k_delta<float, B><<<grid, TPB, 0, s>>>(A); }));
        else ISO_TRY(launch(KD_DELTA, s, [&] { k_delta<float, float><<<grid, TPB, 0, s>>>(A); }));
    }
    return ISO_OK;
}

int32_t iso_topk_mask(const iso_tensor* tau, int32_t n_tensors, const iso_topk_cfg* cfg,
                      uint32_t* const* mask_bits, const iso_merge_stats* stats,
                      void* workspace, size_t ws_bytes, void* stream) {
    if (n_tensors < 0 || !cfg || (n_tensors > 0 && !tau)) return ISO_ERR_ARG;
    ISO_TRY(check_topk(*cfg));
    for (int t = 0; t < n_tensors; ++t) {
        ISO_TRY(check_tensor(tau[t]));
        if (tau[t].dtype != tau[0].dtype) return ISO_ERR_DTYPE;
        if (mask_bits && mask_bits[t] && !aligned16(mask_bits[t])) return ISO_ERR_ALIGN;
    }
    Call c;
    c.x = tau;
    c.n = n_tensors;
    c.K = 1;
    c.ckpt = false;
    c.mask_only = true;
    c.masks = mask_bits;
    c.topk = *cfg;
    c.xdt = n_tensors ? tau[0].dtype : ISO_F32;
    c.bdt = c.xdt;
    set_trim(c, tau);
    std::vector<uint32_t*> mvec;
    if (!mask_bits) { mvec.assign(n_tensors, nullptr); c.masks = mvec.data(); }
    return run_call(c, workspace, ws_bytes, stats, static_cast<cudaStream_t>(stream));
}

int32_t iso_update(const iso_tensor* theta_0, const iso_tensor* update, int32_t update_is_delta,
                   const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg,
                   void* workspace, size_t ws_bytes, const iso_merge_stats* stats, void* stream) {
    Call c;
    ISO_TRY(build_merge_call(c, theta_0, update, 1, update_is_delta, out, n_tensors, cfg));
    return run_call(c, workspace, ws_bytes, stats, static_cast<cudaStream_t>(stream));
}

int32_t iso_merge(const iso_tensor* theta_0, const iso_tensor* experts, int32_t K,
                  int32_t experts_are_deltas, const iso_tensor* out, int32_t n_tensors,
                  const iso_merge_cfg* cfg, void* workspace, size_t ws_bytes,
                  const iso_merge_stats* stats, void* stream) {
    Call c;
    ISO_TRY(build_merge_call(c, theta_0, experts, K, experts_are_deltas, out, n_tensors, cfg));
    return run_call(c, workspace, ws_bytes, stats, static_cast<cudaStream_t>(stream));
}

const char* iso_error_string(int32_t status) {
    switch (status) {
        case ISO_OK: return "ISO_OK: success";
        case ISO_ERR_ARG: return "ISO_ERR_ARG: invalid argument";
        case ISO_ERR_SHAPE: return "ISO_ERR_SHAPE: tensor shapes disagree";
        case ISO_ERR_DTYPE: return "ISO_ERR_DTYPE: unsupported or mismatched dtype";
        case ISO_ERR_ALIGN: return "ISO_ERR_ALIGN: data pointer not 16-byte aligned";
        case ISO_ERR_WORKSPACE: return "ISO_ERR_WORKSPACE: workspace missing, misaligned or too small";
        case ISO_ERR_CUDA: return "ISO_ERR_CUDA: a CUDA launch or runtime call failed";
        case ISO_ERR_NONFINITE: return "ISO_ERR_NONFINITE: an input held NaN or Inf";
        case ISO_ERR_UNSUPPORTED: return "ISO_ERR_UNSUPPORTED: request outside this build's limits";
        case ISO_ERR_TIMEOUT: return "ISO_ERR_TIMEOUT: a kernel's wait for its own copies gave up";
        default: return "unknown iso_status";
    }
}

uint64_t iso_launch_count(void) { return g_launches.load(); }

int32_t iso_force_two_pass(int32_t on) {
    g_two_pass.store(on ? 1 : 0);
    return ISO_OK;
}

int32_t iso_compact_candidates(int32_t on) {
    g_ccv.store(on ? 1 : 0);
    return ISO_OK;
}

int32_t iso_profile_enable(int32_t on) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof.on = on != 0;
    return ISO_OK;
}

int32_t iso_profile_reset(void) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof.used = 0;
    return ISO_OK;
}

int32_t iso_profile_kinds(void) { return KD_COUNT_KINDS; }

const char* iso_profile_name(int32_t kind) {
    if (kind < 0 || kind >= KD_COUNT_KINDS) return "";
    return kKindNames[kind];
}

int32_t iso_profile_read(int32_t kind, int64_t* launches, double* total_ms) {
    if (kind < 0 || kind >= KD_COUNT_KINDS || !launches || !total_ms) return ISO_ERR_ARG;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    long long n = 0;
    double ms = 0.0;
    for (int q = 0; q < g_prof.used; ++q) {
        if (g_prof.kind[q] != kind) continue;
        if (cudaEventSynchronize(g_prof.ev[2 * q + 1]) != cudaSuccess) return ISO_ERR_CUDA;
        float f = 0.0f;
        if (cudaEventElapsedTime(&f, g_prof.ev[2 * q], g_prof.ev[2 * q + 1]) != cudaSuccess) return ISO_ERR_CUDA;
        ms += f;
        ++n;
    }
    *launches = n;
    *total_ms = ms;
    return ISO_OK;
}

}  // extern "C"

// ===========================================================================
// iso_update_noalloc: iso_update on the library's own fixed scratch
// ===========================================================================
// Some callers cannot hand the library a workspace: an inference-engine plugin
// whose enqueue path may not call cudaMalloc, a serving process that freezes
// its allocator after warm-up, or a C host without a device allocator of its
// own.  For them the library keeps one fixed scratch array per device in
// static device memory (ISO_NOALLOC_SCRATCH_BYTES, loaded with the module and
// held until the process exits) and runs the same update through it.
namespace iso {
namespace {

constexpr size_t NOALLOC_SCRATCH_BYTES = (size_t)ISO_NOALLOC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

// Device address of the scratch on the current device.  Looked up once per
// device (with that device current) and cached; the host-side name of the
// array is only a stand-in and is never passed to a kernel.
int noalloc_scratch(void** out) {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess) return ISO_ERR_CUDA;
    static std::mutex mu;
    static std::unordered_map<int, void*> ptrs;
    std::lock_guard<std::mutex> lk(mu);
    auto it = ptrs.find(d);
    if (it != ptrs.end()) { *out = it->second; return ISO_OK; }
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return ISO_ERR_CUDA;
    ptrs[d] = p;
    *out = p;
    return ISO_OK;
}

}  // namespace
}  // namespace iso

extern "C" int32_t iso_update_noalloc(const iso_tensor* theta_0, const iso_tensor* update,
                                      int32_t update_is_delta, const iso_tensor* out,
                                      int32_t n_tensors, const iso_merge_cfg* cfg,
                                      const iso_merge_stats* stats, void* stream) {
    Call c;
    ISO_TRY(build_merge_call(c, theta_0, update, 1, update_is_delta, out, n_tensors, cfg));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (n_tensors == 0) return run_call(c, nullptr, 0, stats, s);
    // reject requests the fixed scratch cannot hold before touching the device
    std::vector<int> bounds;
    ISO_TRY(plan_groups(c, NOALLOC_SCRATCH_BYTES, &bounds));
    void* ws = nullptr;
    ISO_TRY(noalloc_scratch(&ws));
    // run_call clears the scratch's status word and every per-group counter
    // region it uses before the group's kernels run
    return run_call(c, ws, NOALLOC_SCRATCH_BYTES, stats, s);
}

// ---------------------------------------------------------------------------
// the K = 1 update of a parameter set in host memory, pipelined
// ---------------------------------------------------------------------------
namespace iso {
namespace {

__global__ void k_status_first(const int32_t* st, int n, int32_t* out) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    int32_t v = ISO_OK;
    for (int g = 0; g < n && v == ISO_OK; ++g) v = st[g];
    *out = v;
}

size_t bytes_of(const iso_tensor& t) { return (size_t)numel_of(t) * (t.dtype == ISO_BF16 ? 2 : 4); }

// One group of consecutive tensors and where each of its three tensor lists
// sits inside a slot's region.  The region is sized for the tensors packed
// at 256-byte boundaries.  Tensors that follow one another in one host
// allocation form a run, moved by one copy, and keep their host spacing
// inside the region: for a list that is read (theta_0, update) the next
// tensor starts at the first 16-byte boundary after the previous one, for a
// list that is written back (out) right at its end, so no host byte outside
// an out tensor is ever written.  Either spacing takes no more room than the
// packed layout (a gap below 16 bytes never crosses a 256-byte boundary that
// the packed layout would not).
struct HostRun {
    const char* host;                 // first byte of the run in host memory
    size_t off, bytes;                // its offset inside the region, its length
    uintptr_t alloc_end;              // end of the host allocation holding it (0: unknown)
};
struct HostList {
    std::vector<size_t> off;          // per tensor, offset inside the region
    std::vector<HostRun> runs;
    size_t size = 0;                  // bytes of the region the list needs
};
struct HostGroup {
    int t0, t1;
    HostList l[3];                    // theta_0, update, out
    long long unit0;                  // first unit of the group
};

using PtrAttrFn = CUresult (*)(void*, CUpointer_attribute, CUdeviceptr);
PtrAttrFn ptr_attr_fn() {
    static std::once_flag once;
    static PtrAttrFn fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuPointerGetAttribute", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PtrAttrFn>(p);
    });
    return fn;
}

// End of the page-locked allocation that holds host address p, or 0 when the
// driver knows none (pageable memory): a copy may not cross from one
// allocation into the next, so runs stay inside one.
uintptr_t host_alloc_end(const void* p) {
    PtrAttrFn fn = ptr_attr_fn();
    if (!fn) return 0;
    CUdeviceptr start = 0;
    size_t size = 0;
    if (fn(&start, CU_POINTER_ATTRIBUTE_RANGE_START_ADDR, (CUdeviceptr)(uintptr_t)p) != CUDA_SUCCESS) return 0;
    if (fn(&size, CU_POINTER_ATTRIBUTE_RANGE_SIZE, (CUdeviceptr)(uintptr_t)p) != CUDA_SUCCESS) return 0;
    if ((uintptr_t)p < (uintptr_t)start || (uintptr_t)p >= (uintptr_t)start + size) return 0;
    return (uintptr_t)start + size;
}

size_t al16(size_t v) { return (v + 15) & ~(size_t)15; }

// with_runs = false sizes the region only (no CUDA call)
HostList place_list(const iso_tensor* h, int t0, int t1, bool written, bool with_runs) {
    HostList L;
    L.off.assign(t1 - t0, 0);
    size_t packed = 0;
    for (int t = t0; t < t1; ++t) packed += al256(bytes_of(h[t]));
    L.size = packed;
    if (!with_runs) return L;
    size_t o = 0;
    for (int t = t0; t < t1; ++t) {
        const size_t b = bytes_of(h[t]);
        if (b == 0) continue;
        const char* p = static_cast<const char*>(h[t].data);   // 16-byte aligned (check_tensor)
        if (!L.runs.empty()) {
            HostRun& r = L.runs.back();
            const uintptr_t end = (uintptr_t)r.host + r.bytes;
            const uintptr_t next = written ? end : al16(end);
            if ((uintptr_t)p == next && r.alloc_end != 0 && (uintptr_t)p + b <= r.alloc_end) {
                L.off[t - t0] = r.off + (size_t)(p - r.host);
                r.bytes = (size_t)(p - r.host) + b;
                o = al256(r.off + r.bytes);
                continue;
            }
        }
        L.runs.push_back({p, o, b, host_alloc_end(p)});
        L.off[t - t0] = o;
        o = al256(o + b);
    }
    return L;
}

struct HostPlan {
    std::vector<HostGroup> groups;
    size_t region[3] = {0, 0, 0};     // per slot
    size_t slot = 0, ws = 0, total = 0, st_off = 0, ws_off = 0;
};

int plan_host(const iso_tensor* th0, const iso_tensor* upd, const iso_tensor* out, int n,
              const iso_merge_cfg* cfg, size_t group_bytes, bool with_runs, HostPlan& hp) {
    const bool global = cfg->op != ISO_OP_TA && cfg->op != ISO_OP_RAM && cfg->topk.scope == ISO_SCOPE_GLOBAL;
    long long units = 0;
    int t = 0;
    while (t < n) {
        HostGroup g;
        g.t0 = t;
        size_t b = 0;
        // GLOBAL scope has one unit over every tensor: one group
        do { b += bytes_of(th0[t]) + bytes_of(upd[t]) + bytes_of(out[t]); ++t; }
        while (t < n && (global || b < group_bytes));
        g.t1 = t;
        g.l[0] = place_list(th0, g.t0, g.t1, false, with_runs);
        g.l[1] = place_list(upd, g.t0, g.t1, false, with_runs);
        g.l[2] = place_list(out, g.t0, g.t1, true, with_runs);
        size_t mn = 0, full = 0;
        ISO_TRY(iso_workspace_size(th0 + g.t0, g.t1 - g.t0, 1, cfg, &mn, &full));
        g.unit0 = units;
        long long u = 0;
        units_per_expert(th0 + g.t0, g.t1 - g.t0, cfg->topk, &u);
        if (global) u = 1;
        units += u;
        for (int q = 0; q < 3; ++q) hp.region[q] = std::max(hp.region[q], g.l[q].size);
        hp.ws = std::max(hp.ws, al256(full));
        hp.groups.push_back(std::move(g));
    }
    hp.slot = hp.region[0] + hp.region[1] + hp.region[2];
    hp.ws_off = (hp.groups.size() > 1 ? 2 : 1) * hp.slot;    // one group needs one slot
    hp.st_off = hp.ws_off + hp.ws;
    hp.total = hp.st_off + al256(sizeof(int32_t) * std::max<size_t>(1, hp.groups.size()));
    return ISO_OK;
}

// copies of one tensor list between host and a slot region, one per run
int copy_list(const HostList& L, char* dev, bool to_dev, cudaStream_t s) {
    for (const HostRun& r : L.runs) {
        const cudaError_t e = to_dev
            ? cudaMemcpyAsync(dev + r.off, r.host, r.bytes, cudaMemcpyHostToDevice, s)
            : cudaMemcpyAsync(const_cast<char*>(r.host), dev + r.off, r.bytes, cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) return ISO_ERR_CUDA;
    }
    return ISO_OK;
}

}  // namespace
}  // namespace iso

extern "C" {

int32_t iso_update_host_staging_size(const iso_tensor* theta_0, const iso_tensor* update, const iso_tensor* out,
                                     int32_t n_tensors, const iso_merge_cfg* cfg, size_t group_bytes,
                                     size_t* bytes) {
    if (!bytes || !cfg || n_tensors < 0 || (n_tensors > 0 && (!theta_0 || !update || !out))) return ISO_ERR_ARG;
    if (group_bytes == 0) return ISO_ERR_ARG;
    Call c;
    ISO_TRY(build_merge_call(c, theta_0, update, 1, 1, out, n_tensors, cfg));
    HostPlan hp;
    ISO_TRY(plan_host(theta_0, update, out, n_tensors, cfg, group_bytes, false, hp));
    *bytes = hp.total;
    return ISO_OK;
}

int32_t iso_update_host(const iso_tensor* theta_0, const iso_tensor* update, int32_t update_is_delta,
                        const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg, size_t group_bytes,
                        void* staging, size_t staging_bytes, const iso_merge_stats* stats, void* const* streams) {
    if (!cfg || !streams || n_tensors < 0 || group_bytes == 0) return ISO_ERR_ARG;
    Call c;
    ISO_TRY(build_merge_call(c, theta_0, update, 1, update_is_delta, out, n_tensors, cfg));
    if (n_tensors == 0) return ISO_OK;
    HostPlan hp;
    ISO_TRY(plan_host(theta_0, update, out, n_tensors, cfg, group_bytes, false, hp));
    if (!staging || ((uintptr_t)staging & 255u)) return ISO_ERR_WORKSPACE;
    if (staging_bytes < hp.total) return ISO_ERR_WORKSPACE;
    hp = HostPlan{};                  // the same plan, with the host runs placed
    ISO_TRY(plan_host(theta_0, update, out, n_tensors, cfg, group_bytes, true, hp));
    cudaStream_t h2d = static_cast<cudaStream_t>(streams[0]);
    cudaStream_t comp = static_cast<cudaStream_t>(streams[1]);
    cudaStream_t d2h = static_cast<cudaStream_t>(streams[2]);
    char* st = static_cast<char*>(staging);
    int32_t* gstat = reinterpret_cast<int32_t*>(st + hp.st_off);
    // per-slot events; destroyed when the call returns, released by the
    // runtime once the work recorded on them completes
    struct Events {
        cudaEvent_t e[3][2] = {};
        ~Events() {
            for (auto& r : e)
                for (cudaEvent_t x : r)
                    if (x) cudaEventDestroy(x);
        }
    } evs;
    auto& ev = evs.e;
    for (int a = 0; a < 3; ++a)
        for (int b = 0; b < 2; ++b)
            if (cudaEventCreateWithFlags(&ev[a][b], cudaEventDisableTiming) != cudaSuccess) return ISO_ERR_CUDA;
    enum { LOADED = 0, COMPUTED = 1, FREED = 2 };
    const int G = (int)hp.groups.size();
    std::vector<iso_tensor> d0, d1, d2;
    for (int gi = 0; gi < G; ++gi) {
        const HostGroup& g = hp.groups[gi];
        const int slot = gi & 1;
        char* base = st + (size_t)slot * hp.slot;
        char* reg[3] = {base, base + hp.region[0], base + hp.region[0] + hp.region[1]};
        // the slot's previous group has been copied out
        if (gi >= 2 && cudaStreamWaitEvent(h2d, ev[FREED][slot], 0) != cudaSuccess) return ISO_ERR_CUDA;
        for (int q = 0; q < 2; ++q)
            if (copy_list(g.l[q], reg[q], true, h2d) != ISO_OK) return ISO_ERR_CUDA;
        if (cudaEventRecord(ev[LOADED][slot], h2d) != cudaSuccess) return ISO_ERR_CUDA;
        if (cudaStreamWaitEvent(comp, ev[LOADED][slot], 0) != cudaSuccess) return ISO_ERR_CUDA;
        const int nt = g.t1 - g.t0;
        d0.assign(theta_0 + g.t0, theta_0 + g.t1);
        d1.assign(update + g.t0, update + g.t1);
        d2.assign(out + g.t0, out + g.t1);
        for (int t = 0; t < nt; ++t) {
            d0[t].data = bytes_of(d0[t]) ? reg[0] + g.l[0].off[t] : nullptr;
            d1[t].data = bytes_of(d1[t]) ? reg[1] + g.l[1].off[t] : nullptr;
            d2[t].data = bytes_of(d2[t]) ? reg[2] + g.l[2].off[t] : nullptr;
        }
        iso_merge_stats gs{};
        gs.status = gstat + gi;
        if (stats) {
            gs.units = stats->units ? stats->units + g.unit0 : nullptr;
            gs.gram = stats->gram ? stats->gram + g.t0 : nullptr;
            gs.coef = stats->coef ? stats->coef + g.t0 : nullptr;
        }
        const int rc = iso_update(d0.data(), d1.data(), update_is_delta, d2.data(), nt, cfg, st + hp.ws_off, hp.ws,
                                  &gs, comp);
        if (rc != ISO_OK) return rc;
        if (cudaEventRecord(ev[COMPUTED][slot], comp) != cudaSuccess) return ISO_ERR_CUDA;
        if (cudaStreamWaitEvent(d2h, ev[COMPUTED][slot], 0) != cudaSuccess) return ISO_ERR_CUDA;
        if (copy_list(g.l[2], reg[2], false, d2h) != ISO_OK) return ISO_ERR_CUDA;
        if (cudaEventRecord(ev[FREED][slot], d2h) != cudaSuccess) return ISO_ERR_CUDA;
    }
    // the call ends on the compute stream once every copy back has finished
    for (int b = 0; b < 2 && b < G; ++b)
        if (cudaStreamWaitEvent(comp, ev[FREED][(G - 1 - b) & 1], 0) != cudaSuccess) return ISO_ERR_CUDA;
    if (stats && stats->status)
        return launch(KD_STATUS, comp, [&] { k_status_first<<<1, 32, 0, comp>>>(gstat, G, stats->status); });
    return ISO_OK;
}

}  // extern "C"
