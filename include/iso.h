/*
 * iso.h -- C ABI of the GB300 delta-merge library (libiso_gb300.so).
 *
 * The library implements the element-wise, data-parallel pass over parameter
 * updates from "ISO: An RLVR-Native Optimization Stack": for every weight
 * tensor it forms the task vector, trims it with an exact TopKMask, elects
 * signs where the operator has an election, and writes the merged or updated
 * weights
 *
 *     theta_merge = theta_0 + tau_merge                   (App. F, problem statement)
 *
 * for four operators:
 *   ISO_OP_TA    Task Arithmetic   tau = lambda * sum_i tau_i                (App. F)
 *   ISO_OP_TIES  TIES              trim, sign election, disjoint mean,
 *                                  theta_0 + lambda * tau_TIES              (App. F)
 *   ISO_OP_ISO   ISO retention     Gram of the trimmed task vectors,
 *                                  (Gamma + ridge I) c = diag Gamma, clip to
 *                                  [c_min, c_max], theta_0 + sum_i c_i trimmed tau_i;
 *                                  1-D tensors take the plain task-vector
 *                                  average                (Sec. 4.2, App. E, Algorithm 1)
 *   ISO_OP_RAM   RAM               per entry, the experts with |tau_i| > eps_act
 *                                  are active; no active expert: theta_0, one:
 *                                  its value kept whole, several: their mean;
 *                                  theta_0 + lambda * tau_RAM  (App. F, RAM)
 *
 * TopKMask(|tau|, rho) (App. F, TIES trim) keeps the k = floor(rho n + 1/2)
 * entries of largest |tau| in each selection unit; entries with equal |tau|
 * are taken lowest flat index first (in GLOBAL scope: tensor order, then flat
 * index).  |tau| is ranked by its binary32 value.
 *
 * Conventions for every entry point
 *   - All tensor data pointers, mask pointers, stats pointers and the workspace
 *     are DEVICE pointers owned by the caller.  The library never allocates,
 *     frees or retains device memory; it only reads the inputs, writes the
 *     outputs, and uses the caller's workspace as scratch for the duration of
 *     the call.
 *   - Tensors are row-major and contiguous; data pointers must be 16-byte
 *     aligned.  A 1-D tensor is passed as rows = 1, cols = n, is_1d = 1.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and the call returns without waiting.  Inputs must stay valid
 *     and unmodified, and the workspace untouched, until the stream reaches
 *     the end of the call's work.  Calls that share a workspace must be
 *     ordered on one stream.
 *   - The return value is ISO_OK or a negative iso_status.  Argument errors
 *     (ARG, SHAPE, DTYPE, ALIGN, WORKSPACE, UNSUPPORTED) are detected on the
 *     host before anything is enqueued.  ISO_ERR_CUDA means a launch failed.
 *     ISO_ERR_NONFINITE and ISO_ERR_TIMEOUT are detected on the device: they
 *     are written to stats->status (when given) and are valid once the stream
 *     has reached the end of the call; the outputs of such a call are
 *     unspecified.  The
 *     operators that read every task-vector entry's magnitude (TIES, ISO,
 *     RAM) check for it; TA does not.
 *   - No C++ exception crosses this interface.  The library keeps no state
 *     between calls apart from optional profiling counters.
 */
#ifndef ISO_H
#define ISO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ISO_ABI_VERSION 1

typedef enum {
    ISO_OK = 0,
    ISO_ERR_ARG = -1,          /* NULL where a pointer is required, count or enum out of range,
                                  density outside [0, 1], non-finite lambda / ridge / clip bounds */
    ISO_ERR_SHAPE = -2,        /* base, expert, out, mask shapes disagree; negative extents */
    ISO_ERR_DTYPE = -3,        /* dtype outside iso_dtype, out dtype differs from the base, or
                                  experts of mixed dtype */
    ISO_ERR_ALIGN = -4,        /* a data pointer is not 16-byte aligned */
    ISO_ERR_WORKSPACE = -5,    /* workspace NULL, not 256-byte aligned, or smaller than the
                                  minimum reported by iso_workspace_size */
    ISO_ERR_CUDA = -6,         /* a CUDA launch or runtime call failed */
    ISO_ERR_NONFINITE = -7,    /* (device) an input held NaN or +-Inf */
    ISO_ERR_UNSUPPORTED = -8,  /* valid request outside this build: K > ISO_MAX_EXPERTS,
                                  a tensor with 2^32 or more entries, GLOBAL scope larger
                                  than the workspace allows */
    ISO_ERR_TIMEOUT = -9       /* (device) a kernel's wait for its own bulk copies gave up
                                  after its iteration limit; the outputs are unspecified */
} iso_status;

#define ISO_MAX_EXPERTS 8

typedef enum { ISO_BF16 = 0, ISO_F32 = 1 } iso_dtype;

/* One tensor of a flat parameter list. */
typedef struct {
    void*   data;   /* device pointer, 16-byte aligned, rows * cols entries */
    int64_t rows;   /* >= 0; 1 for a 1-D tensor */
    int64_t cols;   /* >= 0 */
    int32_t dtype;  /* iso_dtype */
    int32_t is_1d;  /* 1 for normalisation scales, biases and other 1-D parameters */
} iso_tensor;

typedef enum {
    ISO_SCOPE_TENSOR = 0,  /* one selection unit per tensor */
    ISO_SCOPE_BLOCK = 1,   /* one unit per block_rows x block_cols tile of each tensor,
                              tiles in row-major tile order, partial edge tiles allowed */
    ISO_SCOPE_GLOBAL = 2   /* one unit over the whole task vector (tensor order, then
                              flat index): the paper's global magnitude density */
} iso_scope;

typedef struct {
    double  density;     /* rho in [0, 1]; k = floor(rho * n + 1/2) per unit */
    int32_t scope;       /* iso_scope */
    int32_t block_rows;  /* BLOCK scope: 1..256 (the paper-free default is 128) */
    int32_t block_cols;  /* BLOCK scope: 8..256, a multiple of 8 */
    int32_t reserved;    /* must be 0 */
} iso_topk_cfg;

typedef enum { ISO_OP_TA = 0, ISO_OP_TIES = 1, ISO_OP_ISO = 2, ISO_OP_RAM = 3 } iso_op;

typedef struct {
    int32_t op;          /* iso_op */
    int32_t mask_1d;     /* TIES: 1 = 1-D tensors are trimmed like the rest of the task
                            vector, 0 = used untrimmed.  Ignored by TA (never trims) and
                            ISO (1-D tensors take the average) */
    float   lambda;      /* TA / TIES / RAM scale (the paper uses 1.0; its RAM has no
                            scale, which is lambda = 1) */
    float   eps_act;     /* RAM active-update threshold, finite and >= 0: expert i is
                            active at an entry when the binary32 |tau_i| > eps_act
                            (strict; the paper uses 1e-5).  Ignored by the other
                            operators */
    double  ridge;       /* ISO lambda_ridge (the paper uses 1e-12), >= 0 */
    double  c_min;       /* ISO clip range (the paper uses [0, 1.5]) */
    double  c_max;
    iso_topk_cfg topk;   /* TopKMask of TIES and ISO; ignored by TA and RAM */
} iso_merge_cfg;

/* Per selection unit, written by the device. */
typedef struct {
    uint32_t thresh_key;      /* binary32 bits of the k-th largest |tau|; 0xFFFFFFFF when the
                                 unit selects nothing (k == 0) or is not trimmed */
    uint32_t flags;           /* diagnostics only.  bit 0: resolved by the full-data fallback;
                                 bit 1: fused K = 1 pass took the sampled run of ties as the
                                 threshold; bit 2: fused pass re-applied the unit in full;
                                 bit 3: band keys overflowed their segment; bit 4: fused band
                                 records overflowed; bit 5: the Gram and merge passes read this
                                 unit's compact candidates (iso_compact_candidates) */
    int64_t  k;               /* entries selected; -1 for a unit that is not trimmed */
    int64_t  count_above;     /* entries with |tau| above the threshold */
    int64_t  ties_at_thresh;  /* entries with |tau| equal to the threshold */
    int64_t  ties_taken;      /* of those, how many are selected (lowest index first) */
} iso_unit_stats;

/* Optional device-side outputs of a call; every pointer may be NULL. */
typedef struct {
    int32_t*        status;  /* 1 value: ISO_OK, ISO_ERR_NONFINITE or ISO_ERR_TIMEOUT, valid after the stream
                                reaches the end of the call */
    iso_unit_stats* units;   /* [K][n_units], n_units from iso_num_units; not written by
                                TA and RAM, which trim nothing */
    double*         gram;    /* ISO: [n_tensors][K][K] Gram of the trimmed task vectors
                                (zero for 1-D tensors) */
    double*         coef;    /* ISO: [n_tensors][K] retention coefficients c* */
} iso_merge_stats;

/* Host-only.  Number of selection units per expert for a tensor list under a
 * TopKMask configuration (TENSOR: n_tensors; BLOCK: sum of tile counts;
 * GLOBAL: 1). */
int32_t iso_num_units(const iso_tensor* tensors, int32_t n_tensors, const iso_topk_cfg* topk,
                      int64_t* n_units);

/* Host-only.  Workspace bytes for iso_update / iso_merge (K experts) and, with
 * K = 1, for iso_topk_mask.  *bytes_min receives the smallest workspace the
 * call accepts (tensors are then processed in groups that fit); *bytes_full
 * the size that processes the whole list in one group.  Either pointer may be
 * NULL.  The workspace must be 256-byte aligned. */
int32_t iso_workspace_size(const iso_tensor* tensors, int32_t n_tensors, int32_t K,
                           const iso_merge_cfg* cfg, size_t* bytes_min, size_t* bytes_full);

/* tau[t] = theta_i[t] - theta_0[t] for every tensor (App. F task vector),
 * computed as one binary32 subtraction per entry and stored as ISO_F32.
 * theta_i / theta_0 may be BF16 or F32; tau must be F32 and may not alias the
 * inputs.  Needs no workspace. */
int32_t iso_delta(const iso_tensor* theta_i, const iso_tensor* theta_0, const iso_tensor* tau,
                  int32_t n_tensors, void* stream);

/* TopKMask(|tau|, rho) over a task vector given as n_tensors tensors (BF16 or
 * F32).  mask_bits[t] (device, may be NULL for a tensor, or mask_bits itself
 * NULL) receives ceil(numel / 32) uint32 words: bit j of word w is entry
 * 32 w + j.  stats->units receives [n_units] records; stats->gram / coef are
 * unused. */
int32_t iso_topk_mask(const iso_tensor* tau, int32_t n_tensors, const iso_topk_cfg* cfg,
                      uint32_t* const* mask_bits, const iso_merge_stats* stats,
                      void* workspace, size_t ws_bytes, void* stream);

/* The K = 1 masked update of a base by one expert, the single-expert case of
 * the merge operators (App. F: TIES trim and scale; Sec. 4.2 and App. E:
 * the retention system with K = 1; App. E "Merged parameter scope" for 1-D
 * tensors):
 *   out = theta_0 + c * TopKMask(|tau|) * tau,   tau = update (update_is_delta = 1)
 *                                               or update - theta_0 (a checkpoint)
 * with c = lambda for TIES, c = clip(Gamma / (Gamma + ridge)) for ISO (Gamma the
 * squared norm of the trimmed tensor); ISO leaves 1-D tensors at theta_0 + tau.
 * TA applies lambda * tau untrimmed; RAM with one expert keeps theta_0 +
 * lambda * tau where |tau| > eps_act and theta_0 elsewhere (no TopKMask).
 * out has the base's dtype and may alias
 * theta_0 (each entry is read before it is written by the same thread); it may
 * not alias update. */
int32_t iso_update(const iso_tensor* theta_0, const iso_tensor* update, int32_t update_is_delta,
                   const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg,
                   void* workspace, size_t ws_bytes, const iso_merge_stats* stats, void* stream);

/* Merge K experts (1 <= K <= ISO_MAX_EXPERTS) into the base.  experts holds
 * K * n_tensors descriptors, expert-major (experts[i * n_tensors + t]); they
 * are task vectors (experts_are_deltas = 1) or fine-tuned checkpoints.  All
 * experts share one dtype.  out has the base's dtype and may alias theta_0. */
int32_t iso_merge(const iso_tensor* theta_0, const iso_tensor* experts, int32_t K,
                  int32_t experts_are_deltas, const iso_tensor* out, int32_t n_tensors,
                  const iso_merge_cfg* cfg, void* workspace, size_t ws_bytes,
                  const iso_merge_stats* stats, void* stream);

/* iso_update without a caller workspace.  Some callers cannot allocate device
 * memory where they run the update (an inference-engine plugin whose enqueue
 * path may not call cudaMalloc, a server that freezes its allocator after
 * warm-up, a C host without a device allocator); this entry point serves them.
 * The paper has no counterpart: it is a property of this library's interface.
 *
 * Arguments and results are those of iso_update.  Scratch comes from one
 * static device array of ISO_NOALLOC_SCRATCH_BYTES per device, part of the
 * library's module image and held until the process exits; nothing is
 * allocated or freed.  Tensors are processed in groups that fit the array; a
 * call whose smallest group (one tensor) needs more returns
 * ISO_ERR_WORKSPACE before anything is enqueued.
 *   - The first call on a device looks the array's device address up
 *     (cudaGetSymbolAddress, with that device current) and caches it: make
 *     that first call before any stream capture.
 *   - Every call on a device shares the one array, which keeps the last
 *     call's contents; each call clears what it needs zeroed.  Calls whose
 *     work overlaps on the GPU (different streams, or different host threads
 *     without ordering) race on the array and give undefined results: order
 *     them on one stream. */
#define ISO_NOALLOC_SCRATCH_BYTES (32u << 20)
int32_t iso_update_noalloc(const iso_tensor* theta_0, const iso_tensor* update, int32_t update_is_delta,
                           const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg,
                           const iso_merge_stats* stats, void* stream);

/* ---- One selection unit split over several GPUs (App. F, TIES trim) -------
 *
 * A unit too large for one GPU (a GLOBAL-scope unit, or an embedding split
 * with its tensor) is held as contiguous ranges of its positions, rank r's
 * range before rank r + 1's.  The exact TopKMask of the whole unit is a radix
 * descent over the magnitude keys whose per-digit counts are summed over the
 * ranks; each rank runs the two calls below on its own range and the host
 * exchanges the counts (paper_2607_19331_gb300/shard.py, split_unit_select).
 * The threshold t and the ties each rank keeps follow the library's rules:
 * k = floor(rho N + 1/2) over the unit's N entries, ties at t taken lowest
 * position first over the whole unit.
 *
 * key_e is the binary32 bits of |tau_e| with the sign cleared, tau_e = x_e
 * (base = NULL: x is a task vector) or x_e - base_e in binary32 (x a
 * checkpoint of the base; same shape, either dtype).  [begin, end) is a range
 * of x's flat (row-major) positions.  Device pointers; enqueued on stream;
 * argument errors are returned before anything is enqueued.  Non-finite
 * values are counted by their keys (above 0x7F800000) and not reported. */

/* counts[b] (int64, nbins entries, overwritten) = the number of positions e
 * in [begin, end) with key_e >> pshift == prefix and
 * (key_e >> shift) & (nbins - 1) == b.  nbins a power of two <= 4096,
 * 0 <= shift <= pshift <= 32.  With nbins = 1 and pshift = shift = 0 the one
 * count is the number of keys equal to prefix. */
int32_t iso_range_hist(const iso_tensor* x, const iso_tensor* base, int64_t begin, int64_t end,
                       uint32_t prefix, int32_t pshift, int32_t shift, int32_t nbins, int64_t* counts,
                       void* stream);

/* Host-only.  Workspace bytes of iso_range_mask for a range of n positions. */
int32_t iso_range_mask_workspace_size(int64_t n, size_t* bytes);

/* mask_bits (ceil((end - begin) / 32) uint32 words, bit j of word w for
 * position begin + 32 w + j, bits past end zero): set where key_e > t, or
 * key_e == t and fewer than take keys equal to t lie in [begin, e).  t and
 * take come from the unit's selection (take = this rank's share of the ties
 * the unit keeps); t = 0xFFFFFFFF selects nothing.  The workspace (8-byte
 * aligned) holds per-tile tie counts. */
int32_t iso_range_mask(const iso_tensor* x, const iso_tensor* base, int64_t begin, int64_t end, uint32_t t,
                       int64_t take, uint32_t* mask_bits, void* workspace, size_t ws_bytes, void* stream);

/* ---- The K = 1 update of a parameter set held in host memory --------------
 *
 * The update of iso_update (same operation, same configuration, same results
 * bit for bit) for tensors that live in host memory: a model on the host that
 * is fine-tuned, merged or corrected on the GPU and read back.  The paper has
 * no counterpart; the call is an interface of this library.
 *
 * The tensor list is cut into groups of consecutive tensors of about
 * group_bytes each (theta_0 + update + out bytes; a GLOBAL-scope TopKMask,
 * one unit over every tensor, makes one group of the whole list).  Groups go
 * through two device slots (one when the list forms one group) of the
 * caller's staging buffer in a pipeline over
 * three caller streams: streams[0] copies a group's theta_0 and update in,
 * streams[1] runs iso_update on it, streams[2] copies its out back, so the
 * copies of one group overlap the update of the next.  Tensors whose host
 * copies follow one another in ascending order are moved by one copy (inputs
 * may have gaps below 4096 bytes between them, which are read but not used;
 * outputs only exactly adjacent runs, so no host byte outside an out tensor
 * is written).
 *
 *   theta_0, update, out   host descriptors (16-byte aligned like every
 *                          tensor); the overlap rules of iso_update apply to
 *                          them.  Page-locked host memory (cudaHostAlloc or
 *                          cudaHostRegister) lets the copies run
 *                          asynchronously; with pageable memory the runtime
 *                          makes them synchronous and the pipeline serialises.
 *   staging                device buffer, 256-byte aligned, of at least the
 *                          size iso_update_host_staging_size returns for the
 *                          same descriptors, configuration and group_bytes;
 *                          it holds the two slots, the update's workspace
 *                          and a per-group status array.
 *   stats                  device-side outputs as for iso_update (units, gram
 *                          and coef for the whole list; status combined over
 *                          the groups: the first group's error that is not
 *                          ISO_OK).
 *   streams                three CUDA streams (h2d, compute, d2h); they may
 *                          be one and the same stream (no overlap).
 * The call enqueues and returns.  The whole call has finished, out written
 * in host memory included, once streams[1] reaches the point where the call
 * returned.  Argument errors return before anything is enqueued; a CUDA error
 * while enqueueing returns ISO_ERR_CUDA with earlier groups enqueued. */
int32_t iso_update_host_staging_size(const iso_tensor* theta_0, const iso_tensor* update,
                                     const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg,
                                     size_t group_bytes, size_t* bytes);
int32_t iso_update_host(const iso_tensor* theta_0, const iso_tensor* update, int32_t update_is_delta,
                        const iso_tensor* out, int32_t n_tensors, const iso_merge_cfg* cfg,
                        size_t group_bytes, void* staging, size_t staging_bytes,
                        const iso_merge_stats* stats, void* const* streams);

/* ---- Frame-space ISO-Merger of one weight matrix (App. E) ----------------
 *
 * The paper's merge of K experts fine-tuned from one base, per 2-D weight
 * matrix (App. E, Setup to Retraction and reconstruction): experts' singular
 * frames aligned to the base's sign gauge (Sign canonicalization), their
 * displacements projected onto the Stiefel tangent spaces at the base frames
 * (Stiefel tangent projection) and masked to the leading k_keep modes
 * (Top-k_keep singular-mode masking), retention coefficients from the Gram of
 * the first-order effect proxies (Retention coefficients), the aggregate
 * tangent retracted by the polar factor, and W* = U* S_0 V*^T carrying the
 * base spectrum (Retraction and reconstruction). */
typedef struct {
    double  rho_keep;   /* (0, 1]: k_keep = floor(rho_keep q + 1/2) leading modes, q = min(m, n)
                           (the paper uses 0.9) */
    double  ridge;      /* lambda_ridge >= 0 (the paper uses 1e-12) */
    double  c_min;      /* clip range (the paper uses [0, 1.5]) */
    double  c_max;
    int32_t ns_iters;   /* iteration limit of the inverse square root in the polar factor;
                           0 = the default (16); the iteration stops at convergence */
    int32_t reserved;   /* must be 0 */
} iso_frame_cfg;

/* Host-only.  Workspace bytes of iso_frame_merge for an m x n matrix and K
 * experts (1 <= K <= ISO_MAX_EXPERTS, min(m, n) <= 32768, m, n < 2^24). */
int32_t iso_frame_workspace_size(int64_t m, int64_t n, int32_t K, size_t* bytes);

/* Merge one m x n matrix.  Inputs are thin SVDs, binary64, row-major, on the
 * device, singular values in descending order (q = min(m, n)):
 *   U0 (m x q), S0 (q), Vt0 (q x n)      the base, W_0 = U0 diag(S0) Vt0
 *   U[i] (m x q), Vt[i] (q x n)          expert i's frames (host array of K
 *                                        device pointers); its singular values
 *                                        are not needed
 * W0 is the base matrix itself (ISO_BF16 or ISO_F32, m x n); out (same dtype
 * and shape, may coincide with W0 but share no other byte with it) receives
 *   W* = W0 + (U* S0 V*^T - U0 S0 V0^T),
 * i.e. the paper's U* S0 V*^T with the base's own entries in place of their
 * reconstruction from the factors.  stats (may be NULL): status (ISO_OK or
 * ISO_ERR_TIMEOUT), gram [K][K] (Gamma), coef [K] (c*); units is not used.
 * The workspace (256-byte aligned, iso_frame_workspace_size bytes) is
 * scratch for the duration of the call.  Precision: the large contractions
 * run on the tensor cores as three tf32 products per pair (binary32
 * accumulation, about 2^-21 relative each), the rest in binary64.  Argument
 * errors are returned before anything is enqueued. */
int32_t iso_frame_merge(const double* U0, const double* S0, const double* Vt0, const double* const* U,
                        const double* const* Vt, int32_t K, int64_t m, int64_t n, const iso_tensor* W0,
                        const iso_tensor* out, const iso_frame_cfg* cfg, void* workspace, size_t ws_bytes,
                        const iso_merge_stats* stats, void* stream);

/* ---- ISO-Optimizer step ISO[AdamW] on one weight matrix (Sec. 4.3) -------
 *
 * The fixed-spectrum parameterisation W(U, V) = U S0 V^T with AdamW applied
 * to the frames: the factor gradients G_U = G_W V S0 and G_V = G_W^T U S0
 * (Sec. 4.3, factor gradients), AdamW on U and on V with their own moments
 * (the base optimizer on the factors; decoupled weight decay, bias-corrected
 * moments), the polar retraction U+ = polar(U_bar), V+ = polar(V_bar) and
 * W+ = U+ S0 V+^T (Sec. 4.3 with the polar factor of App. E). */
typedef struct {
    double  lr;            /* learning rate >= 0 */
    double  beta1, beta2;  /* moment decays in [0, 1) */
    double  eps;           /* > 0 */
    double  weight_decay;  /* >= 0 (decoupled; the paper uses 0) */
    int64_t step;          /* this update's step number, from 1 (bias correction) */
    int32_t ns_iters;      /* iteration limit of the polar factor's inverse square root;
                              0 = the default (16); it stops at convergence */
    int32_t reserved;      /* must be 0 */
} iso_adamw_cfg;

/* Host-only.  Workspace bytes of iso_opt_step for an m x n matrix
 * (m, n < 2^24, min(m, n) <= 32768). */
int32_t iso_opt_workspace_size(int64_t m, int64_t n, size_t* bytes);

/* One ISO[AdamW] step of an m x n matrix, q = min(m, n).  Device pointers:
 *   U (m x q), V (n x q)   binary64 frames with orthonormal columns, updated in place
 *   S0 (q)                 the fixed spectrum
 *   G_W                    the gradient with respect to W (m x n, ISO_BF16 or ISO_F32)
 *   mU, vU (m x q), mV, vV (n x q)  binary32 AdamW moments, updated in place
 *                          (zero before the first step)
 *   W                      the current weight matrix U S0 V^T as stored (bf16 / fp32)
 *   W_out                  receives W + (U+ S0 V+^T - U S0 V^T); same dtype, may
 *                          coincide with W (each entry read and written by one
 *                          thread) but share no other byte with it
 * The retraction takes polar(F_bar) = F_bar (F_bar^T F_bar)^(-1/2) with
 * F_bar^T F_bar formed in binary64, so it also restores orthonormality lost
 * to rounding in earlier steps.  Precision: the factor gradients and the
 * retraction's remaining products are three tf32 products per pair with
 * binary32 accumulation (about 2^-22 relative each); the AdamW arithmetic,
 * F_bar^T F_bar and the frames are binary64.  stats->status (may be NULL) receives ISO_OK or
 * ISO_ERR_TIMEOUT.  Argument errors are returned before anything is enqueued. */
int32_t iso_opt_step(double* U, double* V, const double* S0, const iso_tensor* G_W, float* mU, float* vU,
                     float* mV, float* vV, const iso_tensor* W, const iso_tensor* W_out, int64_t m, int64_t n,
                     const iso_adamw_cfg* cfg, void* workspace, size_t ws_bytes, const iso_merge_stats* stats,
                     void* stream);

/* The frame merge's dense product on the tensor cores, for tests of the
 * contraction alone: C (M x N, row stride ldc) = A[:, a_k0 : a_k0 + Kc]
 * B[:, b_k0 : b_k0 + Kc]^T, A (M rows, stride lda) and B (N rows, stride
 * ldb) row-major binary32 read as tf32, binary32 accumulation.  M and N
 * multiples of 128; Kc, a_k0 and b_k0 multiples of 32; strides multiples of
 * 4; pointers 16-byte aligned.  Device pointers; enqueued on stream. */
int32_t iso_gemm_tf32(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                      int64_t N, int64_t Kc, int64_t a_k0, int64_t b_k0, void* stream);

/* Static description of a status code. */
const char* iso_error_string(int32_t status);

/* Diagnostics: number of kernels this process has launched through the
 * library (all streams, all devices). */
uint64_t iso_launch_count(void);

/* Diagnostics: the K = 1 update of a bf16 base by a bf16 update under
 * per-tensor TopKMask normally runs as one fused pass over the inputs
 * (speculative outputs from the sampled threshold, then an exact correction);
 * on = 1 makes later calls take the two-pass form instead (a counting pass,
 * then the apply pass).  Both give the same result.  Process-wide host state. */
int32_t iso_force_two_pass(int32_t on);

/* Diagnostics: whether later K >= 2 TIES and ISO merges at per-tensor scope
 * (density <= 0.3) let the counting pass write each expert's candidate values
 * (the entries at or above the low edge of its sampled band, in position
 * order, with a bit mask per tile), so that the Gram and merge passes read
 * those instead of the full task vectors; off by default.  The results are
 * the same either way. */
int32_t iso_compact_candidates(int32_t on);

/* Diagnostics: when enabled, each launch is bracketed by CUDA events on its
 * stream.  iso_profile_read waits for the recorded events and returns, for
 * kernel `kind` (0 .. iso_profile_kinds()-1), the number of launches and their
 * summed device time since the last reset.  Profiling is host state, not
 * thread-safe, and off by default. */
int32_t     iso_profile_enable(int32_t on);
int32_t     iso_profile_reset(void);
int32_t     iso_profile_kinds(void);
const char* iso_profile_name(int32_t kind);
int32_t     iso_profile_read(int32_t kind, int64_t* launches, double* total_ms);

#ifdef __cplusplus
}
#endif
#endif /* ISO_H */
