/*
 * fademem.h -- C ABI of the GB300 (sm_103a) implementation of FadeMem's
 * per-segment memory step (arxiv 2606.10671, "FadeMem: Distance-Aware Memory
 * Consolidation for Autoregressive Video Diffusion").
 *
 * The memory (Sec. 3.1) is an ordered set of at most M entries per layer.
 * Each entry stores one representative K/V block of N tokens x H heads x D
 * dims, its temporal centre mu and its span s (Sec. 3.3, "Memory entries").
 * Each generated unit (one latent frame, Sec. S4) is inserted as a new entry;
 * when the budget is exceeded, the power-law schedule picks the adjacent pair
 * with the smallest warped gap |(t-mu_{i+1})^beta - (t-mu_i)^beta| and the
 * pair is consolidated (Sec. 3.3; Algorithm S1).  The segment's queries then
 * attend over the consolidated memory, per head and per layer (Sec. 3.3, last
 * paragraph; Sec. 4.1: attention every denoising step, memory update after
 * the last one).
 *
 * Conventions (every entry point):
 *   - Returns a fademem_status; never aborts, never throws across the ABI.
 *     On failure fademem_last_error() describes the problem (thread-local).
 *   - Device pointers are CUDA device addresses; they must be 16-byte
 *     aligned, else FADEMEM_ERR_INVALID_ARG.  Host pointers are plain memory.
 *   - Work is enqueued asynchronously on the given stream (a cudaStream_t
 *     passed as void*; NULL = the legacy default stream).  Calls that return
 *     data to the host synchronise that stream first.
 *   - A handle is not thread-safe; use one handle per thread or serialise.
 *   - Frames are counted from t = 0 (the first inserted frame is the anchor).
 */
#ifndef FADEMEM_H
#define FADEMEM_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define FADEMEM_API __attribute__((visibility("default")))
#else
#define FADEMEM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Largest entry budget M accepted by fademem_create. */
#define FADEMEM_MAX_BUDGET 64
/* Largest number of layers one handle holds. */
#define FADEMEM_MAX_LAYERS 128
/* Largest number of frames pending (inserted, not yet consolidated) per layer. */
#define FADEMEM_MAX_PENDING 64

/* Bits of the device status word (fademem_get_device_status). */
#define FADEMEM_STATUS_TIMEOUT 0x1u
#define FADEMEM_STATUS_COUNT_MISMATCH 0x2u
#define FADEMEM_STATUS_PLAN_OVERFLOW 0x4u
#define FADEMEM_STATUS_NEAR_TIE 0x8u
#define FADEMEM_STATUS_BOUNDS 0x10u

/* Bits of fademem_build_flags(). */
#define FADEMEM_BUILD_DEBUG_BOUNDS 0x1u

typedef enum fademem_status {
    FADEMEM_OK = 0,
    FADEMEM_ERR_INVALID_ARG = 1,    /* NULL / misaligned pointer, out-of-range size or index */
    FADEMEM_ERR_UNSUPPORTED = 2,    /* valid but not implemented (e.g. bf16 with head_dim 64) */
    FADEMEM_ERR_WORKSPACE = 3,      /* workspace too small or misaligned */
    FADEMEM_ERR_EMPTY = 4,          /* attend on a memory with no entries */
    FADEMEM_ERR_PENDING = 5,        /* attend while inserted frames await consolidation */
    FADEMEM_ERR_CUDA = 6,           /* a CUDA runtime call failed (message has the CUDA error) */
    FADEMEM_ERR_DEVICE_TIMEOUT = 7, /* a device-side bounded wait gave up (see device status) */
    FADEMEM_ERR_DEVICE_CHECK = 8    /* a device-side consistency check failed */
} fademem_status;

typedef enum fademem_dtype {
    FADEMEM_F32 = 0,   /* fp32 storage and arithmetic (exact reference path) */
    FADEMEM_BF16 = 1   /* bf16 storage, fp32 accumulation; tensor-core attention */
} fademem_dtype;

/* Consolidation operator (Sec. 3.3; ablation of Table 2). */
typedef enum fademem_merge_op {
    FADEMEM_MERGE_WEIGHTED = 0,       /* default: weights sqrt(s_j), sqrt(s_{j+1}), normalised */
    FADEMEM_MERGE_AVERAGE = 1,        /* unweighted mean of the two blocks */
    FADEMEM_MERGE_SELECT_NEAREST = 2, /* keep the block of the entry nearer the current step (m_{j+1}) */
    FADEMEM_MERGE_MAX_POOL = 3        /* elementwise maximum */
} fademem_merge_op;

typedef struct fademem_config {
    int budget;            /* M: entries per layer, 2 <= M <= FADEMEM_MAX_BUDGET (Sec. 3.1) */
    int heads;             /* H >= 1 */
    int head_dim;          /* D: 64 or 128 (bf16 attention: 128) */
    int tokens_per_frame;  /* N >= 1: tokens in one unit's KV block (Sec. 3.1) */
    int num_layers;        /* L: 1 <= L <= FADEMEM_MAX_LAYERS; all layers share one schedule */
    double beta;           /* warp exponent of u(d) = d^beta, 0 < beta <= 1 (Sec. 3.3) */
    int anchor;            /* 1: keep the first frame as global anchor (Sec. 3.3; Algorithm S1) */
    int merge_op;          /* fademem_merge_op */
    int dtype;             /* fademem_dtype of K, V, Q, out and the stored memory */
    float scale;           /* softmax scale of q.k; 0 selects 1/sqrt(D) */
    /* Temporal RoPE handling (Sec. 3.3, "Boundary and positional handling"):
     * rope_pairs = P complex pairs (dims 2k, 2k+1, k < P) of each head's key
     * carry the temporal rotary phase, frequencies omega_k = theta^(-k/P).
     * 0 turns it off (keys are stored and attended as given).  With P > 0,
     * inserted keys carry their frame's phase (position t = the frame's index)
     * and are stored with it removed; consolidate then writes the keys
     * attention uses: entry i of count (temporal order) rotated to position
     * t_next - count + i, consecutive positions ending right before the next
     * frame t_next, so the exposed range is bounded by M (the paper does not
     * give the re-index rule; this is the library's reading).  Queries and the
     * chunk keys of fademem_attend_ext keep the positions the caller gave. */
    int rope_pairs;        /* 0 <= P <= head_dim / 2 */
    double rope_theta;     /* RoPE base; 0 selects 10000 */
} fademem_config;

typedef struct fademem_ctx *fademem_t;

/* Bytes of device workspace a handle with this configuration needs (the
 * memory of every layer, [L][K|V][H][M][N][D] in the storage dtype -- with
 * temporal RoPE, [L][K|V|K_attention][H][M][N][D] -- plus metadata and the
 * merge plan), or 0 if the configuration is invalid.
 * Host only; no CUDA call. */
FADEMEM_API size_t fademem_workspace_bytes(const fademem_config *cfg);

/* Create a memory (Sec. 3.1: empty, |M_0| = 0) over caller-owned device
 * workspace (>= fademem_workspace_bytes, 256-byte aligned).  The caller keeps
 * ownership of the workspace and must keep it alive until fademem_destroy.
 * Host only: the metadata is initialised by the first device call.
 * Errors: INVALID_ARG (bad config, NULL out), UNSUPPORTED, WORKSPACE. */
FADEMEM_API fademem_status fademem_create(const fademem_config *cfg, void *workspace, size_t workspace_bytes,
                                          fademem_t *out);

/* Register nframes new units for one layer (Sec. 3.3, "insertion": each unit
 * becomes an entry (K_t, V_t, mu = t, s = 1)).  K and V are device arrays of
 * [nframes * N][H][D] in the config dtype (token-major, frames in generation
 * order).  No data moves here: the arrays are borrowed and must stay valid
 * and unmodified until fademem_consolidate has been enqueued and the stream
 * has reached it.  Every layer must register the same frames before the next
 * consolidate.  Errors: INVALID_ARG, PENDING (over FADEMEM_MAX_PENDING). */
FADEMEM_API fademem_status fademem_insert(fademem_t h, int layer, const void *K, const void *V, int nframes);

/* Apply Algorithm S1 once per pending frame, in order, to every layer:
 * append, and while over budget compute the warped gaps on the device, take
 * the argmin (lowest index on ties) over the eligible pairs (all but the pair
 * holding the newest entry), merge its span/centre (anchor rule for the pair
 * holding the first frame), and consolidate the pair's K/V blocks in place.
 * Consecutive frames are fused into one pass over the memory (each source
 * block read once, each changed slot written once).  Asynchronous on stream.
 * Storage slots: the merged entry keeps m_j's slot, the new entry takes
 * m_{j+1}'s; occupied slots are always 0..count-1.
 * The schedule depends on the entry table alone, so the consolidation kernel
 * of a single-pass call also schedules the next pass (assuming the same number
 * of frames) into a second entry-table buffer of the workspace; the next call
 * with that frame count then launches only the consolidation kernel, and any
 * other count schedules as usual.
 * Errors: INVALID_ARG (layers with different pending frames), CUDA. */
FADEMEM_API fademem_status fademem_consolidate(fademem_t h, void *stream);

/* Attention of Lq query tokens over every token of every entry of one layer,
 * per head: out = softmax(scale * Q K^T) V (keys and values of all count*N
 * cached tokens; non-causal, all cached keys precede the queries).  Q, out:
 * device arrays [Lq][H][D] in the config dtype.  Asynchronous on stream.
 * Errors: INVALID_ARG, EMPTY (no entries), PENDING (frames not consolidated),
 * UNSUPPORTED, CUDA. */
FADEMEM_API fademem_status fademem_attend(fademem_t h, int layer, const void *Q, void *out, int Lq, void *stream);

/* Attention over the memory and the current chunk (the paper's attention sees
 * the cached entries plus the frames of the chunk being generated: 12 history
 * + 3 current latent frames by default, Sec. 4.1; Sec. S4).  As
 * fademem_attend, with the key set extended by ncur >= 0 tokens whose keys and
 * values the caller passes: Kcur, Vcur device arrays [ncur][H][D] in the
 * config dtype (for a chunk of F frames, ncur = F * N).  With ncur = 0 this is
 * fademem_attend; with an empty memory the queries attend over the chunk
 * alone.  Errors: INVALID_ARG, EMPTY (no entries and ncur = 0), PENDING,
 * UNSUPPORTED, CUDA. */
FADEMEM_API fademem_status fademem_attend_ext(fademem_t h, int layer, const void *Q, const void *Kcur,
                                              const void *Vcur, int ncur, void *out, int Lq, void *stream);

/* Number of entries (count = min(frames seen, M)) and frames seen so far,
 * counting consolidated frames only.  Host only. */
FADEMEM_API fademem_status fademem_counts(fademem_t h, int *count, int64_t *frames_seen);

/* Copy the entry table back, in temporal order (synchronises stream):
 * slot (storage slot of entry i), first (first unit summarised), span (s),
 * mu2 (2*mu, exact integer).  Arrays hold >= capacity elements; *count gets
 * the number of entries.  Errors: INVALID_ARG (capacity too small), CUDA. */
FADEMEM_API fademem_status fademem_get_entries(fademem_t h, void *stream, int capacity, int *count, int32_t *slot,
                                               int64_t *first, int64_t *span, int64_t *mu2);

/* Size of the most recent consolidation pass's merge plan (synchronises
 * stream): *n_src source blocks read (old entries and new frames), *n_dest
 * slots written, *frames units in the pass.  Each block is N*H*D elements of
 * K plus as many of V per layer, so the pass moves (n_src + n_dest) blocks of
 * K and V per layer: the algorithmic HBM traffic of the consolidation. */
FADEMEM_API fademem_status fademem_last_plan(fademem_t h, void *stream, int *n_src, int *n_dest, int *frames);

/* Counters (synchronises stream; any out pointer may be NULL).  Kept on the
 * device since create/reset: *blocks_moved = the sum over consolidation
 * passes of (sources read + slots written), each block one entry's K and V
 * of every layer, so the algorithmic HBM bytes of all passes are
 * blocks_moved * L * 2*N*H*D*elem; *passes = consolidation passes.  Kept on
 * the host since create (not cleared by reset): *kernel_launches = kernels
 * this handle has launched (schedule, consolidation, attention, self-test). */
FADEMEM_API fademem_status fademem_stats(fademem_t h, void *stream, uint64_t *blocks_moved, uint64_t *passes,
                                        uint64_t *kernel_launches);

/* Device pointers to one layer's stored K and V memory, each laid out as
 * [H][M][N][D] in the storage dtype; storage slot s of head h starts at
 * ((h * M) + s) * N * D elements.  Only slots 0..count-1 hold entries. */
FADEMEM_API fademem_status fademem_layer_memory(fademem_t h, int layer, void **K, void **V);

/* Read and clear the device status word (synchronises stream).  Returns OK,
 * DEVICE_TIMEOUT (a bounded wait in a kernel gave up) or DEVICE_CHECK; the
 * raw word goes to *word when word is not NULL.  Bits of the word:
 *   FADEMEM_STATUS_TIMEOUT         a bounded device wait gave up;
 *   FADEMEM_STATUS_COUNT_MISMATCH  host and device entry counts disagreed;
 *   FADEMEM_STATUS_PLAN_OVERFLOW   a merge plan exceeded its static bounds;
 *   FADEMEM_STATUS_NEAR_TIE        a schedule decision of Algorithm S1 (the
 *     argmin of the warped gaps, Sec. 3.3) was not certified: its best and
 *     second-best gaps were equal within the fp64 evaluation error of d^beta
 *     (2^-48 of the sum of the four u values involved) and not exactly
 *     computable (beta = 1, or beta = 0.5 on exact square roots, are).  The
 *     decision taken (lowest index among the equal minima) is a valid one,
 *     but another fp64 evaluation of d^beta, such as a host libm's, may
 *     choose the other pair.  The message names the first such frame.
 * Every other configuration decides each merge exactly as an fp64 evaluation
 * of Algorithm S1 does.
 *   FADEMEM_STATUS_BOUNDS          (bounds-checking build only, see
 *     fademem_build_flags) a kernel found a global-memory access outside the
 *     buffer it belongs to, or a table index outside its array, and skipped
 *     it; the results of that call are not to be trusted. */
FADEMEM_API fademem_status fademem_get_device_status(fademem_t h, void *stream, uint32_t *word);

/* Diagnostic of device-side failure detection: enqueues one thread that waits,
 * through the same bounded mbarrier wait the kernels use, on a barrier that
 * nothing signals.  After about 1 ms the wait gives up and records a time-out
 * in the status word, so the next fademem_get_device_status returns
 * FADEMEM_ERR_DEVICE_TIMEOUT; the CUDA context stays usable.  The paper has
 * no counterpart.  Errors: INVALID_ARG, CUDA. */
FADEMEM_API fademem_status fademem_selftest_wait_timeout(fademem_t h, void *stream);

/* Forget every entry (count = 0, t = 0).  Enqueued on stream. */
FADEMEM_API fademem_status fademem_reset(fademem_t h, void *stream);

/* Bytes of library-owned device scratch used by fademem_consolidate_noalloc. */
#define FADEMEM_NOALLOC_SCRATCH_BYTES 4096

/* fademem_consolidate without any scratch in the caller's workspace and without
 * any allocation (no cudaMalloc, cudaFree or allocating library call): the
 * per-call working state (a copy of the entry table and the merge plan)
 * lives in a file-scope device array of the library, of
 * FADEMEM_NOALLOC_SCRATCH_BYTES bytes, that every GPU which loads the library
 * holds until the process exits.  The paper has no counterpart: this serves
 * callers that may not allocate device memory once they are running, such as
 * plug-ins of a host framework that owns all device memory, or real-time loops
 * that fix their memory at start-up.  The caller still passes the memory
 * (workspace of fademem_create) and the inserted frames, as for
 * fademem_consolidate, and the results are the same.  The device status word
 * stays in the workspace; no schedule is computed ahead.
 * The first call on each device looks up the array's device address with that
 * device current (cudaGetSymbolAddress); make that first call before any
 * stream capture.  Every call shares the one array: calls that overlap on the
 * GPU (other streams, other handles, other threads) race and must be
 * serialised by the caller.  Nothing in the array needs clearing: each call
 * overwrites it from the handle's workspace before use.  The array holds the
 * entry table of every budget fademem_create accepts (up to
 * FADEMEM_MAX_BUDGET; checked when the library is compiled).  Errors as
 * fademem_consolidate. */
FADEMEM_API fademem_status fademem_consolidate_noalloc(fademem_t h, void *stream);

/* Device staging bytes fademem_step_host needs for segments of `nframes`
 * frames per layer and `Lq` query tokens: two slots, each holding the inputs
 * (K and V of every layer, Q) and the output block of one step.  0 if cfg is
 * invalid or nframes/Lq out of range.  No CUDA call is made. */
FADEMEM_API size_t fademem_host_staging_bytes(const fademem_config *cfg, int nframes, int Lq);

/* One step of a serving loop with the inputs and the result in HOST memory
 * (the paper has no counterpart: it is the library's own serving entry):
 * copy the segment's frames and the queries in, insert the frames on every
 * layer, consolidate (Algorithm S1 and the merges of Sec. 3.3), attend the
 * queries over `layer`'s memory (Sec. 3.3, last paragraph), and copy the
 * output back -- the same work as fademem_insert per layer +
 * fademem_consolidate + fademem_attend, with the same results.
 *   K_host[l], V_host[l]  per layer l < num_layers: [nframes*N][H][D] of the
 *                         storage dtype (page-locked memory lets the copies
 *                         run asynchronously; pageable memory also works)
 *   Q_host                [Lq][H][D]; out_host [Lq][H][D] (written)
 *   staging               caller-owned device memory of at least
 *                         fademem_host_staging_bytes(cfg, nframes, Lq) bytes,
 *                         16-byte aligned, used by this handle only and the
 *                         same on every call with these sizes
 * The step runs on three streams of the handle's own -- host-to-device
 * copies, kernels, device-to-host copy -- and alternates between the two
 * staging slots, so consecutive calls overlap: the next call's input copies
 * and kernels run while this call's output is copied out.  The step starts
 * after the work enqueued on `stream` before the call, and `stream` waits for
 * the step's output copy: once `stream` has synchronised, out_host holds this
 * call's output and the host inputs of this call may be reused.  Other work
 * of this handle must be ordered through `stream` as well.
 * Errors as fademem_insert / fademem_consolidate / fademem_attend, plus
 * FADEMEM_ERR_WORKSPACE if staging is too small or misaligned. */
FADEMEM_API fademem_status fademem_step_host(fademem_t h, const void *const *K_host, const void *const *V_host,
                                            int nframes, int layer, const void *Q_host, void *out_host, int Lq,
                                            void *staging, size_t staging_bytes, void *stream);

/* Checkpoint / resume (the paper has none; for long rollouts such as an
 * hour-long stream).  A snapshot holds the configuration, the entry table
 * (spans, centres, slots, frames seen) and the stored K/V of every layer;
 * the re-indexed RoPE keys are rebuilt on import.  Snapshots are plain host
 * bytes with a versioned header, valid across processes and devices of this
 * library version.
 * fademem_state_bytes: size of a snapshot of this handle (0 if h is NULL). */
FADEMEM_API size_t fademem_state_bytes(fademem_t h);
/* Write a snapshot into host memory (>= fademem_state_bytes).  Synchronises
 * stream first.  Errors: INVALID_ARG, PENDING (frames inserted but not
 * consolidated), WORKSPACE (buffer too small), CUDA. */
FADEMEM_API fademem_status fademem_export_state(fademem_t h, void *host_buf, size_t bytes, void *stream);
/* Replace this handle's memory with a snapshot taken from a handle of the
 * same configuration (every fademem_config field equal).  Any pending frames
 * are dropped.  Synchronises stream.  Errors: INVALID_ARG (not a snapshot,
 * other version, other configuration, inconsistent contents), CUDA. */
FADEMEM_API fademem_status fademem_import_state(fademem_t h, const void *host_buf, size_t bytes, void *stream);

/* Release the handle (NULL-safe).  Does not free the caller's workspace. */
FADEMEM_API void fademem_destroy(fademem_t h);

/* How this library was built (no counterpart in the paper): a set of
 * FADEMEM_BUILD_* bits.  FADEMEM_BUILD_DEBUG_BOUNDS: every kernel checks each
 * global-memory access against the buffer it belongs to (the workspace's
 * memory slabs, the caller's frames, queries and outputs) and each table
 * index against its array, skips an access that fails and sets
 * FADEMEM_STATUS_BOUNDS; built by `build.py --debug-bounds` as
 * libfademem_debug.so, slower, for testing.  0 for the release library.
 * Needs no GPU. */
FADEMEM_API uint32_t fademem_build_flags(void);

/* Message of the last failed call on this thread ("" if none). */
FADEMEM_API const char *fademem_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* FADEMEM_H */
