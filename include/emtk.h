/*
 * emtk.h -- C ABI of the GB300 EmTrackMichelId hit-identification library.
 *
 * The library computes, on one GPU, what arXiv:2009.04509 offloads to its
 * inference servers: for every reconstructed wire hit, a 48x48 patch of
 * deconvolved charge (rows = wires, columns = time intervals of 6 ticks) is
 * cut around the hit (Sec. 2.1), and the EmTrackMichelId network scores it
 * (Sec. 2.2): conv 5x5 with 48 filters + ReLU, dense 128 + ReLU, dense 32 +
 * ReLU, a 3-way softmax (track, em, none) and a 1-way sigmoid (Michel).
 *
 * Conventions for every entry point below:
 *   - Pointers named d_* are device memory owned by the caller (host memory
 *     in emtk_infer_batch_host, which says so).  They must stay valid until
 *     the work enqueued on the caller's stream completes.
 *   - All work is enqueued on the caller's stream; nothing synchronises
 *     unless stated.  A context may be used from one stream at a time.
 *   - Argument errors are reported synchronously and enqueue nothing.
 *     Launch failures return EMTK_ERR_CUDA.  A device-side wait that gave up
 *     (EMTK_ERR_TIMEOUT) is reported by emtk_check().
 *   - For a fixed precision and fixed sizes, results are bit-identical from
 *     run to run.
 *   - Every hit coordinate is valid: pixels that fall outside the plane are
 *     zero, so a hit far outside the plane gets an all-zero patch.
 */
#ifndef EMTK_H
#define EMTK_H

#include <stdint.h>

#if defined(__GNUC__)
#define EMTK_API __attribute__((visibility("default")))
#else
#define EMTK_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as the CUDA runtime's cudaStream_t; NULL is the legacy default
 * stream. */
typedef struct CUstream_st *emtk_stream;

typedef struct emtk_ctx emtk_ctx;

typedef enum {
    EMTK_OK = 0,
    EMTK_ERR_ARG = 1,         /* null pointer, negative size, bad enum, ... */
    EMTK_ERR_ALIGN = 2,       /* d_adc not 16-byte aligned or ld % 4 != 0 */
    EMTK_ERR_OOM = 3,         /* device allocation failed */
    EMTK_ERR_CUDA = 4,        /* a CUDA call or launch failed */
    EMTK_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
    EMTK_ERR_UNSUPPORTED = 6  /* precision or device not supported */
} emtk_status;

/* Arithmetic of the network.
 *   EMTK_FP32: fp32 operands, fp32 accumulation (CUDA cores).
 *   EMTK_BF16: bf16 patch, conv weights, conv activations and dense-1
 *              weights; fp32 accumulation on the tcgen05 tensor cores;
 *              dense-2 and heads in fp32.
 *   EMTK_FP16: as EMTK_BF16 with IEEE fp16 operands (same tensor rate,
 *              8x finer rounding; activations above 65504 saturate).
 *   EMTK_FP8:  the conv as EMTK_BF16; dense-1 (92,928 -> 128, Sec. 2.2)
 *              with FP8 E4M3 operands (4 exponent bits, bias 7, 3 mantissa
 *              bits, largest finite 448; round to nearest even, saturating
 *              to +-448) at twice the bf16 tensor rate.  Both operands are
 *              scaled by powers of two before rounding: activations by
 *              s_a = 2^-4, weights by s_w, the largest power of two with
 *              max|W1| * s_w <= 448; the fp32 sums are multiplied by
 *              1 / (s_a s_w) before the dense-1 bias (emtk_get_fp8_scales).
 *              Patches are bf16.
 *   EMTK_TF32: fp32 accuracy on the tcgen05 tensor cores.  Every fp32
 *              operand of the conv and of dense-1 (patch pixels, conv
 *              weights and bias, conv activations, dense-1 weights) is
 *              written as the sum of two fp16 values, a head and a tail
 *              (22 significant bits together, as many as a TF32 head and
 *              tail), and every product is taken as three fp16 products
 *              (head x head, head x tail, tail x head) accumulated in fp32:
 *              the operand-splitting method of Markidis et al. (2018), at
 *              the fp16 tensor rate, which is twice that of the TF32 format.
 *              Power-of-two scales keep heads and tails inside fp16's range:
 *              pixels by 2^-4, activations by 2^-4, dense-1 weights by the
 *              largest 2^k with max|W1| 2^k <= 2^14, conv weights and bias
 *              (times 2^-4) by the largest 2^k with their largest magnitude
 *              times 2^k <= 2^14.  Interval values and conv activations must
 *              stay below 2^20 in magnitude; beyond that the scores are
 *              undefined. */
typedef enum { EMTK_FP32 = 0, EMTK_TF32 = 1, EMTK_BF16 = 2, EMTK_FP16 = 3, EMTK_FP8 = 4 } emtk_precision;

/* Element type of a patch buffer. */
typedef enum { EMTK_PATCH_F32 = 0, EMTK_PATCH_BF16 = 1, EMTK_PATCH_F16 = 2 } emtk_patch_format;

/* A reconstructed hit: wire index in the plane and raw tick index of its
 * peak time (Sec. 2.1).  The hit's time interval is floor(tick / 6). */
typedef struct {
    int32_t wire;
    int32_t tick;
} emtk_hit;

/* Network weights, host fp32, copied and converted by emtk_create (Sec. 2.2;
 * 11,900,420 values in total):
 *   conv_w [5][5][1][48]  tap row i, tap column j, input channel, filter
 *   conv_b [48]
 *   fc1_w  [92928][128]   row index (y*44 + x)*48 + c: conv map c at (y, x)
 *   fc1_b  [128]
 *   fc2_w  [128][32]   fc2_b [32]
 *   cls_w  [32][3]     cls_b [3]    softmax logits (track, em, none)
 *   mic_w  [32][1]     mic_b [1]    Michel logit */
typedef struct {
    const float *conv_w, *conv_b, *fc1_w, *fc1_b, *fc2_w, *fc2_b, *cls_w, *cls_b, *mic_w, *mic_b;
} emtk_weights;

/* Creation options; emtk_create(w, NULL, ...) uses the defaults in brackets.
 *   precision       [EMTK_BF16]
 *   max_hits        hits processed per internal chunk; sizes the workspace
 *                   [65536]; larger calls are processed in chunks
 *   debug_logits    0: d_scores is [n][4]; 1: d_scores is [n][8], the 4
 *                   scores followed by the 4 logits [0]
 *   wait_timeout_ns limit of every device-side wait in the tensor-core
 *                   kernel, in nanoseconds [2e9]
 *   debug_stall     test knob: 1 makes the tensor-core kernel wait once on
 *                   a barrier nothing arrives at, so the wait runs out and
 *                   the call's emtk_check reports EMTK_ERR_TIMEOUT [0]
 *   profile         1: bracket every kernel launch with CUDA events on the
 *                   caller's stream; emtk_get_stats then reports device time
 *                   per kernel [0] */
typedef struct {
    emtk_precision precision;
    int32_t max_hits;
    int32_t debug_logits;
    int64_t wait_timeout_ns;
    int32_t debug_stall;
    int32_t profile;
} emtk_options;

/* One client request for emtk_infer_batch: a plane and its hits. */
typedef struct {
    const float *d_adc;       /* [nwires][ld] fp32, 16-byte aligned, ld % 4 == 0 */
    int32_t nwires, nticks;
    int64_t ld;
    const emtk_hit *d_hits;   /* [nhits] */
    int32_t nhits;
    float *d_scores;          /* [nhits][4] (or [nhits][8] with debug_logits) */
} emtk_request;

/* Kernel classes of the hot path, for per-kernel timing. */
typedef enum {
    EMTK_KERNEL_INTERVALS = 0, /* plane -> time-interval image */
    EMTK_KERNEL_GATHER = 1,    /* interval image -> 48x48 patches */
    EMTK_KERNEL_NETWORK = 2,   /* conv + dense-1 (tensor cores or fp32) */
    EMTK_KERNEL_HEAD = 3,      /* dense-1 sum + dense-2 + heads */
    EMTK_KERNEL_CONVERT = 4,   /* fp32 patches -> split-fp16 words (emtk_infer_patches, EMTK_TF32) */
    EMTK_KERNEL_HITFIND = 5,   /* hit finding (emtk_find_hits: find, place) */
    EMTK_NUM_KERNELS = 6
} emtk_kernel;

typedef struct {
    /* launches: kernels of this library launched (a tiled patch cut and a
     * hit-finding group are two each); chunks: network launches */
    uint64_t calls, hits, launches, chunks;
    uint64_t batch_hist[8];   /* hits per launch: <256, <1k, <2k, <4k, <8k, <16k, <64k, >=64k */
    /* kernels launched per kernel class and, with options.profile, summed
     * device milliseconds per class (emtk_get_stats waits for the recorded
     * events; a class's time spans all its kernels of one call) */
    uint64_t kernel_launches[EMTK_NUM_KERNELS];
    double kernel_ms[EMTK_NUM_KERNELS];
} emtk_stats;

/* Fills *out with the defaults listed above. */
EMTK_API void emtk_default_options(emtk_options *out);

/* Creates a context on CUDA device `device`: uploads and converts the
 * weights and allocates the workspace.  Returns EMTK_ERR_UNSUPPORTED on a
 * device other than compute capability 10.3 (the library is built for
 * sm_103a only).  *out is NULL on failure. */
EMTK_API emtk_status emtk_create(const emtk_weights *w, const emtk_options *opt, int device, emtk_ctx **out);

/* Frees the context (synchronises its device first).  NULL is accepted. */
EMTK_API emtk_status emtk_destroy(emtk_ctx *ctx);

/* Scores every hit of one plane (Sec. 2.1 + 2.2).
 *   d_adc    [nwires][ld] fp32 deconvolved charge, nticks valid ticks per
 *            row; 16-byte aligned, ld % 4 == 0 and ld >= nticks
 *   d_hits   [nhits]
 *   d_scores [nhits][4] = {p_track, p_em, p_none, p_michel} (fp32)
 * nhits == 0 returns EMTK_OK and enqueues nothing. */
EMTK_API emtk_status emtk_infer(emtk_ctx *ctx, const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld,
                       const emtk_hit *d_hits, int32_t nhits, float *d_scores, emtk_stream stream);

/* Request batching: concatenates the hit lists of `nreq` requests (a host
 * array; each request has its own plane and output) and scores them in one
 * pass of the hot path.  This stands in for the inference server's dynamic
 * batching (Sec. 3.2).  Requests with nhits == 0 are allowed. */
EMTK_API emtk_status emtk_infer_batch(emtk_ctx *ctx, const emtk_request *reqs, int32_t nreq, emtk_stream stream);

/* emtk_infer_batch with HOST buffers: each request's d_adc, d_hits and
 * d_scores point to host memory (the same layouts; pinned memory lets the
 * copies overlap).  The planes and hit lists are copied to one of two device
 * staging areas of the context on its own copy stream, the batch runs on
 * `stream`, and the scores are copied back on `stream`; the call returns
 * once all of it is enqueued.  Consecutive calls use the two areas in turn,
 * so the copy-in of call i+1 overlaps the kernels of call i (the inference
 * server's input transfer, Sec. 3.3, hidden behind the previous batch).
 *   - The hit lists are packed on the host into a pinned buffer of the area
 *     during the call and copied in at once; planes that lie back to back in
 *     host memory are copied in one piece.  The call waits for the copy-in
 *     of the area's previous call (two calls back) before packing.
 *   - The host buffers must stay valid and unchanged until `stream` has
 *     completed the call (cudaStreamSynchronize, or an event recorded on
 *     `stream` after the call), and the scores are final only then.
 *   - A staging area grows to the largest call it has served (a cudaMalloc,
 *     after waiting for that area's previous call).
 *   - ld % 4 == 0 and ld >= nticks, as for emtk_infer_batch; no alignment is
 *     required of the host pointers.
 * Errors as for emtk_infer_batch; EMTK_ERR_OOM if a staging area cannot grow. */
EMTK_API emtk_status emtk_infer_batch_host(emtk_ctx *ctx, const emtk_request *reqs, int32_t nreq,
                                           emtk_stream stream);

/* Patch cut only (Sec. 2.1): d_patches [nhits][48][48] of `fmt`.  F32 is the
 * exact fp32 value; BF16 / F16 are that value rounded to nearest-even. */
EMTK_API emtk_status emtk_extract_patches(emtk_ctx *ctx, const float *d_adc, int32_t nwires, int32_t nticks,
                                 int64_t ld, const emtk_hit *d_hits, int32_t nhits, void *d_patches,
                                 emtk_patch_format fmt, emtk_stream stream);

/* Size of the fixed device array behind emtk_extract_patches_static. */
#define EMTK_STATIC_SCRATCH_BYTES (4u << 20)

/* The patch cut of emtk_extract_patches for callers that cannot allocate
 * device memory.  The paper has no counterpart; it is a service to callers
 * whose device memory is already owned by another allocator (a framework's
 * caching pool, a budget fixed at start-up) or that must avoid the
 * device-wide synchronisation cudaMalloc / cudaFree can cause.  It takes no
 * context (creating one allocates) and calls no allocating routine.
 *   - Same arguments and output as emtk_extract_patches, on the current
 *     device.
 *   - Its scratch is one fixed array of EMTK_STATIC_SCRATCH_BYTES in the
 *     library's static device memory, held by every GPU that loads the
 *     library until the process exits.  The plane's interval image must fit:
 *     nwires * ((nticks/6 rounded up to a multiple of 8)) * (4 for F32, 2 for
 *     BF16/F16) <= EMTK_STATIC_SCRATCH_BYTES, else EMTK_ERR_ARG and nothing is
 *     enqueued (a 960 x 6000 plane fits in every format).
 *   - The first call on each device looks up the array's device address
 *     in the device's current context, and so does the first call after
 *     that context was destroyed and created again (cudaDeviceReset); make
 *     that first call before any stream capture.
 *   - All calls share the array.  Calls that overlap on the GPU (two streams,
 *     two threads) race; serialise them.  Nothing needs clearing between
 *     calls: every interval a call reads, that call wrote. */
EMTK_API emtk_status emtk_extract_patches_static(const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld,
                                                 const emtk_hit *d_hits, int32_t nhits, void *d_patches,
                                                 emtk_patch_format fmt, emtk_stream stream);

/* Network only (Sec. 2.2) on pre-cut fp32 patches [n][48][48] -> d_scores.
 * The 16-bit and fp8 network kernels read the fp32 patches themselves, each
 * value rounded to nearest-even 16 bit as it is loaded; EMTK_TF32 converts
 * them to head/tail words in one launch first.  d_patches 16-byte aligned,
 * d_scores 4-byte aligned; chunks of max_hits patches per launch. */
EMTK_API emtk_status emtk_infer_patches(emtk_ctx *ctx, const float *d_patches, int32_t n, float *d_scores,
                               emtk_stream stream);

/* Synchronises `stream`, then reports (and clears) the context's device
 * status: EMTK_ERR_TIMEOUT if a device-side wait gave up since the last
 * check, EMTK_ERR_CUDA on a sticky CUDA error, else EMTK_OK. */
EMTK_API emtk_status emtk_check(emtk_ctx *ctx, emtk_stream stream);

/* Counters since creation.  In profile mode this first waits for the events
 * of every launch not yet read back. */
EMTK_API emtk_status emtk_get_stats(emtk_ctx *ctx, emtk_stats *out);

/* ---- Hit finding (upstream of the patch cut) ------------------------------
 *
 * Sec. 2.1: the hits that the classifier scores are found on the deconvolved
 * waveform of each wire.  The paper does not give the algorithm; this one
 * takes the plainest reading.  On each wire, a hit is a maximal run of
 * consecutive ticks t < nticks whose value is above the threshold
 * (adc[w][t] > threshold; NaN is never above).  It is placed at the run's
 * largest value (the earliest tick on ties).  A run is one hit even if it
 * holds several local maxima (overlapping pulses are not split). */

/* A found hit's run: first and last tick, the value at the peak tick, and
 * the fp32 sum of the run's values.  The summation order is fixed (the same
 * result on every call): a run within one aligned group of 4 ticks sums in
 * tick order, a longer run adds a pairwise sum per 32-tick step from its
 * start, steps in order; the error stays within the usual fp32 bound of a
 * sum of that length. */
typedef struct {
    int32_t start;
    int32_t end;
    float peak;
    float charge;
} emtk_hit_info;

/* One plane for emtk_find_hits.  d_adc, nwires, nticks and ld are as in
 * emtk_request (d_adc 16-byte aligned, ld % 4 == 0, ld >= nticks).  Outputs
 * are ordered by wire, then tick:
 *   d_hits [capacity]  (wire, peak tick) of each hit: a hit list that
 *                      emtk_infer / emtk_request take as it is;
 *   d_info [capacity]  the run of each hit, or NULL;
 *   n_found            set on return: the number of hits on the plane.  If
 *                      it exceeds capacity, only the first `capacity` hits
 *                      are written. */
typedef struct {
    const float *d_adc;
    int32_t nwires;
    int32_t nticks;
    int64_t ld;
    float threshold;
    int32_t capacity;
    emtk_hit *d_hits;
    emtk_hit_info *d_info;
    int32_t n_found;
    int32_t reserved;
} emtk_hitfind_request;

/* Finds the hits of nreq planes (per group of up to 64 planes: two kernels,
 * find and place; each sample is read once, units with more than 128 runs
 * per 2048 ticks twice).  Returns
 * once the results are complete: it synchronises `stream` to fill each
 * n_found.
 * EMTK_ERR_ARG for negative sizes, ld < nticks, capacity > 0 with a NULL
 * d_hits, a plane holding more than 2^31 - 1 possible runs, or a plane of
 * more 2048-tick wire segments than the workspace's scratch holds (about
 * 104,000, some 214 M samples, for the default workspace); EMTK_ERR_ALIGN
 * as for emtk_infer.  The context's workspace serves as scratch, so calls on
 * one context must not overlap with each other or with its inference calls
 * on another stream. */
EMTK_API emtk_status emtk_find_hits(emtk_ctx *ctx, emtk_hitfind_request *reqs, int32_t nreq, emtk_stream stream);

/* The dense-1 operand scales of an EMTK_FP8 context (see emtk_precision):
 * *s_a = 2^-4 and *s_w; 1 and 1 for every other precision.  Either pointer
 * may be NULL.  EMTK_ERR_ARG for a NULL context. */
EMTK_API emtk_status emtk_get_fp8_scales(const emtk_ctx *ctx, float *s_a, float *s_w);

/* Static English text for a status code. */
EMTK_API const char *emtk_status_string(emtk_status s);

/* ------------------------------------------------------------------------
 * Request batcher: many clients, one GPU.
 *
 * In the paper's setup (Sec. 2.3, 3.2) many CPU processes send inference
 * requests to a server whose dynamic batching merges them into larger
 * batches.  The batcher is that merging step inside one process: client
 * threads submit requests (a plane and its hit list, emtk_request) and wait
 * for their scores; a dispatcher thread forms batches of whole requests and
 * runs each with emtk_infer_batch on one of the batcher's own CUDA streams,
 * each stream with its own workspace (the weights of `ctx` are shared).
 *   - A batch is launched when its requests hold max_hits hits, or when its
 *     oldest request has waited max_delay_us, whichever comes first.  A
 *     request larger than max_hits goes alone.  Requests leave in
 *     submission order.
 *   - The request's buffers (d_adc, d_hits, d_scores) must stay valid and
 *     unchanged until emtk_batcher_wait() has returned for its ticket; they
 *     are read and written on the batcher's streams, not the caller's.
 *   - ctx must outlive the batcher and must not be used from other threads
 *     while the batcher exists; its precision and options apply.
 * -------------------------------------------------------------------- */
typedef struct emtk_batcher emtk_batcher;

/* nstreams in [1, 16]; max_hits > 0; max_delay_us >= 0.  Creates the
 * streams and workspaces (device allocations) and starts the dispatcher and
 * completion threads. */
EMTK_API emtk_status emtk_batcher_create(emtk_ctx *ctx, int32_t nstreams, int32_t max_hits, int64_t max_delay_us,
                                         emtk_batcher **out);

/* Thread-safe, non-blocking: queues one request and returns its ticket (> 0).
 * The request is checked as emtk_infer_batch checks it; an invalid one
 * returns that status and is not queued. */
EMTK_API emtk_status emtk_batcher_submit(emtk_batcher *b, const emtk_request *req, uint64_t *ticket);

/* Thread-safe: blocks until the ticket's scores are complete in device
 * memory, then returns the status of its batch (EMTK_ERR_TIMEOUT if a
 * device-side wait of that batch gave up).  Returns EMTK_ERR_TIMEOUT after
 * timeout_ms (< 0: no limit) without consuming the ticket, and EMTK_ERR_ARG
 * for a ticket that was never issued or was already waited for. */
EMTK_API emtk_status emtk_batcher_wait(emtk_batcher *b, uint64_t ticket, int64_t timeout_ms);

/* Counters since creation: batches launched, requests and hits in them. */
EMTK_API emtk_status emtk_batcher_stats(emtk_batcher *b, int64_t *batches, int64_t *requests, int64_t *hits);

/* Launches what is still queued, waits for every batch, stops the threads
 * and frees the batcher's streams and workspaces.  NULL is allowed.  Tickets
 * not yet waited for are dropped. */
EMTK_API emtk_status emtk_batcher_destroy(emtk_batcher *b);

/* ------------------------------------------------------------------------
 * Test hooks: host-side fault injection.  They make the failures a service
 * must survive (an exhausted device, a dispatcher that stops making progress)
 * happen on the host, with no fault on the GPU.  Not for production use.
 * -------------------------------------------------------------------- */

/* Arms an allocation failure: `after` more device or pinned-host
 * allocations of the library succeed, then the next one fails, once, as if
 * the memory were exhausted (the entry point that made it returns
 * EMTK_ERR_OOM and frees what it had allocated for that call).  after < 0
 * disarms.  Process-wide; every allocation of every context counts. */
EMTK_API void emtk_debug_fail_alloc(int64_t after);

/* Number of device and pinned-host allocations of the library alive now
 * (weights, workspaces, staging areas, batcher state).  Either pointer may be
 * NULL. */
EMTK_API void emtk_debug_alloc_counts(int64_t *device, int64_t *host);

/* stall = 1: the batcher's dispatcher launches nothing until it is called
 * again with stall = 0 (requests stay queued; emtk_batcher_wait with a
 * timeout returns EMTK_ERR_TIMEOUT and keeps the ticket).
 * emtk_batcher_destroy launches what is queued even while stalled.
 * EMTK_ERR_ARG for a NULL batcher or another value of stall. */
EMTK_API emtk_status emtk_debug_batcher_stall(emtk_batcher *b, int32_t stall);

#ifdef __cplusplus
}
#endif
#endif /* EMTK_H */
