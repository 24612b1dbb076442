// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "../../include/emtk.h"

namespace emtk {

// Geometry of the method (Sec. 2.1, Sec. 2.2).
constexpr int kPatch = 48;                           // patch side
constexpr int kDs = 6;                               // ticks per time interval
constexpr int kHalf = kPatch / 2;                    // hit sits at row/col 24
constexpr int kK = 5;                                // conv kernel side
constexpr int kF = 48;                               // conv filters
constexpr int kQ = kPatch - kK + 1;                  // 44
constexpr int kPos = kQ * kQ;                        // 1936 conv positions
constexpr int kFc1In = kPos * kF;                    // 92,928
constexpr int kN1 = 128;
constexpr int kN2 = 32;
constexpr int kNC = 3;
constexpr int kPatchElems = kPatch * kPatch;         // 2304
constexpr int kQuads = kPos / 4;                     // 484 quads of 4 conv positions

// Stream-K split of the tensor-core network: the launch's work is the units
// u = tile * kQuads + quad (tile = 128 hits); CTA c of G takes the contiguous
// units [unit_begin(c), unit_begin(c + 1)).  A tile's dense-1 partial sums
// come from CTAs cta_of_unit(first unit) .. cta_of_unit(last unit), written
// to partial rows 0, 1, ... in that order.
__host__ __device__ inline int64_t unit_begin(int c, int64_t units, int G) { return (int64_t)c * units / G; }
__host__ __device__ inline int cta_of_unit(int64_t u, int64_t units, int G) {
    int c = (int)((u * G) / units);
    while (c > 0 && unit_begin(c, units, G) > u) --c;
    while (c + 1 < G && unit_begin(c + 1, units, G) <= u) ++c;
    return c;
}

// Requests handled by one extraction launch (kernel-parameter table).
constexpr int kMaxReqPerLaunch = 64;

struct ReqDesc {
    const float *adc;
    const emtk_hit *hits;
    float *scores;        // output rows of this request
    int64_t ld;
    int64_t hit_begin;    // first index of this request in the concatenated hit list
    int64_t d_off;        // element offset of its interval image in the workspace
    int32_t nwires;
    int32_t nticks;
    int32_t nhits;
    int32_t nint;         // complete time intervals: nticks / 6
    int32_t pitch;        // row pitch of the interval image (a multiple of 8 elements)
    int32_t halo;         // zero border of the image: element (w, b) is at
                          // d_off + (w + halo) * pitch + (b + halo); rows nwires + 2 halo
    int32_t m_wpb;        // tile mask (launch_cut_tiles): 32-bit words per band of kTileRows rows
    int64_t m_off;        // the request's first mask word
};

// Tiles of an interval image for the cut that skips what no window reads: a
// tile is kTileRows image rows x kTileInts intervals; tile (band, c) of a
// request is bit c % 32 of mask word m_off + band * m_wpb + c / 32.
constexpr int kTileRows = 8;
constexpr int kTileInts = 16;  // 96 ticks: 384-byte pieces of an fp32 row (8 measured slower, 32 read 5% more)
static_assert(2 * kHalf / kTileInts + 1 <= 32, "a window's tile columns fit two mask words");

// Where the tensor-core kernel finds a hit's 48 x 48 window: element (r, c)
// is src[origin + r * pitch + c] when `inside` (the whole window lies in the
// haloed image); otherwise it is the image pixel (wc - 24 + r, bc - 24 + c)
// of the plane at d_off, zero outside [0, nwires) x [0, nint).
struct HitDesc {
    int64_t origin;
    int64_t d_off;
    int32_t pitch;
    int32_t inside;
    int32_t wc, bc;
    int32_t nwires, nint;
};
constexpr int kHalo = kHalf;    // image border for the tensor-core path

struct ReqTable {
    int32_t n;
    int32_t pad;
    ReqDesc r[kMaxReqPerLaunch];
};

// Planes of one hit-finding launch group (emtk_find_hits).  The unit of work
// is a wire segment of kSegTicks ticks; a plane has nwires * nseg units, and
// unit0 is its first unit in the group's concatenated unit list.
constexpr int kMaxHfPlanes = 64;
constexpr int kSegTicks = 2048;
struct HfDesc {
    const float *adc;
    emtk_hit *hits;
    emtk_hit_info *info;
    int64_t ld;
    int64_t unit0;
    int64_t chunk0;  // the plane's first chunk of units (set by launch_find_hits)
    int32_t nticks;
    int32_t nseg;
    int32_t capacity;
    float thr;
};
struct HfTable {
    int32_t n;
    int32_t pad;
    HfDesc r[kMaxHfPlanes];
};

// Per-context workspace (device).
struct Workspace {
    void *dimg = nullptr;        // interval images of the planes of one launch
    size_t dimg_bytes = 0;
    void *patches = nullptr;     // [max_hits][48][48] in the precision's patch format
    HitDesc *hdesc = nullptr;    // [max_hits] window descriptors (tensor-core path)
    float **dest = nullptr;      // [max_hits] output row of each hit
    float *partials = nullptr;   // [max_splits][max_hits_pad][128]
    size_t partial_elems = 0;
    int *status = nullptr;       // device status word (bit 0: a network wait gave up, bit 1: a head wait)
    int *tile_done = nullptr;    // [max_hits / 128 + 1] per tile: epilogue warps whose partial rows are stored
};

struct DeviceWeights {
    float *conv_w = nullptr;     // [25][48] fp32
    float *conv_b = nullptr;     // [48]
    float *fc1_w = nullptr;      // [92928][128] fp32 (fp32 path only)
    float *fc1_b = nullptr;      // [128]
    float *fc2_w = nullptr;      // [128][32]
    float *fc2_b = nullptr;
    float *cls_w = nullptr;      // [32][3]
    float *cls_b = nullptr;
    float *mic_w = nullptr;      // [32]
    float *mic_b = nullptr;
    void *w1_tiles = nullptr;      // dense-1 weights, tiled for TMA: [1452][128][64] of 16 bit or e4m3
                                   // (EMTK_TF32: fp16 heads, then fp16 tails, each so tiled)
    uint16_t *convB = nullptr;     // 16-bit conv B operand: [48][32] (taps 0-24, bias hi, bias lo, zeros)
    void *w1_tmap = nullptr;       // host copies of the TMA descriptors (CUtensorMap[1], or [2]: heads, tails)
    float fc1_scale = 1.0f;        // dense-1 sums are scaled by this before the bias (EMTK_FP8: 1/(s_a s_w))
    float fc1_w_scale = 1.0f;      // EMTK_FP8 / EMTK_TF32: s_w, the power of two the weights were scaled by
    float act_mul = 1.0f;          // EMTK_TF32: s_a / (s_p s_c), applied to the ReLU'd conv sums
    // host copy of the conv weights [25][48] and bias [48]: the fp32 kernel takes
    // them as a launch parameter (constant bank)
    float conv_w_host[kK * kK * kF] = {};
    float conv_b_host[kF] = {};
};

// Operand formats of the tensor-core kernels: 16-bit (cnn_tc.cu, also with
// an e4m3 dense-1), and fp32 operands split into fp16 heads and tails
// (cnn_split.cu, EMTK_TF32).
enum TcMode { kTcBf16 = 0, kTcFp16 = 1, kTcFp8 = 2, kTcSplit = 3 };

// Internal patch / interval-image format of EMTK_TF32: one 32-bit word per
// pixel, the fp16 head of (value x kSplitPatchScale) in the low half and the
// fp16 tail (the rest, rounded to fp16) in the high half.  Not a format of
// the public emtk_patch_format.
constexpr emtk_patch_format kPatchSplit16 = static_cast<emtk_patch_format>(3);
constexpr float kSplitPatchScale = 0.0625f;  // s_p: 2^-4

// Programmatic dependent launch.  A kernel launched with launch_pdl may
// start before the kernel before it on the stream has completed (once every
// CTA of that one has started and executed pdl_trigger, or finished), so its
// set-up overlaps that kernel's tail; before it reads anything that kernel
// (or an earlier one) wrote, it executes pdl_wait, which returns once the
// previous kernel has completed and its writes are visible.
#ifdef __CUDACC__
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
#endif

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

}  // namespace emtk

struct emtk_pending_event {
    int kind;
    cudaEvent_t start, stop;
};

struct emtk_ctx {
    int device = 0;
    std::vector<emtk_pending_event> pending;  // profile mode: launches not yet read back
    emtk_options opt{};
    int max_hits = 0;
    int max_splits = 0;
    int sm_count = 0;
    emtk::DeviceWeights w;
    emtk::Workspace ws;
    emtk_stats stats{};
    bool owns_weights = true;  // false for a batcher lane, which shares its parent's weights
    // emtk_infer_batch_host: two device staging areas used alternately, filled on
    // the context's copy stream; compute_done[k] marks the end of the last call
    // that used area k (its scores copied out), copy_done[k] the end of its copy.
    struct HostStage {
        void *buf = nullptr;
        size_t bytes = 0;
        void *hits_host = nullptr;  // pinned: the call's hit lists packed, copied in at once
        size_t hits_host_bytes = 0;
        cudaEvent_t copy_done = nullptr, compute_done = nullptr;
        bool used = false;
    } stage[2];
    cudaStream_t copy_stream = nullptr;
    uint64_t host_calls = 0;
    int32_t *h_totals = nullptr;  // pinned: emtk_find_hits' per-plane counts (kMaxHfPlanes)
    // emtk_find_hits' chunk sums: two halves of hf_sums_cap, used in turn; each
    // launch clears the other half for the next one
    int32_t *hf_sums = nullptr;
    int64_t hf_sums_cap = 0;
    int hf_parity = 0;
    // tiles of the interval images that the hits' windows touch: two zeroed
    // halves of tile_mask_cap words, used in turn; each tile kernel clears
    // the other half for the next launch
    uint32_t *tile_mask = nullptr;
    int64_t tile_mask_cap = 0;
    int tile_mask_parity = 0;
};

namespace emtk {

// ---- allocations (alloc.cu): every device and pinned-host allocation of the
// library, counted; emtk_debug_fail_alloc can make one of them fail.  *p is
// null after a failure; freeing null is a no-op.
cudaError_t dev_alloc(void **p, size_t bytes);
cudaError_t dev_free(void *p);
cudaError_t host_alloc(void **p, size_t bytes);
cudaError_t host_free(void *p);

// ---- host helpers shared by the API and the request batcher (api.cu)
// The checks emtk_infer_batch applies to one request.
emtk_status validate_request(const emtk_request &q);
// A context for one batcher stream: the parent's weights and options, its own
// workspace.  nullptr (and *st set) on failure.
emtk_ctx *make_lane_ctx(const emtk_ctx *parent, emtk_status *st);
void destroy_lane_ctx(emtk_ctx *c);

// ---- kernels launched from the API (each returns cudaGetLastError()).
// Interval images of every request plane: img[r] is [nwires][nint] of the
// patch format (fp32 or 16-bit), at element offset r.d_off.
// Window descriptors to build along with the images (tensor-core path): hits
// g0 .. g0 + count - 1 of the table into desc[0 ..] and dest[0 ..].
struct DescJob {
    int64_t g0;
    int32_t count;
    HitDesc *desc;
    float **dest;
    int out_stride;
};
cudaError_t launch_interval_images(const ReqTable &t, void *dimg, emtk_patch_format fmt, cudaStream_t s,
                                   const DescJob *job = nullptr);
// The haloed interval images of the table's requests (16-bit, or the split
// fp16 head / tail words of EMTK_TF32), only the tiles
// that some hit's window touches (two launches: the hits mark their tiles in
// mask_cur and the first chunk's window descriptors are built; then one warp
// per tile computes the covered ones, and mask_next, mask_cap words, is
// cleared).  Tiles no window touches keep whatever they held: the window
// reads take their bits only as padding they shift out.  total_hits = all
// hits of the table.
cudaError_t launch_cut_tiles(const ReqTable &t, int64_t total_hits, void *dimg, emtk_patch_format fmt,
                             const DescJob &job, uint32_t *mask_cur, uint32_t *mask_next, int64_t mask_cap,
                             cudaStream_t s);
// Patches of hits [g0, g0+count) of the concatenated list (global index).
// Writes patches[(g - g0)] and, if dest != null, dest[g - g0] = output row.
cudaError_t launch_gather(const ReqTable &t, const void *dimg, emtk_patch_format fmt, int64_t g0,
                          int32_t count, void *patches, float **dest, int out_stride, cudaStream_t s);
// Pre-cut fp32 patches (n values, a multiple of 8, 16-byte aligned) into the
// split-fp16 head / tail words of the EMTK_TF32 network at dst (n words), in
// one launch of at most 8 CTAs per SM.
cudaError_t launch_convert_split(const float *src, void *dst, int64_t n, int sms, cudaStream_t s);
// Window descriptors of hits [g0, g0+count) (images with halo kHalo), and
// the output row of each hit in dest.
cudaError_t launch_hit_desc(const ReqTable &t, int64_t g0, int32_t count, HitDesc *desc, float **dest,
                            int out_stride, cudaStream_t s);
// Hit finding of the group's planes (hitfind.cu): scratch (256-byte aligned)
// holds per-unit run counts and run slots; find_hits_unit_cap gives the most
// units that scratch_bytes holds.  The chunk sums live in sums_cur (zero on
// entry, find_hits_chunks(t, U) of them); the launch zeroes sums_next[0, cap)
// for the next launch.  totals[r] receives plane r's hit count.
int64_t find_hits_unit_cap(size_t scratch_bytes);
int64_t find_hits_chunks(const HfTable &t, int64_t nunits);
cudaError_t launch_find_hits(const HfTable &t, int64_t nunits, void *scratch, int32_t *sums_cur, int32_t *sums_next,
                             int64_t cap, int32_t *totals, cudaStream_t s);

// Network: dense-1 partial sums [splits][n_pad][128] from patches.
cudaError_t launch_cnn_fp32(const DeviceWeights &w, const float *patches, int32_t n, int splits,
                            float *partials, int n_pad, cudaStream_t s);
// Stream-K over G CTAs (one per SM); partials [rows][n_pad][128] with rows
// = streamk_partial_rows(n, G).
// src: 16-bit patches [n][48][48] (desc == nullptr) or the haloed interval
// images of the hits' planes, located through desc.
// tile_done (or null): each epilogue warp adds 1 to tile_done[tile] once its
// partial rows of the tile are in memory (a tile is complete at 4 x its
// partial rows).
// src32 (or null; 16-bit and fp8 modes, desc == nullptr): pre-cut fp32
// patches [n][48][48] that the kernel reads itself, rounding each value as the
// patch conversion does.
cudaError_t launch_cnn_tc(const DeviceWeights &w, const void *src, const HitDesc *desc, TcMode mode, int32_t n,
                          int G, float *partials, int n_pad, int *status, int64_t timeout_ns, int debug_stall,
                          int *tile_done, const float *src32, cudaStream_t s);
// Where the head writes hit h's scores: dest[h], or rows + h * stride when
// rows is not null (pre-cut patches, whose rows are consecutive).
struct OutRows {
    float *const *dest;
    float *rows;
    int stride;
};
int streamk_partial_rows(int32_t n, int G);
// Sum of partials + bias + ReLU, dense-2, heads; hit h's scores where out_rows says.  Partial
// rows: `splits` per hit (G == 0), or the stream-K contributors of the hit's
// tile (G > 0).  With tile_done (stream-K launches for which
// head_counts_tiles(n, G) holds), a tile's head starts once the tile's
// counter is complete instead of after the whole network kernel, gives up
// when bit 0 of *status is set or after timeout_ns (setting bit 1), and
// sets the counter back to zero.
bool head_counts_tiles(int32_t n, int G);
cudaError_t launch_head(const DeviceWeights &w, const float *partials, int splits, int G, int n_pad,
                        int32_t n, OutRows out_rows, int debug_logits, int *tile_done, int *status,
                        int64_t timeout_ns, cudaStream_t s);

// Kernel attributes (dynamic shared memory), set once per device at create.
cudaError_t init_fp32_kernel_attrs();
cudaError_t init_head_kernel_attrs();
cudaError_t init_tc_kernel_attrs();

// Host helpers for the tensor-core weights (cnn_tc.cu, cnn_split.cu).
cudaError_t prepare_tc_weights(DeviceWeights &w, const emtk_weights &hw, TcMode mode);
cudaError_t prepare_split_weights(DeviceWeights &w, const emtk_weights &hw);
cudaError_t init_split_kernel_attrs();
cudaError_t launch_cnn_split(const DeviceWeights &w, const void *src, const HitDesc *desc, int32_t n, int G,
                             float *partials, int n_pad, int *status, int64_t timeout_ns, int debug_stall,
                             int *tile_done, cudaStream_t s);
// EMTK_FP8 weight scale: the largest power of two s_w with max|W1| s_w <= 448.
double fp8_weight_scale(const float *fc1_w, size_t n);
int choose_splits_fp32(int n, int sm_count, int max_splits);

}  // namespace emtk
