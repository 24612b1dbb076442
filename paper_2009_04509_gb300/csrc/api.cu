// C ABI of the library (include/emtk.h): argument checks, workspace, the
// hot-path sequence and counters.  Every launch goes to the caller's stream.
#include <cuda.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <new>

#include "emtk_internal.h"

using namespace emtk;

namespace {

struct DeviceGuard {  // restores the caller's current device
    int prev = -1;
    bool ok = false;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

bool tensor_precision(emtk_precision p) {
    return p == EMTK_BF16 || p == EMTK_FP16 || p == EMTK_FP8 || p == EMTK_TF32;
}

TcMode tc_mode(emtk_precision p) {
    return p == EMTK_FP16 ? kTcFp16 : p == EMTK_FP8 ? kTcFp8 : p == EMTK_TF32 ? kTcSplit : kTcBf16;
}

// EMTK_FP8 keeps the conv in bf16, so its patches are bf16; EMTK_TF32 uses
// fp16 head + tail words
emtk_patch_format patch_format(emtk_precision p) {
    return (p == EMTK_BF16 || p == EMTK_FP8) ? EMTK_PATCH_BF16
           : p == EMTK_FP16                  ? EMTK_PATCH_F16
           : p == EMTK_TF32                  ? kPatchSplit16
                                             : EMTK_PATCH_F32;
}

size_t patch_elem_bytes(emtk_patch_format f) { return (f == EMTK_PATCH_F32 || f == kPatchSplit16) ? 4 : 2; }

int out_stride(const emtk_ctx *c) { return c->opt.debug_logits ? 8 : 4; }

int n_pad_of(int n) { return (n + 127) / 128 * 128; }

constexpr int64_t kPartialCap = 64ll * 1024 * 1024;  // floats of the partial-sum workspace

template <typename T>
cudaError_t dmalloc(T **p, size_t bytes) {
    void *v = nullptr;
    cudaError_t e = dev_alloc(&v, bytes);
    *p = static_cast<T *>(v);
    return e;
}

template <typename T>
cudaError_t upload(T **p, const float *src, size_t n) {
    cudaError_t e = dmalloc(p, n * sizeof(float));
    if (e != cudaSuccess) return e;
    return cudaMemcpy(*p, src, n * sizeof(float), cudaMemcpyHostToDevice);
}

void drain_events(emtk_ctx *c);

void free_ctx(emtk_ctx *c) {
    if (!c) return;
    drain_events(c);
    DeviceWeights &w = c->w;
    if (c->owns_weights) {
        for (void *p : {(void *)w.conv_w, (void *)w.conv_b, (void *)w.fc1_w, (void *)w.fc1_b, (void *)w.fc2_w,
                        (void *)w.fc2_b, (void *)w.cls_w, (void *)w.cls_b, (void *)w.mic_w, (void *)w.mic_b,
                        (void *)w.w1_tiles, (void *)w.convB})
            dev_free(p);
        delete[] static_cast<CUtensorMap *>(w.w1_tmap);
    }
    for (void *p : {c->ws.dimg, c->ws.patches, (void *)c->ws.dest, (void *)c->ws.partials, (void *)c->ws.status,
                    (void *)c->ws.hdesc, (void *)c->ws.tile_done})
        dev_free(p);
    if (c->copy_stream) {
        cudaStreamSynchronize(c->copy_stream);
        cudaStreamDestroy(c->copy_stream);
    }
    host_free(c->h_totals);
    dev_free(c->hf_sums);
    dev_free(c->tile_mask);
    for (auto &st : c->stage) {
        if (st.compute_done) cudaEventSynchronize(st.compute_done);
        dev_free(st.buf);
        host_free(st.hits_host);
        if (st.copy_done) cudaEventDestroy(st.copy_done);
        if (st.compute_done) cudaEventDestroy(st.compute_done);
    }
    delete c;
}

emtk_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return EMTK_OK;
    if (e == cudaErrorMemoryAllocation) return EMTK_ERR_OOM;
    return EMTK_ERR_CUDA;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

emtk_status check_plane(const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld, const emtk_hit *d_hits,
                        int32_t nhits) {
    if (nwires < 0 || nticks < 0 || nhits < 0 || ld < nticks) return EMTK_ERR_ARG;
    if (nhits > 0 && (d_hits == nullptr || d_adc == nullptr)) return EMTK_ERR_ARG;
    if (d_adc != nullptr && (!aligned16(d_adc) || (ld % 4) != 0)) return EMTK_ERR_ALIGN;
    if ((reinterpret_cast<uintptr_t>(d_hits) & 7u) != 0) return EMTK_ERR_ALIGN;
    return EMTK_OK;
}

// Names of the kernel classes in NVTX ranges (a profiler's timeline).
const char *const kNvtxNames[EMTK_NUM_KERNELS] = {"emtk interval images (patch cut)", "emtk gather / descriptors",
                                                  "emtk network (conv + dense-1)", "emtk head (dense-2 + heads)",
                                                  "emtk convert patches", "emtk hit finding"};

// Around the launch of `kernels` kernels of one class: an NVTX range on the
// host thread (always; free unless a profiler is attached), the launch counts
// and, in profile mode, CUDA events on the caller's stream.
struct Prof {
    emtk_ctx *c;
    int kind;
    cudaStream_t s;
    cudaEvent_t a = nullptr, b = nullptr;
    Prof(emtk_ctx *c_, int kind_, cudaStream_t s_, int kernels = 1) : c(c_), kind(kind_), s(s_) {
        nvtxRangePushA(kNvtxNames[kind]);
        c->stats.launches += (uint64_t)kernels;
        c->stats.kernel_launches[kind] += (uint64_t)kernels;
        if (!c->opt.profile) return;
        if (cudaEventCreate(&a) != cudaSuccess || cudaEventCreate(&b) != cudaSuccess) {
            if (a) cudaEventDestroy(a);
            a = b = nullptr;
            return;
        }
        cudaEventRecord(a, s);
    }
    ~Prof() {
        if (a) {
            cudaEventRecord(b, s);
            c->pending.push_back({kind, a, b});
        }
        nvtxRangePop();
    }
};

void drain_events(emtk_ctx *c) {
    for (auto &p : c->pending) {
        float ms = 0.f;
        if (cudaEventSynchronize(p.stop) == cudaSuccess && cudaEventElapsedTime(&ms, p.start, p.stop) == cudaSuccess)
            c->stats.kernel_ms[p.kind] += ms;
        cudaEventDestroy(p.start);
        cudaEventDestroy(p.stop);
    }
    c->pending.clear();
}

void count_launch(emtk_ctx *c, int n) {
    static const int edges[7] = {256, 1024, 2048, 4096, 8192, 16384, 65536};
    int b = 0;
    while (b < 7 && n >= edges[b]) ++b;
    c->stats.batch_hist[b]++;
    c->stats.chunks++;
}

// Interval-image workspace large enough for the requests of one table.
emtk_status ensure_dimg(emtk_ctx *c, size_t bytes, cudaStream_t s) {
    if (bytes <= c->ws.dimg_bytes) return EMTK_OK;
    // earlier work on this stream may still read the old buffer
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_status(e);
    e = dev_free(c->ws.dimg);
    c->ws.dimg = nullptr;
    c->ws.dimg_bytes = 0;
    if (e != cudaSuccess) return cuda_status(e);
    const size_t want = bytes + bytes / 4;
    e = dev_alloc(&c->ws.dimg, want);
    if (e != cudaSuccess) return cuda_status(e);
    c->ws.dimg_bytes = want;
    return EMTK_OK;
}

// Network on `n` patches already in the workspace format -> scores via dest.
// `desc` (tensor-core path only) locates each hit's window in the haloed
// interval images at `patches`; without it `patches` holds the patches.
emtk_status run_network(emtk_ctx *c, const void *patches, const HitDesc *desc, int32_t n, OutRows out_rows,
                        const float *src32, cudaStream_t s) {
    if (n <= 0) return EMTK_OK;
    const int n_pad = n_pad_of(n);
    const int max_splits = (int)std::max<int64_t>(1, kPartialCap / ((int64_t)n_pad * kN1));
    cudaError_t e;
    int splits = 0, G = 0;
    int *tile_done = nullptr;
    if (tensor_precision(c->opt.precision)) {
        // one persistent CTA per SM (stream-K), fewer if the partial rows would not fit
        G = c->sm_count;
        while (G > 1 && streamk_partial_rows(n, G) > max_splits) G /= 2;
        // the head of a large launch takes each tile as soon as its partial rows are stored
        if (head_counts_tiles(n, G)) tile_done = c->ws.tile_done;
        Prof prof(c, EMTK_KERNEL_NETWORK, s);
        e = launch_cnn_tc(c->w, patches, desc, tc_mode(c->opt.precision), n, G, c->ws.partials, n_pad,
                          c->ws.status, c->opt.wait_timeout_ns, c->opt.debug_stall, tile_done, src32, s);
    } else {
        splits = choose_splits_fp32(n, c->sm_count, max_splits);
        Prof prof(c, EMTK_KERNEL_NETWORK, s);
        e = launch_cnn_fp32(c->w, static_cast<const float *>(patches), n, splits, c->ws.partials, n_pad, s);
    }
    if (e != cudaSuccess) return cuda_status(e);
    {
        Prof prof(c, EMTK_KERNEL_HEAD, s);
        e = launch_head(c->w, c->ws.partials, splits, G, n_pad, n, out_rows, c->opt.debug_logits, tile_done,
                        c->ws.status, c->opt.wait_timeout_ns, s);
    }
    count_launch(c, n);
    return cuda_status(e);
}

// Fills a table from requests [r0, r1); returns total hits and image bytes.
void build_table(const emtk_ctx *c, const emtk_request *reqs, int r0, int r1, emtk_patch_format fmt, int halo,
                 ReqTable &t, int64_t &hits, size_t &img_bytes) {
    std::memset(&t, 0, sizeof(t));
    t.n = r1 - r0;
    hits = 0;
    int64_t elems = 0;
    for (int i = 0; i < t.n; ++i) {
        const emtk_request &q = reqs[r0 + i];
        ReqDesc &d = t.r[i];
        d.adc = q.d_adc;
        d.hits = q.d_hits;
        d.scores = q.d_scores;
        d.ld = q.ld;
        d.nwires = q.nwires;
        d.nticks = q.nticks;
        d.nhits = q.nhits;
        d.nint = q.nticks / kDs;
        d.pitch = (d.nint + 2 * halo + 7) / 8 * 8;
        d.halo = halo;
        d.hit_begin = hits;
        d.d_off = elems;
        hits += q.nhits;
        elems += (int64_t)(d.nwires + 2 * halo) * d.pitch;
    }
    // 64 bytes of slack: window rows are read with aligned 16-byte loads
    img_bytes = (size_t)elems * patch_elem_bytes(fmt) + 64;
    (void)c;
}

// Plane bytes (requests with hits) from which a launch cuts only the tiles its
// windows touch: a 256-hit call on one 11.5 MB plane took 30.8 us that way
// against 28.8 us reading the whole plane; the 368.6 MB event 52.3 against 69.6.
constexpr int64_t kTiledCutMinBytes = (int64_t)96 << 20;

// Tile-mask geometry of the table's images (bands of kTileRows rows, words of
// 32 tiles of kTileInts intervals); returns the words of the whole table.
int64_t assign_tile_masks(ReqTable &t) {
    int64_t words = 0;
    for (int i = 0; i < t.n; ++i) {
        ReqDesc &d = t.r[i];
        const int64_t rows = d.nwires > 0 ? (int64_t)d.nwires + 2 * d.halo : 0;
        const int64_t bands = (rows + kTileRows - 1) / kTileRows;
        const int64_t chunks = ((int64_t)d.pitch + kTileInts - 1) / kTileInts;
        d.m_wpb = (int32_t)((chunks + 31) / 32);
        d.m_off = words;
        words += bands * d.m_wpb;
    }
    return words;
}

// Two zeroed halves of at least `words` mask words each (context field tile_mask).
emtk_status ensure_tile_masks(emtk_ctx *c, int64_t words, cudaStream_t s) {
    if (words <= c->tile_mask_cap) return EMTK_OK;
    cudaError_t e = cudaStreamSynchronize(s);  // earlier launches may still use the old halves
    if (e == cudaSuccess) e = dev_free(c->tile_mask);
    c->tile_mask = nullptr;
    c->tile_mask_cap = 0;
    const int64_t cap = words + words / 4 + 64;
    if (e == cudaSuccess) e = dmalloc(&c->tile_mask, 2 * cap * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaMemsetAsync(c->tile_mask, 0, 2 * cap * sizeof(uint32_t), s);
    if (e != cudaSuccess) return cuda_status(e);
    c->tile_mask_cap = cap;
    c->tile_mask_parity = 0;
    return EMTK_OK;
}

emtk_status run_requests(emtk_ctx *c, const emtk_request *reqs, int32_t nreq, cudaStream_t s) {
    const emtk_patch_format fmt = patch_format(c->opt.precision);
    ReqTable *t = new (std::nothrow) ReqTable;
    if (!t) return EMTK_ERR_OOM;
    emtk_status st = EMTK_OK;
    for (int r0 = 0; r0 < nreq && st == EMTK_OK; r0 += kMaxReqPerLaunch) {
        const int r1 = std::min<int>(nreq, r0 + kMaxReqPerLaunch);
        int64_t hits;
        size_t img_bytes;
        const bool tc = tensor_precision(c->opt.precision);
        build_table(c, reqs, r0, r1, fmt, tc ? kHalo : 0, *t, hits, img_bytes);
        if (hits == 0) continue;
        // planes of requests without hits need no interval image
        for (int i = 0; i < t->n; ++i)
            if (t->r[i].nhits == 0) t->r[i].nwires = 0;
        st = ensure_dimg(c, img_bytes, s);
        if (st != EMTK_OK) break;
        // images for the tensor-core kernels: only the tiles some window touches, where
        // the planes are large enough that the bytes skipped (about a third on dense
        // events) outweigh the marking kernel's launch (a few microseconds)
        int64_t plane_bytes = 0;
        for (int i = 0; i < t->n; ++i) plane_bytes += (int64_t)t->r[i].nwires * t->r[i].ld * (int64_t)sizeof(float);
        const bool tiles = tc && plane_bytes >= kTiledCutMinBytes &&
                           (fmt == EMTK_PATCH_BF16 || fmt == EMTK_PATCH_F16 || fmt == kPatchSplit16);
        const int64_t mask_words = tiles ? assign_tile_masks(*t) : 0;
        if (tiles) {
            st = ensure_tile_masks(c, mask_words, s);
            if (st != EMTK_OK) break;
        }
        cudaError_t e;
        {
            // the tensor-core kernel reads the windows straight from the images; the
            // first chunk's window descriptors are built in the same launch
            const DescJob job{0, (int32_t)std::min<int64_t>(c->max_hits, hits), c->ws.hdesc, c->ws.dest,
                              out_stride(c)};
            Prof prof(c, EMTK_KERNEL_INTERVALS, s, tiles ? 2 : 1);  // the tiled cut: marks, then tiles
            if (tiles) {
                uint32_t *cur = c->tile_mask + (int64_t)c->tile_mask_parity * c->tile_mask_cap;
                uint32_t *next = c->tile_mask + (int64_t)(1 - c->tile_mask_parity) * c->tile_mask_cap;
                e = launch_cut_tiles(*t, hits, c->ws.dimg, fmt, job, cur, next, c->tile_mask_cap, s);
                if (e == cudaSuccess)
                    c->tile_mask_parity ^= 1;
                else
                    c->tile_mask_cap = 0;  // the next call reallocates and zeroes both halves
            } else {
                e = launch_interval_images(*t, c->ws.dimg, fmt, s, tc ? &job : nullptr);
            }
        }
        if (e != cudaSuccess) {
            st = cuda_status(e);
            break;
        }
        for (int64_t g0 = 0; g0 < hits && st == EMTK_OK; g0 += c->max_hits) {
            const int32_t cnt = (int32_t)std::min<int64_t>(c->max_hits, hits - g0);
            if (tc && g0 > 0) {
                Prof prof(c, EMTK_KERNEL_GATHER, s);
                e = launch_hit_desc(*t, g0, cnt, c->ws.hdesc, c->ws.dest, out_stride(c), s);
            } else if (!tc) {
                Prof prof(c, EMTK_KERNEL_GATHER, s);
                e = launch_gather(*t, c->ws.dimg, fmt, g0, cnt, c->ws.patches, c->ws.dest, out_stride(c), s);
            }
            if (e != cudaSuccess) {
                st = cuda_status(e);
                break;
            }
            const OutRows out{c->ws.dest, nullptr, 0};
            st = tc ? run_network(c, c->ws.dimg, c->ws.hdesc, cnt, out, nullptr, s)
                    : run_network(c, c->ws.patches, nullptr, cnt, out, nullptr, s);
        }
        c->stats.hits += hits;
    }
    delete t;
    return st;
}

// Workspace of a context, sized by its max_hits.  The patch buffer is only
// needed by the fp32 path and emtk_infer_patches (`patches`).
cudaError_t alloc_workspace(emtk_ctx *c, bool patches) {
    const emtk_options &o = c->opt;
    const emtk_patch_format fmt = patch_format(o.precision);
    cudaError_t e = cudaSuccess;
    // the 16-bit and fp8 tensor-core kernels read pre-cut fp32 patches themselves
    if ((patches && fmt == kPatchSplit16) || !tensor_precision(o.precision))
        e = dmalloc(&c->ws.patches, (size_t)o.max_hits * kPatchElems * patch_elem_bytes(fmt));
    if (e == cudaSuccess) e = dmalloc(&c->ws.dest, (size_t)o.max_hits * sizeof(float *));
    if (e == cudaSuccess && tensor_precision(o.precision))
        e = dmalloc(&c->ws.hdesc, (size_t)o.max_hits * sizeof(HitDesc));
    if (e == cudaSuccess) {
        c->ws.partial_elems = (size_t)std::max<int64_t>(kPartialCap, (int64_t)n_pad_of(o.max_hits) * kN1);
        e = dmalloc(&c->ws.partials, c->ws.partial_elems * sizeof(float));
    }
    if (e == cudaSuccess) e = dmalloc(&c->ws.status, sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(c->ws.status, 0, sizeof(int));
    const size_t ntiles = (size_t)(o.max_hits + 127) / 128 + 1;
    if (e == cudaSuccess) e = dmalloc(&c->ws.tile_done, ntiles * sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(c->ws.tile_done, 0, ntiles * sizeof(int));
    return e;
}

}  // namespace

namespace emtk {

emtk_status validate_request(const emtk_request &q) {
    emtk_status st = check_plane(q.d_adc, q.nwires, q.nticks, q.ld, q.d_hits, q.nhits);
    if (st != EMTK_OK) return st;
    if (q.nhits > 0 && q.d_scores == nullptr) return EMTK_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(q.d_scores) & 3u) != 0) return EMTK_ERR_ALIGN;
    return EMTK_OK;
}

emtk_ctx *make_lane_ctx(const emtk_ctx *parent, emtk_status *st) {
    emtk_ctx *c = new (std::nothrow) emtk_ctx;
    if (!c) {
        *st = EMTK_ERR_OOM;
        return nullptr;
    }
    c->device = parent->device;
    c->opt = parent->opt;
    c->opt.profile = 0;
    c->max_hits = parent->max_hits;
    c->sm_count = parent->sm_count;
    c->w = parent->w;
    c->owns_weights = false;
    DeviceGuard g(c->device);
    cudaError_t e = g.ok ? alloc_workspace(c, false) : cudaErrorInvalidDevice;
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        free_ctx(c);
        *st = cuda_status(e);
        return nullptr;
    }
    *st = EMTK_OK;
    return c;
}

void destroy_lane_ctx(emtk_ctx *c) {
    if (!c) return;
    DeviceGuard g(c->device);
    free_ctx(c);
}

}  // namespace emtk

extern "C" {

void emtk_default_options(emtk_options *o) {
    if (!o) return;
    o->precision = EMTK_BF16;
    o->max_hits = 65536;
    o->debug_logits = 0;
    o->wait_timeout_ns = 2000000000ll;
    o->debug_stall = 0;
    o->profile = 0;
}

const char *emtk_status_string(emtk_status s) {
    switch (s) {
        case EMTK_OK: return "ok";
        case EMTK_ERR_ARG: return "invalid argument";
        case EMTK_ERR_ALIGN: return "misaligned buffer or leading dimension";
        case EMTK_ERR_OOM: return "device allocation failed";
        case EMTK_ERR_CUDA: return "CUDA error";
        case EMTK_ERR_TIMEOUT: return "a device-side wait gave up";
        case EMTK_ERR_UNSUPPORTED: return "unsupported precision or device";
    }
    return "unknown status";
}

emtk_status emtk_create(const emtk_weights *w, const emtk_options *opt, int device, emtk_ctx **out) {
    if (out) *out = nullptr;
    if (!w || !out || device < 0) return EMTK_ERR_ARG;
    const float *all[10] = {w->conv_w, w->conv_b, w->fc1_w, w->fc1_b, w->fc2_w,
                            w->fc2_b,  w->cls_w,  w->cls_b, w->mic_w, w->mic_b};
    for (const float *p : all)
        if (!p) return EMTK_ERR_ARG;
    emtk_options o;
    emtk_default_options(&o);
    if (opt) o = *opt;
    if (o.precision != EMTK_FP32 && o.precision != EMTK_TF32 && o.precision != EMTK_BF16 &&
        o.precision != EMTK_FP16 && o.precision != EMTK_FP8)
        return EMTK_ERR_ARG;
    if (o.max_hits <= 0 || o.wait_timeout_ns <= 0 || (o.debug_logits != 0 && o.debug_logits != 1) ||
        (o.profile != 0 && o.profile != 1) || (o.debug_stall != 0 && o.debug_stall != 1))
        return EMTK_ERR_ARG;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device >= ndev) return EMTK_ERR_CUDA;
    DeviceGuard g(device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess) return EMTK_ERR_CUDA;
    if (!(prop.major == 10 && prop.minor == 3)) return EMTK_ERR_UNSUPPORTED;  // built for sm_103a only

    emtk_ctx *c = new (std::nothrow) emtk_ctx;
    if (!c) return EMTK_ERR_OOM;
    c->device = device;
    c->opt = o;
    c->max_hits = o.max_hits;
    c->sm_count = prop.multiProcessorCount;
    cudaError_t e = cudaSuccess;
    DeviceWeights &d = c->w;
    if (e == cudaSuccess) e = upload(&d.conv_w, w->conv_w, (size_t)kK * kK * kF);
    if (e == cudaSuccess) e = upload(&d.conv_b, w->conv_b, kF);
    std::copy(w->conv_w, w->conv_w + kK * kK * kF, d.conv_w_host);
    std::copy(w->conv_b, w->conv_b + kF, d.conv_b_host);
    if (e == cudaSuccess) e = upload(&d.fc1_b, w->fc1_b, kN1);
    if (e == cudaSuccess) e = upload(&d.fc2_w, w->fc2_w, (size_t)kN1 * kN2);
    if (e == cudaSuccess) e = upload(&d.fc2_b, w->fc2_b, kN2);
    if (e == cudaSuccess) e = upload(&d.cls_w, w->cls_w, (size_t)kN2 * kNC);
    if (e == cudaSuccess) e = upload(&d.cls_b, w->cls_b, kNC);
    if (e == cudaSuccess) e = upload(&d.mic_w, w->mic_w, kN2);
    if (e == cudaSuccess) e = upload(&d.mic_b, w->mic_b, 1);
    if (e == cudaSuccess) {
        if (o.precision == EMTK_TF32) {
            e = prepare_split_weights(d, *w);
            if (e == cudaSuccess) e = init_split_kernel_attrs();
        } else if (tensor_precision(o.precision)) {
            e = prepare_tc_weights(d, *w, tc_mode(o.precision));
            if (e == cudaSuccess) e = init_tc_kernel_attrs();
        } else {
            e = upload(&d.fc1_w, w->fc1_w, (size_t)kFc1In * kN1);
            if (e == cudaSuccess) e = init_fp32_kernel_attrs();
        }
    }
    if (e == cudaSuccess) e = init_head_kernel_attrs();
    if (e == cudaSuccess) e = alloc_workspace(c, true);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        free_ctx(c);
        return cuda_status(e);
    }
    *out = c;
    return EMTK_OK;
}

emtk_status emtk_destroy(emtk_ctx *c) {
    if (!c) return EMTK_OK;
    DeviceGuard g(c->device);
    cudaDeviceSynchronize();
    free_ctx(c);
    return EMTK_OK;
}

emtk_status emtk_infer_batch(emtk_ctx *c, const emtk_request *reqs, int32_t nreq, emtk_stream stream) {
    if (!c || nreq < 0 || (nreq > 0 && !reqs)) return EMTK_ERR_ARG;
    for (int i = 0; i < nreq; ++i) {
        const emtk_status st = validate_request(reqs[i]);
        if (st != EMTK_OK) return st;
    }
    c->stats.calls++;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    return run_requests(c, reqs, nreq, reinterpret_cast<cudaStream_t>(stream));
}

emtk_status emtk_infer(emtk_ctx *c, const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld,
                       const emtk_hit *d_hits, int32_t nhits, float *d_scores, emtk_stream stream) {
    if (!c) return EMTK_ERR_ARG;
    emtk_request q{d_adc, nwires, nticks, ld, d_hits, nhits, d_scores};
    return emtk_infer_batch(c, &q, 1, stream);
}

emtk_status emtk_extract_patches(emtk_ctx *c, const float *d_adc, int32_t nwires, int32_t nticks, int64_t ld,
                                 const emtk_hit *d_hits, int32_t nhits, void *d_patches, emtk_patch_format fmt,
                                 emtk_stream stream) {
    if (!c) return EMTK_ERR_ARG;
    if (fmt != EMTK_PATCH_F32 && fmt != EMTK_PATCH_BF16 && fmt != EMTK_PATCH_F16) return EMTK_ERR_ARG;
    emtk_status st = check_plane(d_adc, nwires, nticks, ld, d_hits, nhits);
    if (st != EMTK_OK) return st;
    if (nhits == 0) return EMTK_OK;
    if (!d_patches) return EMTK_ERR_ARG;
    if (!aligned16(d_patches)) return EMTK_ERR_ALIGN;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    emtk_request q{d_adc, nwires, nticks, ld, d_hits, nhits, nullptr};
    ReqTable *t = new (std::nothrow) ReqTable;
    if (!t) return EMTK_ERR_OOM;
    int64_t hits;
    size_t img_bytes;
    build_table(c, &q, 0, 1, fmt, 0, *t, hits, img_bytes);
    st = ensure_dimg(c, img_bytes, s);
    if (st == EMTK_OK) {
        Prof prof(c, EMTK_KERNEL_INTERVALS, s);
        st = cuda_status(launch_interval_images(*t, c->ws.dimg, fmt, s));
    }
    if (st == EMTK_OK) {
        Prof prof(c, EMTK_KERNEL_GATHER, s);
        st = cuda_status(launch_gather(*t, c->ws.dimg, fmt, 0, nhits, d_patches, nullptr, 0, s));
    }
    c->stats.calls++;
    delete t;
    return st;
}

emtk_status emtk_infer_patches(emtk_ctx *c, const float *d_patches, int32_t n, float *d_scores,
                               emtk_stream stream) {
    if (!c || n < 0) return EMTK_ERR_ARG;
    if (n == 0) return EMTK_OK;
    if (!d_patches || !d_scores) return EMTK_ERR_ARG;
    if (!aligned16(d_patches) || (reinterpret_cast<uintptr_t>(d_scores) & 3u) != 0) return EMTK_ERR_ALIGN;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const emtk_patch_format fmt = patch_format(c->opt.precision);
    emtk_status st = EMTK_OK;
    for (int64_t h0 = 0; h0 < n && st == EMTK_OK; h0 += c->max_hits) {
        const int32_t cnt = (int32_t)std::min<int64_t>(c->max_hits, n - h0);
        const float *src = d_patches + h0 * kPatchElems;
        // the head writes hit h's scores to rows + h * stride (no pointer table)
        const OutRows out{nullptr, d_scores + h0 * out_stride(c), out_stride(c)};
        if (fmt == EMTK_PATCH_BF16 || fmt == EMTK_PATCH_F16) {
            // the tensor-core kernel reads the fp32 patches itself: no conversion launch
            st = run_network(c, nullptr, nullptr, cnt, out, src, s);
        } else if (fmt == kPatchSplit16) {
            {
                // the split-fp16 network reads head / tail words: one conversion launch first
                Prof prof(c, EMTK_KERNEL_CONVERT, s);
                st = cuda_status(launch_convert_split(src, c->ws.patches, (int64_t)cnt * kPatchElems, c->sm_count, s));
            }
            if (st == EMTK_OK) st = run_network(c, c->ws.patches, nullptr, cnt, out, nullptr, s);
        } else {
            st = run_network(c, src, nullptr, cnt, out, nullptr, s);  // the fp32 kernel reads the patches
        }
    }
    c->stats.calls++;
    c->stats.hits += (uint64_t)n;
    return st;
}

emtk_status emtk_check(emtk_ctx *c, emtk_stream stream) {
    if (!c) return EMTK_ERR_ARG;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return EMTK_ERR_CUDA;
    int status = 0;
    e = cudaMemcpy(&status, c->ws.status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return EMTK_ERR_CUDA;
    if (status != 0) {
        e = cudaMemset(c->ws.status, 0, sizeof(int));
        // a launch that gave up may have left tile counters part-way
        const size_t ntiles = (size_t)(c->opt.max_hits + 127) / 128 + 1;
        if (e == cudaSuccess && c->ws.tile_done) e = cudaMemset(c->ws.tile_done, 0, ntiles * sizeof(int));
        c->tile_mask_cap = 0;  // and tile masks: the next call reallocates and zeroes them
        if (e != cudaSuccess) return EMTK_ERR_CUDA;
        return EMTK_ERR_TIMEOUT;
    }
    return EMTK_OK;
}

emtk_status emtk_get_stats(emtk_ctx *c, emtk_stats *out) {
    if (!c || !out) return EMTK_ERR_ARG;
    if (!c->pending.empty()) {
        DeviceGuard g(c->device);
        drain_events(c);
    }
    *out = c->stats;
    return EMTK_OK;
}

emtk_status emtk_infer_batch_host(emtk_ctx *c, const emtk_request *reqs, int32_t nreq, emtk_stream stream) {
    if (!c || nreq < 0 || (nreq > 0 && !reqs)) return EMTK_ERR_ARG;
    // staging layout: each plane at a 256-byte boundary, then the hit lists, then the scores
    const int stride = out_stride(c);
    auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
    std::vector<size_t> off_adc(nreq), off_hits(nreq), off_sc(nreq);
    size_t need = 0;
    for (int32_t i = 0; i < nreq; ++i) {
        const emtk_request &q = reqs[i];
        if (q.nwires < 0 || q.nticks < 0 || q.nhits < 0 || q.ld < q.nticks || (q.ld % 4) != 0) return EMTK_ERR_ARG;
        if (q.nhits > 0 && (!q.d_adc || !q.d_hits || !q.d_scores)) return EMTK_ERR_ARG;
        off_adc[i] = need;
        need = up(need + (q.nhits > 0 ? (size_t)q.nwires * (size_t)q.ld * sizeof(float) : 0));
    }
    // the hit lists back to back (8-byte aligned), so that one copy brings them all
    const size_t hits0 = need;
    for (int32_t i = 0; i < nreq; ++i) {
        off_hits[i] = need;
        need += (size_t)reqs[i].nhits * sizeof(emtk_hit);
    }
    const size_t hit_bytes = need - hits0;
    need = up(need);
    for (int32_t i = 0; i < nreq; ++i) {
        off_sc[i] = need;
        need = up(need + (size_t)reqs[i].nhits * stride * sizeof(float));
    }
    if (need == 0) return EMTK_OK;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    if (!c->copy_stream) e = cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking);
    emtk_ctx::HostStage &st = c->stage[c->host_calls % 2];
    if (e == cudaSuccess && !st.copy_done) e = cudaEventCreateWithFlags(&st.copy_done, cudaEventDisableTiming);
    if (e == cudaSuccess && !st.compute_done) e = cudaEventCreateWithFlags(&st.compute_done, cudaEventDisableTiming);
    if (e == cudaSuccess && st.bytes < need) {  // grow: wait for the area's last call, then reallocate
        if (st.used) e = cudaEventSynchronize(st.compute_done);
        if (e == cudaSuccess) e = dev_free(st.buf);
        st.buf = nullptr;
        st.bytes = 0;
        if (e == cudaSuccess) e = dev_alloc(&st.buf, need);
        if (e == cudaSuccess) st.bytes = need;
    }
    // the pinned host area for the hit lists: its last copy (two calls back) has landed
    if (e == cudaSuccess && st.used) e = cudaEventSynchronize(st.copy_done);
    if (e == cudaSuccess && st.hits_host_bytes < hit_bytes) {
        e = host_free(st.hits_host);
        st.hits_host = nullptr;
        st.hits_host_bytes = 0;
        if (e == cudaSuccess) e = host_alloc(&st.hits_host, hit_bytes + hit_bytes / 4);
        if (e == cudaSuccess) st.hits_host_bytes = hit_bytes + hit_bytes / 4;
    }
    if (e != cudaSuccess) return cuda_status(e);
    char *base = static_cast<char *>(st.buf);
    // copy in on the copy stream, once the area's previous call is done with it
    if (st.used) e = cudaStreamWaitEvent(c->copy_stream, st.compute_done, 0);
    std::vector<emtk_request> dq(reqs, reqs + nreq);
    // planes: one copy per run of planes contiguous both on the host and in the area
    const char *run_src = nullptr;
    size_t run_dst = 0, run_len = 0;
    auto flush = [&]() {
        if (run_len > 0 && e == cudaSuccess)
            e = cudaMemcpyAsync(base + run_dst, run_src, run_len, cudaMemcpyHostToDevice, c->copy_stream);
        run_len = 0;
    };
    for (int32_t i = 0; i < nreq && e == cudaSuccess; ++i) {
        const emtk_request &q = reqs[i];
        if (q.nhits == 0) {  // nothing of it is read: no host pointer reaches the batch
            dq[i].d_adc = nullptr;
            dq[i].d_hits = nullptr;
            dq[i].d_scores = nullptr;
            continue;
        }
        const char *src = reinterpret_cast<const char *>(q.d_adc);
        const size_t len = (size_t)q.nwires * q.ld * sizeof(float);
        if (run_len > 0 && src == run_src + run_len && off_adc[i] == run_dst + run_len) {
            run_len += len;
        } else {
            flush();
            run_src = src;
            run_dst = off_adc[i];
            run_len = len;
        }
        std::memcpy(static_cast<char *>(st.hits_host) + (off_hits[i] - hits0), q.d_hits,
                    (size_t)q.nhits * sizeof(emtk_hit));
        dq[i].d_adc = reinterpret_cast<const float *>(base + off_adc[i]);
        dq[i].d_hits = reinterpret_cast<const emtk_hit *>(base + off_hits[i]);
        dq[i].d_scores = reinterpret_cast<float *>(base + off_sc[i]);
    }
    flush();
    if (e == cudaSuccess && hit_bytes > 0)
        e = cudaMemcpyAsync(base + hits0, st.hits_host, hit_bytes, cudaMemcpyHostToDevice, c->copy_stream);
    if (e == cudaSuccess) e = cudaEventRecord(st.copy_done, c->copy_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, st.copy_done, 0);
    if (e != cudaSuccess) return cuda_status(e);
    // the batch on the caller's stream, then the scores back to the caller's buffers
    emtk_status r = emtk_infer_batch(c, dq.data(), nreq, stream);
    for (int32_t i = 0; i < nreq && r == EMTK_OK; ++i) {
        const emtk_request &q = reqs[i];
        if (q.nhits == 0) continue;
        e = cudaMemcpyAsync(q.d_scores, base + off_sc[i], (size_t)q.nhits * stride * sizeof(float),
                            cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) r = cuda_status(e);
    }
    e = cudaEventRecord(st.compute_done, s);
    if (e != cudaSuccess && r == EMTK_OK) r = cuda_status(e);
    st.used = true;
    c->host_calls++;
    return r;
}

emtk_status emtk_find_hits(emtk_ctx *c, emtk_hitfind_request *reqs, int32_t nreq, emtk_stream stream) {
    if (!c || nreq < 0 || (nreq > 0 && !reqs)) return EMTK_ERR_ARG;
    // the most runs a plane can hold: one per two ticks on every wire
    auto max_runs = [](const emtk_hitfind_request &q) { return (int64_t)q.nwires * ((q.nticks + 1) / 2); };
    // scratch (the partial-sum workspace): plane totals in its first 256 bytes, then the
    // group's per-wire scratch
    const size_t scratch_bytes = c->ws.partial_elems * sizeof(float) - 256;
    const int64_t unit_cap = find_hits_unit_cap(scratch_bytes);
    // a plane's units: wire segments of kSegTicks ticks (none without ticks)
    auto units = [](const emtk_hitfind_request &q) {
        return q.nticks > 0 ? (int64_t)q.nwires * ((q.nticks + kSegTicks - 1) / kSegTicks) : 0;
    };
    for (int32_t i = 0; i < nreq; ++i) {
        const emtk_hitfind_request &q = reqs[i];
        if (q.nwires < 0 || q.nticks < 0 || q.ld < q.nticks || q.capacity < 0) return EMTK_ERR_ARG;
        if (q.capacity > 0 && q.d_hits == nullptr) return EMTK_ERR_ARG;
        if (q.nwires > 0 && q.nticks > 0 && q.d_adc == nullptr) return EMTK_ERR_ARG;
        if (max_runs(q) > INT32_MAX || units(q) > unit_cap) return EMTK_ERR_ARG;
        if (q.d_adc != nullptr && (!aligned16(q.d_adc) || (q.ld % 4) != 0)) return EMTK_ERR_ALIGN;
        if ((reinterpret_cast<uintptr_t>(q.d_hits) & 7u) != 0 || (reinterpret_cast<uintptr_t>(q.d_info) & 3u) != 0)
            return EMTK_ERR_ALIGN;
    }
    for (int32_t i = 0; i < nreq; ++i) reqs[i].n_found = 0;
    if (nreq == 0) return EMTK_OK;
    DeviceGuard g(c->device);
    if (!g.ok) return EMTK_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (!c->h_totals) {
        void *h = nullptr;
        if (host_alloc(&h, sizeof(int32_t) * kMaxHfPlanes) != cudaSuccess) return EMTK_ERR_OOM;
        c->h_totals = static_cast<int32_t *>(h);
    }
    int32_t *totals = reinterpret_cast<int32_t *>(c->ws.partials);
    void *scratch = reinterpret_cast<char *>(c->ws.partials) + 256;
    int32_t i = 0;
    while (i < nreq) {
        // a group: up to kMaxHfPlanes planes whose units fit the scratch
        HfTable t{};
        int64_t U = 0;
        const int32_t first = i;
        while (i < nreq && t.n < kMaxHfPlanes) {
            const emtk_hitfind_request &q = reqs[i];
            const int64_t nu = units(q);
            if (t.n > 0 && U + nu > unit_cap) break;
            HfDesc &d = t.r[t.n++];
            d.adc = q.d_adc;
            d.hits = q.d_hits;
            d.info = q.d_info;
            d.ld = q.ld;
            d.unit0 = U;
            d.nticks = q.nticks;
            d.nseg = (q.nticks + kSegTicks - 1) / kSegTicks;
            d.capacity = q.capacity;
            d.thr = q.threshold;
            U += nu;
            ++i;
        }
        // the chunk sums: two zeroed halves of hf_sums_cap, grown (and zeroed) when needed
        cudaError_t e = cudaSuccess;
        const int64_t nchunks = find_hits_chunks(t, U);
        if (nchunks > c->hf_sums_cap) {
            e = cudaStreamSynchronize(s);
            if (e == cudaSuccess) e = dev_free(c->hf_sums);
            c->hf_sums = nullptr;
            c->hf_sums_cap = 0;
            const int64_t cap = nchunks + nchunks / 4 + 64;
            if (e == cudaSuccess) e = dmalloc(&c->hf_sums, 2 * cap * sizeof(int32_t));
            if (e == cudaSuccess) e = cudaMemsetAsync(c->hf_sums, 0, 2 * cap * sizeof(int32_t), s);
            if (e != cudaSuccess) return cuda_status(e);
            c->hf_sums_cap = cap;
            c->hf_parity = 0;
        }
        int32_t *cur = c->hf_sums + (int64_t)c->hf_parity * c->hf_sums_cap;
        int32_t *next = c->hf_sums + (int64_t)(1 - c->hf_parity) * c->hf_sums_cap;
        {
            Prof prof(c, EMTK_KERNEL_HITFIND, s, U > 0 ? 2 : 0);  // find, then place
            e = launch_find_hits(t, U, scratch, cur, next, c->hf_sums_cap, totals, s);
        }
        if (e == cudaSuccess && U > 0) c->hf_parity ^= 1;
        if (e == cudaSuccess) e = cudaMemcpyAsync(c->h_totals, totals, sizeof(int32_t) * t.n, cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) {
            // the launch or the kernels may have stopped before the place kernel cleared
            // the other half: the next call reallocates and zeroes both halves
            c->hf_sums_cap = 0;
            return cuda_status(e);
        }
        for (int r = 0; r < t.n; ++r) reqs[first + r].n_found = c->h_totals[r];
    }
    return EMTK_OK;
}

emtk_status emtk_get_fp8_scales(const emtk_ctx *c, float *s_a, float *s_w) {
    if (!c) return EMTK_ERR_ARG;
    const bool f8 = c->opt.precision == EMTK_FP8;
    if (s_a) *s_a = f8 ? 1.0f / (c->w.fc1_scale * c->w.fc1_w_scale) : 1.0f;
    if (s_w) *s_w = f8 ? c->w.fc1_w_scale : 1.0f;
    return EMTK_OK;
}

}  // extern "C"
