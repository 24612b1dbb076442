// Patch extraction (Sec. 2.1): every hit gets a 48x48 patch, rows = wires,
// columns = time intervals of 6 ticks, centred on the hit (row 24 / column
// 24); pixels outside the plane are zero.
//
// Two HBM-friendly passes instead of one gather per hit:
//   1. interval image: each plane's ticks are reduced once to its interval
//      values (fp32 sum of the 6 ticks left to right, one fp32 divide by 6),
//      stored in the patch format.  Reads every plane byte exactly once
//      (16-byte vector loads, streaming), writes 1/6 of it (stays in L2).
//   2. gather: each patch is copied out of the L2-resident interval image.
// Hits of windows that overlap read the same interval values, so the plane
// is never re-read per hit.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "emtk_internal.h"

namespace emtk {
namespace {

__device__ __forceinline__ float interval_sum(float a0, float a1, float a2, float a3, float a4, float a5) {
    // fixed order: ((((a0 + a1) + a2) + a3) + a4) + a5, no contraction possible
    float s = __fadd_rn(a0, a1);
    s = __fadd_rn(s, a2);
    s = __fadd_rn(s, a3);
    s = __fadd_rn(s, a4);
    s = __fadd_rn(s, a5);
    return __fdiv_rn(s, 6.0f);
}

// One pixel of the EMTK_TF32 image: the fp16 head of v * s_p in the low half,
// the fp16 tail (v * s_p - head, rounded) in the high half.  s_p is a power
// of two, so the product is exact.
__device__ __forceinline__ uint32_t split_word(float v) {
    const float x = __fmul_rn(v, kSplitPatchScale);
    const __half h = __float2half_rn(x);
    const __half t = __float2half_rn(__fsub_rn(x, __half2float(h)));
    return (uint32_t)__half_as_ushort(h) | ((uint32_t)__half_as_ushort(t) << 16);
}

template <int FMT>
__device__ __forceinline__ void store2(void *base, int64_t idx, float v0, float v1, bool two) {
    if (FMT == kPatchSplit16) {
        uint32_t *p = static_cast<uint32_t *>(base) + idx;
        if (two) {
            *reinterpret_cast<uint2 *>(p) = make_uint2(split_word(v0), split_word(v1));
        } else {
            p[0] = split_word(v0);
        }
    } else if (FMT == EMTK_PATCH_F32) {
        float *p = static_cast<float *>(base) + idx;
        if (two) {
            *reinterpret_cast<float2 *>(p) = make_float2(v0, v1);
        } else {
            p[0] = v0;
        }
    } else if (FMT == EMTK_PATCH_BF16) {
        __nv_bfloat16 *p = static_cast<__nv_bfloat16 *>(base) + idx;
        if (two) {
            __nv_bfloat162 h;
            h.x = __float2bfloat16_rn(v0);
            h.y = __float2bfloat16_rn(v1);
            *reinterpret_cast<__nv_bfloat162 *>(p) = h;
        } else {
            p[0] = __float2bfloat16_rn(v0);
        }
    } else {
        __half *p = static_cast<__half *>(base) + idx;
        if (two) {
            *reinterpret_cast<__half2 *>(p) = __halves2half2(__float2half_rn(v0), __float2half_rn(v1));
        } else {
            p[0] = __float2half_rn(v0);
        }
    }
}

// One thread = two consecutive image columns of one image row; inside the
// plane that is two intervals of one wire (12 ticks = 48 bytes, 16-byte
// aligned because ld % 4 == 0, the plane is 16-byte aligned and the halo is
// even), outside it (the zero halo, the pitch padding) zeros.  The image
// of request r, grid-stride over its column pairs along x; the pitch and the
// image offset are even, so the pair store is aligned too.
template <int FMT>
__device__ __forceinline__ void interval_request(const ReqDesc &r, void *img) {
    if (r.nwires == 0) return;
    const int npairs = r.pitch >> 1;
    const int rows = r.nwires + 2 * r.halo;
    const int64_t work = (int64_t)rows * npairs;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < work;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int wr = (int)(i / npairs);
        const int cb = 2 * (int)(i - (int64_t)wr * npairs);
        const int w = wr - r.halo;
        const int b = cb - r.halo;
        float v0 = 0.0f, v1 = 0.0f;
        if (w >= 0 && w < r.nwires && b >= 0 && b < r.nint) {
            const float *src = r.adc + (int64_t)w * r.ld + 6 * b;
            const float4 x0 = __ldcs(reinterpret_cast<const float4 *>(src));
            const float2 x1 = __ldcs(reinterpret_cast<const float2 *>(src + 4));
            v0 = interval_sum(x0.x, x0.y, x0.z, x0.w, x1.x, x1.y);
            if (b + 1 < r.nint) {
                const float2 x2 = __ldcs(reinterpret_cast<const float2 *>(src + 6));
                const float4 x3 = __ldcs(reinterpret_cast<const float4 *>(src + 8));
                v1 = interval_sum(x2.x, x2.y, x3.x, x3.y, x3.z, x3.w);
            }
        }
        store2<FMT>(img, r.d_off + (int64_t)wr * r.pitch + cb, v0, v1, true);
    }
}

// grid.y = request.
template <int FMT>
__global__ void __launch_bounds__(256) interval_image_kernel(const __grid_constant__ ReqTable t, void *img) {
    pdl_trigger();  // the network kernel may set up while this one finishes; it waits for it
    interval_request<FMT>(t.r[blockIdx.y], img);
}

template <int FMT>
struct Elem;
template <>
struct Elem<EMTK_PATCH_F32> {
    using T = float;
};
template <>
struct Elem<EMTK_PATCH_BF16> {
    using T = unsigned short;
};
template <>
struct Elem<EMTK_PATCH_F16> {
    using T = unsigned short;
};

__device__ __forceinline__ int find_request(const ReqTable &t, int64_t g) {
    int lo = 0, hi = t.n - 1;
    while (lo < hi) {  // last request with hit_begin <= g
        const int mid = (lo + hi + 1) >> 1;
        if (t.r[mid].hit_begin <= g)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ int64_t floor_div6(int64_t a) {
    int64_t q = a / 6;
    if ((a % 6) != 0 && a < 0) q -= 1;
    return q;
}

// One block per hit: 48 rows x (48 / V) vectors of V elements (16 bytes).
template <int FMT>
__global__ void __launch_bounds__(288) gather_kernel(const __grid_constant__ ReqTable t, const void *img,
                                                     int64_t g0, void *patches, float **dest,
                                                     int out_stride) {
    using T = typename Elem<FMT>::T;
    constexpr int V = 16 / sizeof(T);
    constexpr int CH = kPatch / V;
    const int64_t local = blockIdx.x;
    const int64_t g = g0 + local;
    const int ri = find_request(t, g);
    const ReqDesc &r = t.r[ri];
    const int64_t hloc = g - r.hit_begin;
    const emtk_hit hit = r.hits[hloc];
    const int64_t wc = hit.wire;
    const int64_t bc = floor_div6(hit.tick);
    const T *src = static_cast<const T *>(img) + r.d_off;
    T *out = static_cast<T *>(patches) + local * kPatchElems;
    if (dest != nullptr && threadIdx.x == 0) dest[local] = r.scores + hloc * out_stride;
    for (int task = threadIdx.x; task < kPatch * CH; task += blockDim.x) {
        const int row = task / CH;
        const int c0 = (task - row * CH) * V;
        const int64_t w = wc - kHalf + row;
        union {
            T e[V];
            uint4 u;
        } v;
        const bool wire_ok = (w >= 0 && w < r.nwires);
#pragma unroll
        for (int e = 0; e < V; ++e) {
            const int64_t b = bc - kHalf + c0 + e;
            v.e[e] = (wire_ok && b >= 0 && b < r.nint) ? src[(w + r.halo) * r.pitch + b + r.halo] : T(0);
        }
        *reinterpret_cast<uint4 *>(out + row * kPatch + c0) = v.u;
    }
}

// Pre-cut fp32 patches -> the split-fp16 head / tail words of the EMTK_TF32
// network (emtk_infer_patches; the 16-bit kernels read fp32 patches
// themselves): eight values per thread and step (two 16-byte streaming loads,
// so the dense-1 weights keep their place in L2), four steps in flight; the
// same word per value as the interval images.  n8 = values / 8 (a patch is
// 2,304 values).
__global__ void convert_split_kernel(const float *__restrict__ src, uint4 *__restrict__ dst, int64_t n8) {
    pdl_trigger();  // the network kernel may set up while this one runs; it waits for it
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t nthreads = (int64_t)gridDim.x * blockDim.x;
    const float4 *s4 = reinterpret_cast<const float4 *>(src);
    constexpr int kU = 4;
    for (int64_t base = tid; base < n8; base += nthreads * kU) {
        float4 a[kU], b[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int64_t i = base + u * nthreads;
            if (i < n8) {
                a[u] = __ldcs(s4 + 2 * i);
                b[u] = __ldcs(s4 + 2 * i + 1);
            }
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int64_t i = base + u * nthreads;
            if (i >= n8) continue;
            dst[2 * i] = make_uint4(split_word(a[u].x), split_word(a[u].y), split_word(a[u].z), split_word(a[u].w));
            dst[2 * i + 1] =
                make_uint4(split_word(b[u].x), split_word(b[u].y), split_word(b[u].z), split_word(b[u].w));
        }
    }
}

// The window descriptor of hit g0 + local of the table (and its output row).
__device__ __forceinline__ void hit_desc_one(const ReqTable &t, int64_t g0, int64_t local, HitDesc *desc,
                                             float **dest, int out_stride) {
    const int64_t g = g0 + local;
    const ReqDesc &r = t.r[find_request(t, g)];
    const int64_t hloc = g - r.hit_begin;
    const emtk_hit hit = r.hits[hloc];
    const int64_t bc = floor_div6(hit.tick);
    HitDesc d;
    d.wc = hit.wire;
    d.bc = (int32_t)bc;  // |tick| < 2^31, so the interval fits
    d.nwires = r.nwires;
    d.nint = r.nint;
    d.pitch = r.pitch;
    d.d_off = r.d_off;
    // the window [wc-24, wc+24) x [bc-24, bc+24) lies in the haloed image iff
    // the hit itself lies in the plane (the halo is 24 wide)
    d.inside = (hit.wire >= 0 && hit.wire < r.nwires && bc >= 0 && bc < r.nint) ? 1 : 0;
    d.origin = d.inside ? r.d_off + (int64_t)(hit.wire - kHalf + r.halo) * r.pitch + (bc - kHalf + r.halo) : 0;
    desc[local] = d;
    if (dest != nullptr) dest[local] = r.scores + hloc * out_stride;
}

__global__ void hit_desc_kernel(const __grid_constant__ ReqTable t, int64_t g0, int32_t count, HitDesc *desc,
                                float **dest, int out_stride) {
    pdl_trigger();
    const int64_t local = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (local < count) hit_desc_one(t, g0, local, desc, dest, out_stride);
}

// The images (grid rows 0 .. t.n - 1) and, in one more grid row, the window
// descriptors of hits g0 .. g0 + count - 1: the descriptors' few bytes ride
// along with the images' stream instead of taking a launch of their own.
template <int FMT>
__global__ void __launch_bounds__(256) interval_desc_kernel(const __grid_constant__ ReqTable t, void *img, int64_t g0,
                                                            int32_t count, HitDesc *desc, float **dest,
                                                            int out_stride) {
    pdl_trigger();
    if ((int)blockIdx.y < t.n) {
        interval_request<FMT>(t.r[blockIdx.y], img);
        return;
    }
    for (int64_t local = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; local < count;
         local += (int64_t)gridDim.x * blockDim.x)
        hit_desc_one(t, g0, local, desc, dest, out_stride);
}

// The tiles of request r's image that the window of `hit` touches: image rows
// [wire, wire + 47] x image columns [bc, bc + 47] (halo 24), clipped to the
// image; a hit outside its plane marks the part of its window inside the
// image (its in-plane pixels are all there).  The window spans at most 7
// bands and 48 / kTileInts + 1 tile columns, in at most 2 mask words;
// `valid` false marks nothing.
struct WindowTiles {
    int64_t band0;    // first band
    int nbands;       // 0 .. 7
    int w0, nwords;   // first mask word of a band row, 1 or 2
    uint32_t bits[2]; // tile bits in words w0, w0 + 1
};
__device__ __forceinline__ WindowTiles window_tiles(const ReqDesc &r, const emtk_hit &hit, bool valid) {
    WindowTiles wt{0, 0, 0, 0, {0u, 0u}};
    if (!valid) return wt;
    const int64_t rows = (int64_t)r.nwires + 2 * r.halo;
    const int64_t bc = floor_div6(hit.tick);
    const int64_t r0 = hit.wire > 0 ? hit.wire : 0;
    const int64_t r1 = (int64_t)hit.wire + 2 * kHalf - 1 < rows - 1 ? (int64_t)hit.wire + 2 * kHalf - 1 : rows - 1;
    const int64_t c0 = bc > 0 ? bc : 0;
    const int64_t c1 = bc + 2 * kHalf - 1 < r.pitch - 1 ? bc + 2 * kHalf - 1 : (int64_t)r.pitch - 1;
    if (r0 > r1 || c0 > c1) return wt;
    const int t0 = (int)(c0 / kTileInts), t1 = (int)(c1 / kTileInts);
    wt.band0 = r0 / kTileRows;
    wt.nbands = (int)(r1 / kTileRows - wt.band0 + 1);
    wt.w0 = t0 >> 5;
    wt.nwords = (t1 >> 5) - wt.w0 + 1;
    for (int k = 0; k < wt.nwords; ++k) {
        const int wd = wt.w0 + k;
        const int lo = t0 > 32 * wd ? t0 - 32 * wd : 0;
        const int hi = t1 < 32 * wd + 31 ? t1 - 32 * wd : 31;
        wt.bits[k] = (hi == 31 ? 0xffffffffu : ((1u << (hi + 1)) - 1u)) & ~((1u << lo) - 1u);
    }
    return wt;
}

// Every hit of request blockIdx.y marks its window's tiles (one thread per
// hit).  The hits of a block (consecutive in the list: a track or a shower
// of one plane) mostly mark the same few words, and atomics to one word
// serialize in L2, so a block first ORs its marks into a shared-memory copy
// of the plane's mask and then sends each non-zero word once.  A plane whose
// mask is larger than kMarkSmemWords words marks global memory directly.
constexpr int kMarkSmemWords = 8192;  // 32 KB
__global__ void __launch_bounds__(256) mark_tiles_kernel(const __grid_constant__ ReqTable t, uint32_t *mask,
                                                         int smem_words) {
    extern __shared__ uint32_t plane_mask[];
    pdl_trigger();  // the tile kernel may be scheduled; it waits for this one
    const ReqDesc &r = t.r[blockIdx.y];
    const int64_t rows = r.nwires > 0 ? (int64_t)r.nwires + 2 * r.halo : 0;
    const int64_t words = (rows + kTileRows - 1) / kTileRows * r.m_wpb;
    const bool local = words <= smem_words;
    if (local) {
        for (int64_t i = threadIdx.x; i < words; i += blockDim.x) plane_mask[i] = 0u;
        __syncthreads();
    }
    uint32_t *dst = local ? plane_mask : mask + r.m_off;
    for (int64_t h = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; h < r.nhits;
         h += (int64_t)gridDim.x * blockDim.x) {
        const WindowTiles wt = window_tiles(r, r.hits[h], r.nwires > 0);
        uint32_t *row0 = dst + wt.band0 * r.m_wpb + wt.w0;
        for (int b = 0; b < wt.nbands; ++b)
            for (int k = 0; k < wt.nwords; ++k) atomicOr(row0 + b * r.m_wpb + k, wt.bits[k]);
    }
    if (local) {
        __syncthreads();
        for (int64_t i = threadIdx.x; i < words; i += blockDim.x)
            if (plane_mask[i]) atomicOr(mask + r.m_off + i, plane_mask[i]);
    }
}

// One warp per tile (kTileRows rows x kTileInts intervals = 8 x 8 column
// pairs) of request blockIdx.y: a tile no window touches is left as it is;
// the others are computed as in interval_request (same sums, same rounding),
// two column pairs per lane with every load issued before the first sum.
// Grid row blockIdx.y == t.n builds the window descriptors and output rows
// of hits [g0, g0 + count).  All threads together clear mask_next for the
// next launch.
constexpr int kTileWarps = 8;
template <int FMT>
__global__ void __launch_bounds__(kTileWarps * 32) interval_tiles_kernel(const __grid_constant__ ReqTable t, void *img,
                                                                         const uint32_t *mask_cur, uint32_t *mask_next,
                                                                         int64_t mask_cap, int64_t g0, int32_t count,
                                                                         HitDesc *desc, float **dest, int out_stride) {
    pdl_trigger();  // the network kernel may set up while this one runs; it waits for it
    const int64_t nthr = (int64_t)gridDim.x * gridDim.y * blockDim.x;
    for (int64_t i = ((int64_t)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x; i < mask_cap;
         i += nthr)
        mask_next[i] = 0u;
    if ((int)blockIdx.y == t.n) {  // the descriptors need nothing from the marking kernel
        for (int64_t local = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; local < count;
             local += (int64_t)gridDim.x * blockDim.x)
            hit_desc_one(t, g0, local, desc, dest, out_stride);
        return;
    }
    pdl_wait();     // the marks come from the kernel before
    const ReqDesc &r = t.r[blockIdx.y];
    if (r.nwires == 0) return;
    const int lane = threadIdx.x & 31;
    const int rows = r.nwires + 2 * r.halo;
    const int npairs = r.pitch >> 1;
    const int nbands = (rows + kTileRows - 1) / kTileRows;
    const int nchunks = (r.pitch + kTileInts - 1) / kTileInts;
    const int64_t tile = (int64_t)blockIdx.x * kTileWarps + (threadIdx.x >> 5);
    if (tile >= (int64_t)nbands * nchunks) return;
    const int band = (int)(tile / nchunks), chunk = (int)(tile - (int64_t)band * nchunks);
    if (((mask_cur[r.m_off + (int64_t)band * r.m_wpb + (chunk >> 5)] >> (chunk & 31)) & 1u) == 0) return;
    constexpr int kPairs = kTileInts / 2;          // column pairs per tile row
    constexpr int kU = kTileRows * kPairs / 32;    // pairs per lane
    float4 xa[kU], xd[kU];
    float2 xb[kU], xc[kU];
    bool in0[kU], in1[kU];
    int64_t dst[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
        const int j = lane + 32 * u;
        const int wr = band * kTileRows + j / kPairs;
        const int cp = chunk * kPairs + j % kPairs;
        const int cb = 2 * cp;
        const int w = wr - r.halo, b = cb - r.halo;
        in0[u] = wr < rows && cp < npairs && w >= 0 && w < r.nwires && b >= 0 && b < r.nint;
        in1[u] = in0[u] && b + 1 < r.nint;
        dst[u] = (wr < rows && cp < npairs) ? r.d_off + (int64_t)wr * r.pitch + cb : -1;
        const float *src = r.adc + (int64_t)w * r.ld + 6 * b;
        if (in0[u]) {
            xa[u] = __ldcs(reinterpret_cast<const float4 *>(src));
            xb[u] = __ldcs(reinterpret_cast<const float2 *>(src + 4));
        }
        if (in1[u]) {
            xc[u] = __ldcs(reinterpret_cast<const float2 *>(src + 6));
            xd[u] = __ldcs(reinterpret_cast<const float4 *>(src + 8));
        }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
        if (dst[u] < 0) continue;
        const float v0 = in0[u] ? interval_sum(xa[u].x, xa[u].y, xa[u].z, xa[u].w, xb[u].x, xb[u].y) : 0.0f;
        const float v1 = in1[u] ? interval_sum(xc[u].x, xc[u].y, xd[u].x, xd[u].y, xd[u].z, xd[u].w) : 0.0f;
        store2<FMT>(img, dst[u], v0, v1, true);
    }
}

}  // namespace

cudaError_t launch_interval_images(const ReqTable &t, void *dimg, emtk_patch_format fmt, cudaStream_t s,
                                   const DescJob *job) {
    int64_t most = 0;
    for (int i = 0; i < t.n; ++i) {
        const int64_t w = t.r[i].nwires ? (int64_t)(t.r[i].nwires + 2 * t.r[i].halo) * (t.r[i].pitch / 2) : 0;
        most = w > most ? w : most;
    }
    if (job != nullptr && job->count > 0) {
        if (most == 0 || t.n == 0)  // no image to cut: the descriptors alone
            return launch_hit_desc(t, job->g0, job->count, job->desc, job->dest, job->out_stride, s);
        const int64_t want = most > job->count ? most : job->count;
        int64_t bx = (want + 255) / 256;
        if (bx > 4096) bx = 4096;
        dim3 grid((unsigned)bx, (unsigned)t.n + 1);
        if (fmt == kPatchSplit16)
            interval_desc_kernel<kPatchSplit16><<<grid, 256, 0, s>>>(t, dimg, job->g0, job->count, job->desc,
                                                                     job->dest, job->out_stride);
        else if (fmt == EMTK_PATCH_F32)
            interval_desc_kernel<EMTK_PATCH_F32><<<grid, 256, 0, s>>>(t, dimg, job->g0, job->count, job->desc,
                                                                      job->dest, job->out_stride);
        else if (fmt == EMTK_PATCH_BF16)
            interval_desc_kernel<EMTK_PATCH_BF16><<<grid, 256, 0, s>>>(t, dimg, job->g0, job->count, job->desc,
                                                                       job->dest, job->out_stride);
        else
            interval_desc_kernel<EMTK_PATCH_F16><<<grid, 256, 0, s>>>(t, dimg, job->g0, job->count, job->desc,
                                                                      job->dest, job->out_stride);
        return cudaGetLastError();
    }
    if (most == 0 || t.n == 0) return cudaSuccess;
    int64_t bx = (most + 255) / 256;
    if (bx > 4096) bx = 4096;
    dim3 grid((unsigned)bx, (unsigned)t.n);
    if (fmt == kPatchSplit16)
        interval_image_kernel<kPatchSplit16><<<grid, 256, 0, s>>>(t, dimg);
    else if (fmt == EMTK_PATCH_F32)
        interval_image_kernel<EMTK_PATCH_F32><<<grid, 256, 0, s>>>(t, dimg);
    else if (fmt == EMTK_PATCH_BF16)
        interval_image_kernel<EMTK_PATCH_BF16><<<grid, 256, 0, s>>>(t, dimg);
    else
        interval_image_kernel<EMTK_PATCH_F16><<<grid, 256, 0, s>>>(t, dimg);
    return cudaGetLastError();
}

cudaError_t launch_cut_tiles(const ReqTable &t, int64_t total_hits, void *dimg, emtk_patch_format fmt,
                             const DescJob &job, uint32_t *mask_cur, uint32_t *mask_next, int64_t mask_cap,
                             cudaStream_t s) {
    if (total_hits <= 0 || t.n == 0) return cudaSuccess;
    int64_t most_hits = 0, most_words = 0;
    for (int i = 0; i < t.n; ++i) {
        const ReqDesc &r = t.r[i];
        most_hits = r.nhits > most_hits ? r.nhits : most_hits;
        const int64_t rows = r.nwires > 0 ? (int64_t)r.nwires + 2 * r.halo : 0;
        const int64_t words = (rows + kTileRows - 1) / kTileRows * r.m_wpb;
        most_words = words > most_words ? words : most_words;
    }
    int64_t mb = (most_hits + 255) / 256;
    if (mb > 4096) mb = 4096;
    const int smem_words = (int)(most_words < kMarkSmemWords ? most_words : kMarkSmemWords);
    mark_tiles_kernel<<<dim3((unsigned)(mb > 0 ? mb : 1), (unsigned)t.n), 256, (size_t)smem_words * 4, s>>>(
        t, mask_cur, smem_words);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int64_t most = 0;  // tiles of the largest image
    for (int i = 0; i < t.n; ++i) {
        const ReqDesc &r = t.r[i];
        if (r.nwires == 0) continue;
        const int64_t tiles = (((int64_t)r.nwires + 2 * r.halo + kTileRows - 1) / kTileRows) *
                              ((r.pitch + kTileInts - 1) / kTileInts);
        most = tiles > most ? tiles : most;
    }
    int64_t bx = (most + kTileWarps - 1) / kTileWarps;
    const int64_t desc_blocks = (job.count + kTileWarps * 32 - 1) / (kTileWarps * 32);
    bx = bx > desc_blocks ? bx : desc_blocks;
    bx = bx > 0 ? bx : 1;
    const dim3 grid((unsigned)bx, (unsigned)t.n + 1);  // the last row builds the descriptors
    const uint32_t *mc = mask_cur;
    if (fmt == kPatchSplit16)
        return launch_pdl(interval_tiles_kernel<kPatchSplit16>, grid, dim3(kTileWarps * 32), 0, s, t, dimg, mc,
                          mask_next, mask_cap, job.g0, job.count, job.desc, job.dest, job.out_stride);
    if (fmt == EMTK_PATCH_F16)
        return launch_pdl(interval_tiles_kernel<EMTK_PATCH_F16>, grid, dim3(kTileWarps * 32), 0, s, t, dimg, mc,
                          mask_next, mask_cap, job.g0, job.count, job.desc, job.dest, job.out_stride);
    return launch_pdl(interval_tiles_kernel<EMTK_PATCH_BF16>, grid, dim3(kTileWarps * 32), 0, s, t, dimg, mc,
                      mask_next, mask_cap, job.g0, job.count, job.desc, job.dest, job.out_stride);
}

cudaError_t launch_gather(const ReqTable &t, const void *dimg, emtk_patch_format fmt, int64_t g0, int32_t count,
                          void *patches, float **dest, int out_stride, cudaStream_t s) {
    if (count <= 0) return cudaSuccess;
    if (fmt == EMTK_PATCH_F32)
        gather_kernel<EMTK_PATCH_F32><<<count, 288, 0, s>>>(t, dimg, g0, patches, dest, out_stride);
    else if (fmt == EMTK_PATCH_BF16)
        gather_kernel<EMTK_PATCH_BF16><<<count, 288, 0, s>>>(t, dimg, g0, patches, dest, out_stride);
    else
        gather_kernel<EMTK_PATCH_F16><<<count, 288, 0, s>>>(t, dimg, g0, patches, dest, out_stride);
    return cudaGetLastError();
}

cudaError_t launch_convert_split(const float *src, void *dst, int64_t n, int sms, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int64_t n8 = n / 8;
    int64_t blocks = (n8 + 256 * 4 - 1) / (256 * 4);
    if (blocks > (int64_t)sms * 8) blocks = (int64_t)sms * 8;
    if (blocks < 1) blocks = 1;
    convert_split_kernel<<<(unsigned)blocks, 256, 0, s>>>(src, static_cast<uint4 *>(dst), n8);
    return cudaGetLastError();
}

cudaError_t launch_hit_desc(const ReqTable &t, int64_t g0, int32_t count, HitDesc *desc, float **dest,
                            int out_stride, cudaStream_t s) {
    if (count <= 0) return cudaSuccess;
    hit_desc_kernel<<<(count + 255) / 256, 256, 0, s>>>(t, g0, count, desc, dest, out_stride);
    return cudaGetLastError();
}

}  // namespace emtk
