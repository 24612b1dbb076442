// Network tail (Sec. 2.2), fp32: sum of the dense-1 partial-sum rows in row
// order, times the dense-1 scale s1 (1, or the inverse of the operand scales
// of the e4m3 path), + bias + ReLU, dense 128->32 + ReLU, the 3-way softmax
// head (track, em, none) and the Michel sigmoid head.  The rows of a hit are
// the K-splits of the fp32 path, or the stream-K CTAs that shared its tile.
// Three kernels, chosen by launch_head, with the same sums in the same order
// (so the same bits), except where noted:
//   head_kernel       small launches with few rows: a thread per hit streams
//                     its dense-1 outputs four at a time into the 32 dense-2
//                     sums (weights broadcast from shared memory);
//   head_rows_kernel  many rows per hit (small launches spread each tile
//                     over many CTAs): a warp per hit sums the rows, 16 deep
//                     (from 32 rows on, four warps per hit each sum a
//                     quarter of the rows and the quarters are added in
//                     order: the same bits run to run, a different rounding
//                     order than the other two kernels);
//   head_tile_kernel  large launches: one CTA per 128-hit tile (coalesced
//                     row sums, a register-tiled dense-2).
#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kThreadsHead = 128;

__device__ __forceinline__ unsigned long long global_timer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// The dense-2 weights [128][32] into shared memory (16-byte aligned): every
// load issued before the first store, so that staging costs one round trip.
template <int kThreads>
__device__ __forceinline__ void stage_w2(float *w2, const float *__restrict__ fc2_w) {
    constexpr int kN4 = kN1 * kN2 / 4;
    static_assert(kN4 % kThreads == 0, "whole float4s per thread");
    float4 v[kN4 / kThreads];
#pragma unroll
    for (int k = 0; k < kN4 / kThreads; ++k)
        v[k] = __ldg(reinterpret_cast<const float4 *>(fc2_w) + threadIdx.x + k * kThreads);
#pragma unroll
    for (int k = 0; k < kN4 / kThreads; ++k) reinterpret_cast<float4 *>(w2)[threadIdx.x + k * kThreads] = v[k];
}
constexpr int kManyRows = 4;  // above this many partial rows per hit, reduce them with a warp per hit
constexpr int kSplitRows = 32;  // from this many, with four warps per hit

__global__ void __launch_bounds__(kThreadsHead) head_kernel(const float *__restrict__ partials, int splits, int G,
                                                           int n_pad, int32_t n, float s1,
                                                           const float *__restrict__ fc1_b,
                                                           const float *__restrict__ fc2_w,
                                                           const float *__restrict__ fc2_b,
                                                           const float *__restrict__ cls_w,
                                                           const float *__restrict__ cls_b,
                                                           const float *__restrict__ mic_w,
                                                           const float *__restrict__ mic_b, OutRows out_rows,
                                                           int debug_logits) {
    __shared__ __align__(16) float w2[kN1][kN2];
    __shared__ __align__(16) float wc[kN2][kNC + 1];
    __shared__ __align__(16) float b1[kN1];
    __shared__ float b2[kN2];
    stage_w2<kThreadsHead>(&w2[0][0], fc2_w);
    for (int i = threadIdx.x; i < kN2 * kNC; i += blockDim.x) wc[i / kNC][i % kNC] = cls_w[i];
    for (int i = threadIdx.x; i < kN2; i += blockDim.x) {
        wc[i][kNC] = mic_w[i];
        b2[i] = fc2_b[i];
    }
    for (int i = threadIdx.x; i < kN1; i += blockDim.x) b1[i] = fc1_b[i];
    pdl_wait();  // the partial sums and output rows come from the kernels before
    __syncthreads();

    const int64_t h = (int64_t)blockIdx.x * kThreadsHead + threadIdx.x;
    if (h >= n) return;
    int rows = splits;
    if (G > 0) {
        const int64_t units = (int64_t)((n + 127) / 128) * kQuads;
        const int64_t tile = h >> 7;
        rows = cta_of_unit(tile * kQuads + kQuads - 1, units, G) - cta_of_unit(tile * kQuads, units, G) + 1;
    }

    float h2[kN2];
#pragma unroll
    for (int j = 0; j < kN2; ++j) h2[j] = b2[j];
    const float4 *prow = reinterpret_cast<const float4 *>(partials + h * kN1);
    const int64_t row_stride = (int64_t)n_pad * kN1 / 4;  // float4s between partial rows
#pragma unroll 2
    for (int c = 0; c < kN1 / 4; ++c) {
        float4 a = prow[c];
        for (int s = 1; s < rows; ++s) {
            const float4 v = prow[s * row_stride + c];
            a.x += v.x;
            a.y += v.y;
            a.z += v.z;
            a.w += v.w;
        }
        const float4 bb = *reinterpret_cast<const float4 *>(&b1[4 * c]);
        // s1 is a power of two: a * s1 + b rounds once, as a + b does for s1 = 1
        const float h1[4] = {fmaxf(fmaf(a.x, s1, bb.x), 0.f), fmaxf(fmaf(a.y, s1, bb.y), 0.f),
                             fmaxf(fmaf(a.z, s1, bb.z), 0.f), fmaxf(fmaf(a.w, s1, bb.w), 0.f)};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float4 *wr = reinterpret_cast<const float4 *>(&w2[4 * c + e][0]);
#pragma unroll
            for (int q = 0; q < kN2 / 4; ++q) {
                const float4 wv = wr[q];
                h2[4 * q + 0] = fmaf(h1[e], wv.x, h2[4 * q + 0]);
                h2[4 * q + 1] = fmaf(h1[e], wv.y, h2[4 * q + 1]);
                h2[4 * q + 2] = fmaf(h1[e], wv.z, h2[4 * q + 2]);
                h2[4 * q + 3] = fmaf(h1[e], wv.w, h2[4 * q + 3]);
            }
        }
    }
    float z[kNC + 1] = {cls_b[0], cls_b[1], cls_b[2], mic_b[0]};
#pragma unroll
    for (int j = 0; j < kN2; ++j) {
        const float v = fmaxf(h2[j], 0.f);
        const float4 wv = *reinterpret_cast<const float4 *>(&wc[j][0]);
        z[0] = fmaf(v, wv.x, z[0]);
        z[1] = fmaf(v, wv.y, z[1]);
        z[2] = fmaf(v, wv.z, z[2]);
        z[3] = fmaf(v, wv.w, z[3]);
    }
    const float m = fmaxf(fmaxf(z[0], z[1]), z[2]);
    const float e0 = expf(z[0] - m), e1 = expf(z[1] - m), e2 = expf(z[2] - m);
    const float sum = e0 + e1 + e2;
    float *out = out_rows.rows ? out_rows.rows + h * (int64_t)out_rows.stride : out_rows.dest[h];
    out[0] = e0 / sum;
    out[1] = e1 / sum;
    out[2] = e2 / sum;
    out[3] = 1.0f / (1.0f + expf(-z[kNC]));
    if (debug_logits) {
        out[4] = z[0];
        out[5] = z[1];
        out[6] = z[2];
        out[7] = z[3];
    }
}

// The same tail when a hit has many partial rows (a small launch, whose
// tiles are split over many CTAs): one warp per hit sums the rows, lane l
// taking dense-1 outputs 4l .. 4l+3 of every row (512 contiguous bytes per
// row), and writes bias + ReLU to shared memory; every thread then computes
// dense-2 outputs (one per hit and output), and one thread per hit the heads.  HITS hits per block: 8 for small launches (more
// blocks, so more rows summed at once), 32 above kSmallLaunch hits (fewer
// blocks loading the dense-2 weights).
constexpr int kThreadsRows = 256;
constexpr int kSmallLaunch = 2048;
constexpr int kH1Stride = kN1 + 1;  // shared h1 rows padded: thread t reads row t conflict-free

// kSplit warps share a hit: warp k of the hit sums its rows [k R / kSplit,
// (k+1) R / kSplit) in order, and the kSplit partial sums are then added in
// k order (kSplit = 1: all rows in order, as head_kernel does).  More warps
// per hit put more of the GPU on a small launch's many rows.
template <int kHitsRows, int kSplit = 1>
__global__ void __launch_bounds__(kThreadsRows) head_rows_kernel(const float *__restrict__ partials, int splits,
                                                                int G, int n_pad, int32_t n, float s1,
                                                                const float *__restrict__ fc1_b,
                                                                const float *__restrict__ fc2_w,
                                                                const float *__restrict__ fc2_b,
                                                                const float *__restrict__ cls_w,
                                                                const float *__restrict__ cls_b,
                                                                const float *__restrict__ mic_w,
                                                                const float *__restrict__ mic_b, OutRows out_rows,
                                                                int debug_logits) {
    static_assert(kHitsRows * kSplit <= kThreadsRows / 32 || kSplit == 1, "a warp per (hit, row share)");
    __shared__ float h1s[kHitsRows * kH1Stride];
    __shared__ __align__(16) float4 part[kSplit > 1 ? kHitsRows * kSplit * 32 : 1];
    __shared__ float h2s[kHitsRows * (kN2 + 1)];
    __shared__ __align__(16) float w2[kN1][kN2];
    __shared__ __align__(16) float wc[kN2][kNC + 1];
    __shared__ float b2[kN2];
    stage_w2<kThreadsRows>(&w2[0][0], fc2_w);
    for (int i = threadIdx.x; i < kN2 * kNC; i += blockDim.x) wc[i / kNC][i % kNC] = cls_w[i];
    for (int i = threadIdx.x; i < kN2; i += blockDim.x) {
        wc[i][kNC] = mic_w[i];
        b2[i] = fc2_b[i];
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    pdl_wait();  // the partial sums and output rows come from the kernels before
    const int64_t h0 = (int64_t)blockIdx.x * kHitsRows;
    const int64_t row_stride = (int64_t)n_pad * kN1 / 4;  // float4s between partial rows
    const float4 bb = reinterpret_cast<const float4 *>(fc1_b)[lane];
    for (int jw = warp; jw < kHitsRows * kSplit; jw += kThreadsRows / 32) {
        const int j = jw / kSplit, share = jw % kSplit;
        const int64_t h = h0 + j;
        if (h >= n) {
            if (kSplit > 1) continue;
            break;
        }
        int rows = splits;
        if (G > 0) {
            const int64_t units = (int64_t)((n + 127) / 128) * kQuads;
            const int64_t tile = h >> 7;
            rows = cta_of_unit(tile * kQuads + kQuads - 1, units, G) - cta_of_unit(tile * kQuads, units, G) + 1;
        }
        const int r_end = (int)((int64_t)rows * (share + 1) / kSplit);
        const float4 *p = reinterpret_cast<const float4 *>(partials + h * kN1) + lane;
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
        // this warp's rows in order, loaded kDepth at a time (the last batch
        // predicated), so that a hit's rows cost one round trip per kDepth rows
        constexpr int kDepth = 16;
        for (int r = (int)((int64_t)rows * share / kSplit); r < r_end; r += kDepth) {
            float4 v[kDepth];
#pragma unroll
            for (int k = 0; k < kDepth; ++k)
                if (r + k < r_end) v[k] = p[(r + k) * row_stride];
#pragma unroll
            for (int k = 0; k < kDepth; ++k) {
                if (r + k < r_end) {
                    a.x += v[k].x;
                    a.y += v[k].y;
                    a.z += v[k].z;
                    a.w += v[k].w;
                }
            }
        }
        if (kSplit > 1) {
            part[jw * 32 + lane] = a;
            continue;
        }
        float *o = h1s + j * kH1Stride + 4 * lane;
        o[0] = fmaxf(fmaf(a.x, s1, bb.x), 0.f);
        o[1] = fmaxf(fmaf(a.y, s1, bb.y), 0.f);
        o[2] = fmaxf(fmaf(a.z, s1, bb.z), 0.f);
        o[3] = fmaxf(fmaf(a.w, s1, bb.w), 0.f);
    }
    if (kSplit > 1) {  // the shares of each hit, added in share order
        __syncthreads();
        for (int jw = warp; jw < kHitsRows; jw += kThreadsRows / 32) {
            float4 a = part[(jw * kSplit) * 32 + lane];
#pragma unroll
            for (int k = 1; k < kSplit; ++k) {
                const float4 v = part[(jw * kSplit + k) * 32 + lane];
                a.x += v.x;
                a.y += v.y;
                a.z += v.z;
                a.w += v.w;
            }
            float *o = h1s + jw * kH1Stride + 4 * lane;
            o[0] = fmaxf(fmaf(a.x, s1, bb.x), 0.f);
            o[1] = fmaxf(fmaf(a.y, s1, bb.y), 0.f);
            o[2] = fmaxf(fmaf(a.z, s1, bb.z), 0.f);
            o[3] = fmaxf(fmaf(a.w, s1, bb.w), 0.f);
        }
    }
    __syncthreads();
    // dense-2 with every thread: output j of hit i is thread (32 i + j) mod 256's,
    // the same fmaf chain over k as head_kernel's
    for (int o = threadIdx.x; o < kHitsRows * kN2; o += kThreadsRows) {
        const int i = o / kN2, j = o % kN2;
        const float *h1 = h1s + i * kH1Stride;
        float acc = b2[j];
#pragma unroll 8
        for (int k = 0; k < kN1; ++k) acc = fmaf(h1[k], w2[k][j], acc);
        h2s[i * (kN2 + 1) + j] = acc;
    }
    __syncthreads();
    if (threadIdx.x >= kHitsRows) return;
    const int64_t h = h0 + threadIdx.x;
    if (h >= n) return;
    const float *h2 = h2s + threadIdx.x * (kN2 + 1);
    float z[kNC + 1] = {cls_b[0], cls_b[1], cls_b[2], mic_b[0]};
#pragma unroll
    for (int j = 0; j < kN2; ++j) {
        const float v = fmaxf(h2[j], 0.f);
        const float4 wv = *reinterpret_cast<const float4 *>(&wc[j][0]);
        z[0] = fmaf(v, wv.x, z[0]);
        z[1] = fmaf(v, wv.y, z[1]);
        z[2] = fmaf(v, wv.z, z[2]);
        z[3] = fmaf(v, wv.w, z[3]);
    }
    const float m = fmaxf(fmaxf(z[0], z[1]), z[2]);
    const float e0 = expf(z[0] - m), e1 = expf(z[1] - m), e2 = expf(z[2] - m);
    const float sum = e0 + e1 + e2;
    float *out = out_rows.rows ? out_rows.rows + h * (int64_t)out_rows.stride : out_rows.dest[h];
    out[0] = e0 / sum;
    out[1] = e1 / sum;
    out[2] = e2 / sum;
    out[3] = 1.0f / (1.0f + expf(-z[kNC]));
    if (debug_logits) {
        out[4] = z[0];
        out[5] = z[1];
        out[6] = z[2];
        out[7] = z[3];
    }
}

// The tail of a large launch with few partial rows per hit: one CTA per
// 128-hit tile (every hit of a tile has the same rows), 256 threads.
//   1. warp w sums the rows of hits 16w .. 16w+15, lane l taking dense-1
//      outputs l, l+32, l+64, l+96 (four coalesced 128-byte reads per row),
//      and writes bias + ReLU transposed, h1t[k][hit];
//   2. dense-2: thread (hit group tid % 32, output group tid / 32) keeps 4
//      hits x 4 outputs, reading 4 activations and 4 weights (a broadcast)
//      per input k; sums to h2s[hit][j];
//   3. a thread per hit: ReLU, the heads.
// Sums run in the same order as head_kernel's (rows in order; k in order for
// every output), so all three kernels give the same bits.
constexpr int kTileHits = 128;
constexpr int kThreadsTile = 256;
constexpr int kH1tStride = kTileHits + 4;  // rows of h1t: 16-byte aligned, banks shifted per k

__global__ void __launch_bounds__(kThreadsTile) head_tile_kernel(const float *__restrict__ partials, int splits,
                                                                int G, int n_pad, int32_t n, float s1,
                                                                const float *__restrict__ fc1_b,
                                                                const float *__restrict__ fc2_w,
                                                                const float *__restrict__ fc2_b,
                                                                const float *__restrict__ cls_w,
                                                                const float *__restrict__ cls_b,
                                                                const float *__restrict__ mic_w,
                                                                const float *__restrict__ mic_b, OutRows out_rows,
                                                                int debug_logits, int *tile_done, int *status,
                                                                long long timeout_ns) {
    extern __shared__ __align__(16) float tsm[];
    float *h1t = tsm;                                    // [kN1][kH1tStride]
    float *w2 = h1t + kN1 * kH1tStride;                  // [kN1][kN2]
    float *h2s = w2 + kN1 * kN2;                         // [kTileHits][kN2 + 1]
    __shared__ __align__(16) float wc[kN2][kNC + 1];
    __shared__ float b2[kN2];
    __shared__ int go;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    stage_w2<kThreadsTile>(w2, fc2_w);
    for (int i = tid; i < kN2 * kNC; i += kThreadsTile) wc[i / kNC][i % kNC] = cls_w[i];
    for (int i = tid; i < kN2; i += kThreadsTile) {
        wc[i][kNC] = mic_w[i];
        b2[i] = fc2_b[i];
    }
    const int64_t h0 = (int64_t)blockIdx.x * kTileHits;
    const int64_t tile = h0 >> 7;
    int rows = splits;
    if (G > 0) {
        const int64_t units = (int64_t)((n + 127) / 128) * kQuads;
        rows = cta_of_unit(tile * kQuads + kQuads - 1, units, G) - cta_of_unit(tile * kQuads, units, G) + 1;
    }
    if (tile_done != nullptr) {
        // the tile's partial rows are complete once the 4 epilogue warps of each of its `rows`
        // CTAs counted theirs; the output rows were written before those CTAs read their
        // windows.  Every network CTA is running (this kernel is scheduled after all of them
        // started), so the wait ends unless the network kernel gave up (bit 0 of *status)
        if (tid == 0) {
            int ok = 1;
            const int want = 4 * rows;
            const long long t0 = (long long)global_timer();
            for (;;) {
                int v;
                asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(tile_done + tile) : "memory");
                if (v >= want) break;
                if (*reinterpret_cast<volatile int *>(status) & 1) {
                    ok = 0;
                    break;
                }
                if ((long long)global_timer() - t0 > timeout_ns) {
                    atomicOr(status, 2);
                    ok = 0;
                    break;
                }
                __nanosleep(200);
            }
            go = ok;
        }
        __syncthreads();
        if (!go) {
            if (tid == 0) tile_done[tile] = 0;
            return;
        }
    } else {
        pdl_wait();  // the partial sums and output rows come from the kernels before
    }
    const int64_t row_stride = (int64_t)n_pad * kN1;  // floats between partial rows
    float bb[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) bb[e] = fc1_b[lane + 32 * e];
    // the warp's hits warp, warp + 8, ...: eight at a time, so that 32 loads per lane
    // are in flight before the first is used
    constexpr int kBatch = 8;
    for (int j0 = warp; j0 < kTileHits; j0 += kBatch * (kThreadsTile / 32)) {
        float a[kBatch][4];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int64_t h = h0 + j0 + u * (kThreadsTile / 32);
            const float *p = partials + (h < n ? h : 0) * kN1 + lane;
#pragma unroll
            for (int e = 0; e < 4; ++e) a[u][e] = h < n ? __ldcg(p + 32 * e) : 0.f;
        }
        for (int r = 1; r < rows; ++r) {
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int64_t h = h0 + j0 + u * (kThreadsTile / 32);
                const float *p = partials + (h < n ? h : 0) * kN1 + lane + r * row_stride;
#pragma unroll
                for (int e = 0; e < 4; ++e) a[u][e] += h < n ? __ldcg(p + 32 * e) : 0.f;
            }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u)
#pragma unroll
            for (int e = 0; e < 4; ++e)
                h1t[(lane + 32 * e) * kH1tStride + j0 + u * (kThreadsTile / 32)] = fmaxf(fmaf(a[u][e], s1, bb[e]), 0.f);
    }
    __syncthreads();
    if (tile_done != nullptr && tid == 0) tile_done[tile] = 0;  // the tile's rows are read: zero for the next launch
    {
        const int hg = lane, og = warp;  // hits 4hg .. 4hg+3, outputs 4og .. 4og+3
        float acc[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[i][q] = b2[4 * og + q];
#pragma unroll 4
        for (int k = 0; k < kN1; ++k) {
            const float4 x = *reinterpret_cast<const float4 *>(h1t + k * kH1tStride + 4 * hg);
            const float4 wv = *reinterpret_cast<const float4 *>(w2 + k * kN2 + 4 * og);
            const float xs[4] = {x.x, x.y, x.z, x.w};
            const float ws[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int q = 0; q < 4; ++q) acc[i][q] = fmaf(xs[i], ws[q], acc[i][q]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int q = 0; q < 4; ++q) h2s[(4 * hg + i) * (kN2 + 1) + 4 * og + q] = acc[i][q];
    }
    __syncthreads();
    if (tid >= kTileHits) return;
    const int64_t h = h0 + tid;
    if (h >= n) return;
    const float *h2 = h2s + tid * (kN2 + 1);
    float z[kNC + 1] = {cls_b[0], cls_b[1], cls_b[2], mic_b[0]};
#pragma unroll
    for (int j = 0; j < kN2; ++j) {
        const float v = fmaxf(h2[j], 0.f);
        const float4 wv = *reinterpret_cast<const float4 *>(&wc[j][0]);
        z[0] = fmaf(v, wv.x, z[0]);
        z[1] = fmaf(v, wv.y, z[1]);
        z[2] = fmaf(v, wv.z, z[2]);
        z[3] = fmaf(v, wv.w, z[3]);
    }
    const float m = fmaxf(fmaxf(z[0], z[1]), z[2]);
    const float e0 = expf(z[0] - m), e1 = expf(z[1] - m), e2 = expf(z[2] - m);
    const float sum = e0 + e1 + e2;
    // through L2: the rows were written by a kernel that is not ordered before this one by its launch
    float *out = out_rows.rows ? out_rows.rows + h * (int64_t)out_rows.stride
                               : reinterpret_cast<float *>(
                                     __ldcg(reinterpret_cast<const unsigned long long *>(out_rows.dest + h)));
    out[0] = e0 / sum;
    out[1] = e1 / sum;
    out[2] = e2 / sum;
    out[3] = 1.0f / (1.0f + expf(-z[kNC]));
    if (debug_logits) {
        out[4] = z[0];
        out[5] = z[1];
        out[6] = z[2];
        out[7] = z[3];
    }
}
constexpr int kTileSmem = (kN1 * kH1tStride + kN1 * kN2 + kTileHits * (kN2 + 1)) * 4;

}  // namespace

cudaError_t init_head_kernel_attrs() {
    return cudaFuncSetAttribute(head_tile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTileSmem);
}

bool head_counts_tiles(int32_t n, int G) {
    return G > 0 && n > kSmallLaunch && streamk_partial_rows(n, G) <= kManyRows;
}

cudaError_t launch_head(const DeviceWeights &w, const float *partials, int splits, int G, int n_pad, int32_t n,
                        OutRows out_rows, int debug_logits, int *tile_done, int *status, int64_t timeout_ns,
                        cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    // most partial rows a hit has: many when a small launch spreads each tile over many CTAs
    const int rows = G > 0 ? streamk_partial_rows(n, G) : splits;
    // launched as dependents of the network kernel: the weights are staged while it finishes
    const float s1 = w.fc1_scale;
    const float *b1 = w.fc1_b, *w2 = w.fc2_w, *b2 = w.fc2_b, *wc = w.cls_w, *bc = w.cls_b, *wm = w.mic_w,
                *bm = w.mic_b;
    if (rows > kManyRows) {
        if (rows >= kSplitRows && n <= kSmallLaunch)  // a hit's rows over 4 warps, 2 hits per block
            return launch_pdl(head_rows_kernel<2, 4>, dim3((n + 1) / 2), dim3(kThreadsRows), 0, s, partials, splits,
                              G, n_pad, n, s1, b1, w2, b2, wc, bc, wm, bm, out_rows, debug_logits);
        if (n <= kSmallLaunch)
            return launch_pdl(head_rows_kernel<8>, dim3((n + 7) / 8), dim3(kThreadsRows), 0, s, partials, splits, G,
                              n_pad, n, s1, b1, w2, b2, wc, bc, wm, bm, out_rows, debug_logits);
        return launch_pdl(head_rows_kernel<32>, dim3((n + 31) / 32), dim3(kThreadsRows), 0, s, partials, splits, G,
                          n_pad, n, s1, b1, w2, b2, wc, bc, wm, bm, out_rows, debug_logits);
    }
    if (n > kSmallLaunch) {
        const long long tmo = (long long)timeout_ns;
        return launch_pdl(head_tile_kernel, dim3((n + kTileHits - 1) / kTileHits), dim3(kThreadsTile), kTileSmem, s,
                          partials, splits, G, n_pad, n, s1, b1, w2, b2, wc, bc, wm, bm, out_rows, debug_logits,
                          head_counts_tiles(n, G) ? tile_done : nullptr, status, tmo);
    }
    return launch_pdl(head_kernel, dim3((n + kThreadsHead - 1) / kThreadsHead), dim3(kThreadsHead), 0, s, partials,
                      splits, G, n_pad, n, s1, b1, w2, b2, wc, bc, wm, bm, out_rows, debug_logits);
}

}  // namespace emtk
