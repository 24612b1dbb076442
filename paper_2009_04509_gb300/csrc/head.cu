// Network tail (Sec. 2.2), fp32: sum of the dense-1 partial-sum rows in row
// order + bias + ReLU, dense 128->32 + ReLU, the 3-way softmax head (track,
// em, none) and the Michel sigmoid head.  One warp per hit; lane l owns
// dense-1 outputs 4l..4l+3 and dense-2 output l.  The rows of a hit are the
// K-splits of the fp32 path, or the stream-K CTAs that shared its tile.
#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kWarps = 8;
constexpr int kHitsPerWarp = 8;  // each block stages the tail weights once for 64 hits

__global__ void __launch_bounds__(kWarps * 32) head_kernel(const float *__restrict__ partials, int splits, int G, int n_pad,
                                                          int32_t n, const float *__restrict__ fc1_b,
                                                          const float *__restrict__ fc2_w,
                                                          const float *__restrict__ fc2_b,
                                                          const float *__restrict__ cls_w,
                                                          const float *__restrict__ cls_b,
                                                          const float *__restrict__ mic_w,
                                                          const float *__restrict__ mic_b, float *const *dest,
                                                          int debug_logits) {
    __shared__ float w2[kN1][kN2];
    __shared__ float wc[kN2][kNC + 1];
    for (int i = threadIdx.x; i < kN1 * kN2; i += blockDim.x) w2[i / kN2][i % kN2] = fc2_w[i];
    for (int i = threadIdx.x; i < kN2 * kNC; i += blockDim.x) wc[i / kNC][i % kNC] = cls_w[i];
    for (int i = threadIdx.x; i < kN2; i += blockDim.x) wc[i][kNC] = mic_w[i];
    __syncthreads();

    const int lane = threadIdx.x & 31;
    for (int j = 0; j < kHitsPerWarp; ++j) {
    const int64_t h = ((int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5)) * kHitsPerWarp + j;
    if (h >= n) return;

    int rows = splits;
    if (G > 0) {
        const int64_t units = (int64_t)((n + 127) / 128) * kQuads;
        const int64_t tile = h >> 7;
        rows = cta_of_unit(tile * kQuads + kQuads - 1, units, G) - cta_of_unit(tile * kQuads, units, G) + 1;
    }
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s = 0; s < rows; ++s) {
        const float4 v = __ldcs(reinterpret_cast<const float4 *>(partials + ((int64_t)s * n_pad + h) * kN1) + lane);
        a.x += v.x;
        a.y += v.y;
        a.z += v.z;
        a.w += v.w;
    }
    const float4 b1 = reinterpret_cast<const float4 *>(fc1_b)[lane];
    float h1[4] = {fmaxf(a.x + b1.x, 0.f), fmaxf(a.y + b1.y, 0.f), fmaxf(a.z + b1.z, 0.f), fmaxf(a.w + b1.w, 0.f)};

    float h2 = fc2_b[lane];
    for (int l = 0; l < 32; ++l) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float v = __shfl_sync(0xffffffffu, h1[e], l);
            h2 = fmaf(v, w2[4 * l + e][lane], h2);
        }
    }
    h2 = fmaxf(h2, 0.f);

    float z[kNC + 1];
#pragma unroll
    for (int c = 0; c <= kNC; ++c) {
        float v = h2 * wc[lane][c];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        z[c] = v;
    }
    if (lane == 0) {
#pragma unroll
        for (int c = 0; c < kNC; ++c) z[c] += cls_b[c];
        z[kNC] += mic_b[0];
        const float m = fmaxf(fmaxf(z[0], z[1]), z[2]);
        const float e0 = expf(z[0] - m), e1 = expf(z[1] - m), e2 = expf(z[2] - m);
        const float sum = e0 + e1 + e2;
        float *out = dest[h];
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
    }
}

}  // namespace

cudaError_t launch_head(const DeviceWeights &w, const float *partials, int splits, int G, int n_pad, int32_t n,
                        float *const *dest, int debug_logits, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int per_block = kWarps * kHitsPerWarp;
    head_kernel<<<(n + per_block - 1) / per_block, kWarps * 32, 0, s>>>(partials, splits, G, n_pad, n, w.fc1_b, w.fc2_w,
                                                                  w.fc2_b, w.cls_w, w.cls_b, w.mic_w, w.mic_b,
                                                                  dest, debug_logits);
    return cudaGetLastError();
}

}  // namespace emtk
