// fp32 network path on CUDA cores (EMTK_FP32): conv 5x5x48 + ReLU fused
// with dense-1 (Sec. 2.2), split over the dense-1 input dimension.
//
// Block = 32 hits x one segment of conv positions.  Per position the block
// computes the 32 x 48 conv activations into shared memory from a 5-row
// band of the 32 patches, stages the 48 x 128 dense-1 rows of that position
// and accumulates 2 hits x 8 outputs per thread in fp32.  Segment partial
// sums go to partials[segment][hit][128]; the head kernel adds them in
// segment order, so results are deterministic.
#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kHT = 32;      // hits per block
constexpr int kThreads = 256;
constexpr int kSmemBytes = (kF * kN1 + kK * kHT * kPatch + kHT * (kF + 1) + kK * kK * kF + kF) * 4;

__global__ void __launch_bounds__(kThreads) cnn_fp32_kernel(const float *__restrict__ patches, int n,
                                                            const float *__restrict__ conv_w,
                                                            const float *__restrict__ conv_b,
                                                            const float *__restrict__ fc1_w, int splits,
                                                            float *__restrict__ partials, int n_pad) {
    extern __shared__ float4 smem_f4[];
    auto &w1s = *reinterpret_cast<float (*)[kF][kN1]>(smem_f4);
    auto &band = *reinterpret_cast<float (*)[kK][kHT][kPatch]>(&w1s[kF][0]);  // rows by (row % 5)
    auto &act = *reinterpret_cast<float (*)[kHT][kF + 1]>(&band[kK][0][0]);
    auto &cw = *reinterpret_cast<float (*)[kK * kK][kF]>(&act[kHT][0]);
    float *cb = &cw[kK * kK][0];

    const int tid = threadIdx.x;
    const int hit0 = blockIdx.x * kHT;
    const int seg = blockIdx.y;
    const int p_begin = (int)((int64_t)seg * kPos / splits);
    const int p_end = (int)((int64_t)(seg + 1) * kPos / splits);

    for (int i = tid; i < kK * kK * kF; i += kThreads) cw[i / kF][i % kF] = conv_w[i];
    for (int i = tid; i < kF; i += kThreads) cb[i] = conv_b[i];

    // dense-1 mapping: hits 2*hp, 2*hp+1; outputs n0..n0+7
    const int hp = tid >> 4;
    const int n0 = (tid & 15) * 8;
    float acc[2][8];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[a][e] = 0.0f;

    // conv mapping: hit ch = tid >> 3, filters c0..c0+5
    const int ch = tid >> 3;
    const int c0 = (tid & 7) * 6;

    int band_y = -100;  // first patch row held in band
    for (int p = p_begin; p < p_end; ++p) {
        const int y = p / kQ;
        const int x = p - y * kQ;
        if (y != band_y) {
            __syncthreads();
            for (int i = tid; i < kK * kHT * kPatch; i += kThreads) {
                const int rr = i / (kHT * kPatch);
                const int rem = i - rr * kHT * kPatch;
                const int h = rem / kPatch;
                const int col = rem - h * kPatch;
                const int prow = y + rr;
                const int gh = hit0 + h;
                band[prow % kK][h][col] = gh < n ? patches[(int64_t)gh * kPatchElems + prow * kPatch + col] : 0.0f;
            }
            band_y = y;
        }
        // stage the 48 x 128 dense-1 rows of this position
        const float4 *src = reinterpret_cast<const float4 *>(fc1_w + (int64_t)p * kF * kN1);
        for (int i = tid; i < kF * kN1 / 4; i += kThreads)
            reinterpret_cast<float4 *>(&w1s[0][0])[i] = __ldg(src + i);
        __syncthreads();
        // conv + ReLU for (hit ch, filters c0..c0+5)
        float s[6];
#pragma unroll
        for (int f = 0; f < 6; ++f) s[f] = cb[c0 + f];
#pragma unroll
        for (int i = 0; i < kK; ++i) {
            const float *row = &band[(y + i) % kK][ch][x];
#pragma unroll
            for (int j = 0; j < kK; ++j) {
                const float v = row[j];
#pragma unroll
                for (int f = 0; f < 6; ++f) s[f] = fmaf(v, cw[i * kK + j][c0 + f], s[f]);
            }
        }
#pragma unroll
        for (int f = 0; f < 6; ++f) act[ch][c0 + f] = fmaxf(s[f], 0.0f);
        __syncthreads();
        // dense-1 accumulate
#pragma unroll 4
        for (int c = 0; c < kF; ++c) {
            const float a0 = act[2 * hp][c];
            const float a1 = act[2 * hp + 1][c];
            const float4 wa = *reinterpret_cast<const float4 *>(&w1s[c][n0]);
            const float4 wb = *reinterpret_cast<const float4 *>(&w1s[c][n0 + 4]);
            const float w[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                acc[0][e] = fmaf(a0, w[e], acc[0][e]);
                acc[1][e] = fmaf(a1, w[e], acc[1][e]);
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 2; ++a) {
        const int gh = hit0 + 2 * hp + a;
        if (gh < n) {
            float *dst = partials + ((int64_t)seg * n_pad + gh) * kN1 + n0;
            reinterpret_cast<float4 *>(dst)[0] = make_float4(acc[a][0], acc[a][1], acc[a][2], acc[a][3]);
            reinterpret_cast<float4 *>(dst)[1] = make_float4(acc[a][4], acc[a][5], acc[a][6], acc[a][7]);
        }
    }
}

}  // namespace

cudaError_t init_fp32_kernel_attrs() {
    return cudaFuncSetAttribute(cnn_fp32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
}

int choose_splits_fp32(int n, int sm_count, int max_splits) {
    const int blocks = (n + kHT - 1) / kHT;
    int s = (2 * sm_count + blocks - 1) / blocks;
    if (s > kPos / 16) s = kPos / 16;
    if (s > max_splits) s = max_splits;
    return s < 1 ? 1 : s;
}

cudaError_t launch_cnn_fp32(const DeviceWeights &w, const float *patches, int32_t n, int splits, float *partials,
                            int n_pad, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    dim3 grid((n + kHT - 1) / kHT, splits);
    cnn_fp32_kernel<<<grid, kThreads, kSmemBytes, s>>>(patches, n, w.conv_w, w.conv_b, w.fc1_w, splits, partials, n_pad);
    return cudaGetLastError();
}

}  // namespace emtk
