// fp32 network path on CUDA cores (EMTK_FP32): conv 5x5x48 + ReLU fused
// with dense-1 (Sec. 2.2), split over the dense-1 input dimension (the conv
// positions) into `splits` segments.
//
// Block = 128 hits x one segment of conv positions, 256 threads.  Per
// position the block
//   - computes the 128 x 48 conv activations (thread: one hit, 24 filters;
//     each warp one half of the filters) from a 5-row band of the hits'
//     patches held in shared memory (rows kept by row % 5, one new row per
//     output row), transposed into act[48][128].  The conv weights are a
//     launch parameter, so the FMAs read them from the constant bank: one
//     shared-memory load per tap and thread;
//   - multiplies them into the dense-1 sums with the position's 48 x 128
//     weights, which cp.async brought into one of two shared buffers while
//     the previous position was computed: thread (hit group g, output group
//     o) accumulates hits 8g..8g+7 x outputs 4o..4o+3 and 64+4o..64+4o+3 in
//     64 registers (the split keeps the weight loads free of bank
//     conflicts), 16 FMAs per shared-memory load.
// Segment partial sums go to partials[segment][hit][128]; the head kernel
// adds them in segment order, so results are deterministic.
#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kHT = 128;      // hits per block
constexpr int kThreads = 256;
constexpr int kBandStride = kPatch + 1;  // 49: conflict-free per-hit reads
constexpr int kW1Pos = kF * kN1;         // 6144 weights of one position (24 KB)
// shared memory: band[5][128][49], w1[2][48][128], act[48][128]
constexpr int kSmemFloats = kK * kHT * kBandStride + 2 * kW1Pos + kF * kHT;
constexpr int kSmemBytes = kSmemFloats * 4;
static_assert(kSmemBytes <= 232448, "shared memory budget");
static_assert(kW1Pos % (4 * kThreads) == 0 && kHT % 32 == 0 && kThreads == 2 * kHT && kThreads / 16 * 8 == kHT,
              "thread layout: two conv filter halves of kHT hits; 16 threads per 8 hits in dense-1");

__device__ __forceinline__ void cp_async16(float *smem_dst, const float *gmem_src) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_prev() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

// The 48 x 128 dense-1 weights of position p into dst (each thread 6 x 16 bytes).
__device__ __forceinline__ void load_w1(float *dst, const float *__restrict__ fc1_w, int p, int tid) {
    const float *src = fc1_w + (int64_t)p * kW1Pos;
#pragma unroll
    for (int k = 0; k < kW1Pos / 4 / kThreads; ++k) {
        const int i = (tid + k * kThreads) * 4;
        cp_async16(dst + i, src + i);
    }
}

// Patch row `prow` of the block's 128 hits into band slot prow % 5 (zero past n).
__device__ __forceinline__ void load_band_row(float *band, const float *__restrict__ patches, int n, int hit0, int prow,
                                              int tid) {
    float *slot = band + (prow % kK) * kHT * kBandStride;
    for (int i = tid; i < kHT * kPatch / 4; i += kThreads) {
        const int h = i / (kPatch / 4), c4 = i - h * (kPatch / 4);
        const int gh = hit0 + h;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (gh < n) v = __ldg(reinterpret_cast<const float4 *>(patches + (int64_t)gh * kPatchElems + prow * kPatch) + c4);
        float *d = slot + h * kBandStride + 4 * c4;
        d[0] = v.x;
        d[1] = v.y;
        d[2] = v.z;
        d[3] = v.w;
    }
}

// The conv weights [25][48] and bias [48], passed by value.
struct ConvParams {
    float w[kK * kK * kF];
    float b[kF];
};

// Conv + ReLU of hit `hit` at position (y, x), filters F0 .. F0+23, into act.
template <int F0>
__device__ __forceinline__ void conv_half(const ConvParams &cp, const float *band, int y, int x, int hit, float *act) {
    float s[24];
#pragma unroll
    for (int f = 0; f < 24; ++f) s[f] = cp.b[F0 + f];
#pragma unroll
    for (int i = 0; i < kK; ++i) {
        const float *row = band + ((y + i) % kK) * kHT * kBandStride + hit * kBandStride + x;
#pragma unroll
        for (int j = 0; j < kK; ++j) {
            const float v = row[j];
#pragma unroll
            for (int f = 0; f < 24; ++f) s[f] = fmaf(v, cp.w[(i * kK + j) * kF + F0 + f], s[f]);
        }
    }
#pragma unroll
    for (int f = 0; f < 24; ++f) act[(F0 + f) * kHT + hit] = fmaxf(s[f], 0.0f);
}

__global__ void __launch_bounds__(kThreads, 1) cnn_fp32_kernel(const float *__restrict__ patches, int n,
                                                               const __grid_constant__ ConvParams cp,
                                                               const float *__restrict__ fc1_w, int splits,
                                                               float *__restrict__ partials, int n_pad) {
    extern __shared__ float4 smem_f4[];
    float *band = reinterpret_cast<float *>(smem_f4);  // [5][128][49]
    float *w1 = band + kK * kHT * kBandStride;          // [2][48][128]
    float *act = w1 + 2 * kW1Pos;                       // [48][128]

    const int tid = threadIdx.x;
    const int hit0 = blockIdx.x * kHT;
    const int seg = blockIdx.y;
    const int p_begin = (int)((int64_t)seg * kPos / splits);
    const int p_end = (int)((int64_t)(seg + 1) * kPos / splits);

    const int g = tid >> 4, o = tid & 15;  // dense-1: hits 8g.., outputs 4o.. and 64+4o..
    const int ch = tid & (kHT - 1);        // conv: hit ch, filter half tid / 128 (one per warp)
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;

    if (p_begin < p_end) load_w1(w1, fc1_w, p_begin, tid);
    cp_async_commit();
    int band_y = -1;
    for (int p = p_begin; p < p_end; ++p) {
        const int y = p / kQ, x = p - y * kQ;
        // the next position's weights into the other buffer (free since the last barrier)
        if (p + 1 < p_end) load_w1(w1 + ((p + 1 - p_begin) & 1) * kW1Pos, fc1_w, p + 1, tid);
        cp_async_commit();
        if (y != band_y) {  // rows y..y+4: all five at the segment's start, then the one new row
            for (int r = band_y < 0 ? y : y + kK - 1; r < y + kK; ++r) load_band_row(band, patches, n, hit0, r, tid);
            band_y = y;
            __syncthreads();
        }
        // conv + ReLU, transposed into act
        if (tid < kHT)
            conv_half<0>(cp, band, y, x, ch, act);
        else
            conv_half<24>(cp, band, y, x, ch, act);
        cp_async_wait_prev();  // this position's weights have landed
        __syncthreads();
        // dense-1: 8 hits x 8 outputs per thread
        const float *wp = w1 + ((p - p_begin) & 1) * kW1Pos;
#pragma unroll 4
        for (int c = 0; c < kF; ++c) {
            const float4 a0 = *reinterpret_cast<const float4 *>(act + c * kHT + 8 * g);
            const float4 a1 = *reinterpret_cast<const float4 *>(act + c * kHT + 8 * g + 4);
            const float4 b0 = *reinterpret_cast<const float4 *>(wp + c * kN1 + 4 * o);
            const float4 b1 = *reinterpret_cast<const float4 *>(wp + c * kN1 + 64 + 4 * o);
            const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int gh = hit0 + 8 * g + i;
        if (gh < n) {
            float *dst = partials + ((int64_t)seg * n_pad + gh) * kN1;
            reinterpret_cast<float4 *>(dst + 4 * o)[0] = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
            reinterpret_cast<float4 *>(dst + 64 + 4 * o)[0] = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
        }
    }
}

}  // namespace

cudaError_t init_fp32_kernel_attrs() {
    return cudaFuncSetAttribute(cnn_fp32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
}

// K splits: about four waves of one-block-per-SM work, at least 16 positions per split.
int choose_splits_fp32(int n, int sm_count, int max_splits) {
    const int blocks = (n + kHT - 1) / kHT;
    int s = (4 * sm_count + blocks - 1) / blocks;
    if (s > kPos / 16) s = kPos / 16;
    if (s > max_splits) s = max_splits;
    return s < 1 ? 1 : s;
}

cudaError_t launch_cnn_fp32(const DeviceWeights &w, const float *patches, int32_t n, int splits, float *partials,
                            int n_pad, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    ConvParams cp;
    for (int i = 0; i < kK * kK * kF; ++i) cp.w[i] = w.conv_w_host[i];
    for (int i = 0; i < kF; ++i) cp.b[i] = w.conv_b_host[i];
    dim3 grid((n + kHT - 1) / kHT, splits);
    cnn_fp32_kernel<<<grid, kThreads, kSmemBytes, s>>>(patches, n, cp, w.fc1_w, splits, partials, n_pad);
    return cudaGetLastError();
}

}  // namespace emtk
