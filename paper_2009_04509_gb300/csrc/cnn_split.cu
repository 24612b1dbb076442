// Tensor-core network path with fp32 accuracy (EMTK_TF32): the conv 5x5x48 +
// ReLU (Sec. 2.2) fused into dense-1 (92,928 -> 128) as in cnn_tc.cu, with
// every fp32 operand of the two contractions written as the sum of two fp16
// values, a head h = fp16(x) and a tail t = fp16(x - h) (22 significant bits
// together, as many as a TF32 head and tail), and every product taken as
// three fp16 tensor-core products, h_a h_b + h_a t_b + t_a h_b, accumulated in
// fp32; the dropped t_a t_b is below 2^-22 of the product.  This is the
// operand-splitting method of Markidis et al. (2018, "NVIDIA Tensor Core
// Programmability, Performance & Precision"), with power-of-two scales that
// keep heads and tails inside fp16's range (as in Ootomo and Yokota, 2022).
// The split runs at the fp16 tensor rate, twice that of tcgen05 kind::tf32,
// and its A operands take 16-bit TMEM columns, so the 4-slot TMEM ring of the
// 16-bit kernel stays as it is.
//
// Scales (powers of two: multiplying by them is exact):
//   patch pixels     x s_p = 2^-4, when the interval image is written
//   conv weights     x s_c, the largest 2^k with max(|conv_w|, s_p |conv_b|) s_c <= 2^14
//   conv bias        x s_p s_c, carried by two bias taps (1.0) of the im2col row
//   activations      the epilogue multiplies the ReLU'd conv sum by s_a / (s_p s_c):
//                    dense-1's A operand is the activation times s_a = 2^-4
//   dense-1 weights  x s_w, the largest 2^k with max|W1| s_w <= 2^14
//   dense-1 sums     x 1 / (s_a s_w) in the head, before the dense-1 bias
// Interval values and activations must stay below 2^20 in magnitude (2^20
// s_p is fp16's largest finite value, nearly).
//
// Work units, stream-K split and warp roles are those of cnn_tc.cu.  The
// differences:
//   builder warps   an interval-image pixel is a 32-bit word (fp16 head in
//                   the low half, tail in the high half).  A whole window row
//                   of words does not fit the registers, so a thread slides
//                   along each output row instead: it keeps the 16-byte chunks
//                   the next quad shares with this one and loads one new chunk
//                   per window row, a quad ahead; it writes two im2col tiles,
//                   heads and tails;
//   conv issuer     6 MMAs per pair (heads x head weights, heads x tail
//                   weights, tails x head weights; K = 32 each, as two K16);
//   epilogue        each position's 48 fp32 conv sums become 48 fp16 heads
//                   (TMEM columns 0-23 of the position) and 48 tails
//                   (columns 24-47), written over them;
//   dense-1 issuer  18 MMAs per pair; the pair's W1 heads and tails arrive by
//                   TMA (3 boxes of 32 inputs x 128 outputs each, 64-byte
//                   swizzle) into one of 3 stages; the accumulator restarts
//                   every kSegPairs pairs and the epilogue adds the segments
//                   up in fp32 (see kSegPairs).
#include <cuda.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <vector>

#include "emtk_internal.h"
#include "tc_ptx.cuh"

namespace emtk {
namespace {

constexpr int kThreadsSp = 352;  // 11 warps, roles as in cnn_tc.cu
constexpr int kTmaWarpSp = 0;
constexpr int kConvWarpSp = 1;
constexpr int kFc1WarpSp = 3;    // warps 4-7: epilogue
__host__ __device__ constexpr int builder_of(int warp) { return warp == 2 ? 0 : warp >= 8 ? warp - 7 : -1; }
constexpr int kPairNSp = 2 * kF;                              // 96 conv outputs per pair
constexpr int kPairsPerTile = 2 * kQuads;                     // 968
constexpr int kStagesSp = 3;                                  // W1 stages, one pair each
constexpr int kImBufsSp = 2;                                  // im2col buffers, one quad each
constexpr int kSlotsSp = 4;                                   // TMEM conv/activation slots
constexpr int kBoxKSp = 32;                                   // dense-1 inputs per TMA box (64-byte rows)
constexpr int kBoxBytesSp = kBoxKSp * kN1 * 2;                // 8192
constexpr int kBoxesPerPair = kPairNSp / kBoxKSp;             // 3
constexpr int kHalfStageSp = kBoxesPerPair * kBoxBytesSp;     // 24576: heads (or tails) of a pair
constexpr int kStageBytesSp = 2 * kHalfStageSp;               // 49152
constexpr int kImTileSp = 128 * 128;                          // 128 hits x 2 pairs x 32 taps x 2 B
constexpr int kImBufSp = 2 * kImTileSp;                       // heads and tails
constexpr int kConvBHalfSp = kPairNSp * 64;                   // 96 rows of 32 taps, 64-byte swizzle
constexpr uint32_t kTmemColsSp = 512;
constexpr uint32_t kAccColSp = 0;
constexpr uint32_t kSlotCol0Sp = 128;
constexpr float kActScaleSp = 0.0625f;                        // s_a
// The tensor core's fp32 accumulation rounds each MMA's sum toward zero, so a
// long run of MMAs into one accumulator drifts: measured over a tile's 17,424
// MMAs, 82% of the dense-1 sums came out smaller in magnitude than the exact
// ones (relative error up to 5e-2 on small sums), against 49% for fp32 FMA
// on the CUDA cores.  So the accumulator restarts every kSegPairs pairs
// (792 MMAs) and the epilogue adds each segment's sums to the CTA's partial
// row with round-to-nearest fp32 adds, in pair order (deterministic).
constexpr int kSegPairs = 44;
static_assert((2 * kQuads) % kSegPairs == 0, "segments tile the pairs of a tile");

constexpr int kOffW1Sp = 0;
constexpr int kOffImSp = kOffW1Sp + kStagesSp * kStageBytesSp;
constexpr int kOffConvBSp = kOffImSp + kImBufsSp * kImBufSp;
constexpr int kOffBarSp = kOffConvBSp + 2 * kConvBHalfSp;
constexpr int kBW1Full = 0;
constexpr int kBW1Empty = kBW1Full + kStagesSp;
constexpr int kBImFull = kBW1Empty + kStagesSp;   // im2col tiles written (4 builder warps)
constexpr int kBImFree = kBImFull + kImBufsSp;    // im2col tiles read by their convs (commit)
constexpr int kBConv = kBImFree + kImBufsSp;      // a pair's conv sums done (commit)
constexpr int kBAct = kBConv + kSlotsSp;          // a pair's heads and tails written (4 epilogue warps)
constexpr int kBFree = kBAct + kSlotsSp;          // a pair's dense-1 done (commit)
constexpr int kBAcc = kBFree + kSlotsSp;          // a tile's dense-1 done (commit)
constexpr int kBAccEmpty = kBAcc + 1;             // accumulator drained (4 epilogue warps)
constexpr int kBStall = kBAccEmpty + 1;
constexpr int kBDrain = kBStall + 1;
constexpr int kNumBarsSp = kBDrain + 1;
constexpr int kOffTmemSlotSp = kOffBarSp + kNumBarsSp * 8;
constexpr int kOffAbortSp = kOffTmemSlotSp + 4;
constexpr int kSmemBytesSp = kOffAbortSp + 4 + 1024;  // slack for 1024-byte alignment
static_assert(kSmemBytesSp <= 232448, "shared memory budget");
static_assert(kOffImSp % 1024 == 0 && kOffConvBSp % 1024 == 0 && kImTileSp % 1024 == 0 &&
                  kConvBHalfSp % 512 == 0 && kBoxBytesSp % 1024 == 0,
              "swizzle atoms must stay aligned");
static_assert(kSlotCol0Sp + kSlotsSp * kPairNSp <= kTmemColsSp, "TMEM budget");

// fp16 head and tail of two fp32 values, packed: element 0 in the low half.
__device__ __forceinline__ void split2(float v0, float v1, uint32_t &head, uint32_t &tail) {
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(head) : "f"(v1), "f"(v0));
    const float h0 = __half2float(__ushort_as_half((unsigned short)(head & 0xFFFFu)));
    const float h1 = __half2float(__ushort_as_half((unsigned short)(head >> 16)));
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(tail) : "f"(__fsub_rn(v1, h1)), "f"(__fsub_rn(v0, h0)));
}

// Words x0 .. x0+7 of window row r for a hit whose window leaves the haloed
// image: every pixel checked against the plane, zero outside.
__device__ __forceinline__ void load_words8_checked(const uint32_t *__restrict__ src, const HitDesc &hd, int r,
                                                   int x0, uint32_t (&out)[8]) {
    const int w = hd.wc - kHalf + r;
    const bool wok = w >= 0 && w < hd.nwires;
    const uint32_t *rowp = src + hd.d_off + (int64_t)(wok ? w + kHalo : 0) * hd.pitch + kHalo;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const int64_t b = (int64_t)hd.bc - kHalf + x0 + j;
        out[j] = (wok && b >= 0 && b < hd.nint) ? rowp[b] : 0u;
    }
}

__global__ void __launch_bounds__(kThreadsSp, 1)
    cnn_split_kernel(const __grid_constant__ CUtensorMap tmap_hi, const __grid_constant__ CUtensorMap tmap_lo,
                     const uint32_t *__restrict__ src, const HitDesc *__restrict__ desc, int n,
                     const uint16_t *__restrict__ convB_g, float act_mul, float *__restrict__ partials, int n_pad,
                     long long units, int *status, long long timeout_ns, int debug_stall, int *tile_done) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t base = (raw_u32 + 1023u) & ~1023u;
    uint8_t *gbase = smem_raw + (base - raw_u32);
    const uint32_t sW1 = base + kOffW1Sp;
    const uint32_t sIm = base + kOffImSp;
    const uint32_t sConvB = base + kOffConvBSp;
    auto bar = [&](int i) -> uint32_t { return base + kOffBarSp + 8u * (uint32_t)i; };
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(gbase + kOffTmemSlotSp);
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(gbase + kOffAbortSp);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cta = blockIdx.x;
    const int G = gridDim.x;
    const int64_t u0 = unit_begin(cta, units, G);  // this CTA's quads [u0, u1)
    const int64_t u1 = unit_begin(cta + 1, units, G);
    const int nq = (int)(u1 - u0);
    const int np = 2 * nq;                         // pairs, in order
    const int qt0 = (int)(u0 % kQuads);
    const int tile0 = (int)(u0 / kQuads);
    const Guard guard{abort_flag, status, (int64_t)timeout_ns};

    // the next kernel (the head) may be scheduled as SMs free up; it waits for this one
    pdl_trigger();
    // ---- set-up: conv B heads and tails into 64-byte-swizzled smem, barriers, TMEM
    for (int idx = threadIdx.x; idx < 2 * kPairNSp * 4; idx += kThreadsSp) {
        const int h = idx / (kPairNSp * 4), rem = idx % (kPairNSp * 4);
        const int row = rem >> 2, chunk = rem & 3;
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(convB_g + (h * kPairNSp + row) * 32) + chunk);
        *reinterpret_cast<uint4 *>(gbase + kOffConvBSp + h * kConvBHalfSp + row * 64 +
                                   ((chunk ^ ((row >> 1) & 3)) << 4)) = v;
    }
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStagesSp; ++i) {
            mbar_init(bar(kBW1Full + i), 1);
            mbar_init(bar(kBW1Empty + i), 1);
        }
        for (int i = 0; i < kImBufsSp; ++i) {
            mbar_init(bar(kBImFull + i), 4);
            mbar_init(bar(kBImFree + i), 1);
        }
        for (int i = 0; i < kSlotsSp; ++i) {
            mbar_init(bar(kBConv + i), 1);
            mbar_init(bar(kBAct + i), 4);
            mbar_init(bar(kBFree + i), 1);
        }
        mbar_init(bar(kBAcc), 1);
        mbar_init(bar(kBAccEmpty), 4);
        mbar_init(bar(kBStall), 1);
        mbar_init(bar(kBDrain), 2);
        *abort_flag = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (warp == kConvWarpSp) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(base + kOffTmemSlotSp),
                     "r"(kTmemColsSp)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == kTmaWarpSp) {
        // ================================================ TMA producer (W1)
        if (lane == 0) {
            int issued = 0;
            bool ok = true;
            int pt = 2 * qt0;  // pair in tile
            for (int jj = 0; jj < np; ++jj, pt = (pt + 1 == kPairsPerTile) ? 0 : pt + 1) {
                const int wj = jj % kStagesSp;
                const uint32_t use = (uint32_t)(jj / kStagesSp);
                if (jj >= kStagesSp && !wait_bounded(bar(kBW1Empty + wj), (use - 1u) & 1u, guard)) {
                    ok = false;
                    break;
                }
                if (*abort_flag) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(bar(kBW1Full + wj), kStageBytesSp);
                const uint32_t dst = sW1 + wj * kStageBytesSp;
#pragma unroll
                for (int b = 0; b < kBoxesPerPair; ++b) {
                    const int kb32 = kBoxesPerPair * pt + b;  // box of 32 inputs: half of a 64-input tile
                    const int c0 = (kb32 & 1) * kBoxKSp, c2 = kb32 >> 1;
                    tma_load_3d(dst + b * kBoxBytesSp, &tmap_hi, bar(kBW1Full + wj), c0, 0, c2);
                    tma_load_3d(dst + kHalfStageSp + b * kBoxBytesSp, &tmap_lo, bar(kBW1Full + wj), c0, 0, c2);
                }
                ++issued;
            }
            if (!ok) {  // let copies in flight land before the CTA's memory goes away
                for (int jj = issued > kStagesSp ? issued - kStagesSp : 0; jj < issued; ++jj) {
                    const uint32_t b = bar(kBW1Full + jj % kStagesSp);
                    const uint32_t par = (uint32_t)(jj / kStagesSp) & 1u;
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(b, par) && (int64_t)(global_timer_ns() - t0) < (int64_t)timeout_ns) {
                    }
                }
            }
        }
    } else if (warp == kConvWarpSp || warp == kFc1WarpSp) {
        // ====================================================== MMA issuers
        if (lane == 0) {
            bool ok = true;
            if (warp == kConvWarpSp) {
                constexpr uint32_t idesc = make_idesc(128, kPairNSp, true);
                const uint64_t bh = sw64_desc(sConvB), bl = sw64_desc(sConvB + kConvBHalfSp);
                if (debug_stall) ok = wait_bounded(bar(kBStall), 0u, guard);  // nothing arrives here
                for (int q = 0; ok && q < nq; ++q) {
                    const int ib = q % kImBufsSp;
                    if (!wait_bounded(bar(kBImFull + ib), (uint32_t)(q / kImBufsSp) & 1u, guard)) {
                        ok = false;
                        break;
                    }
                    const uint64_t ah0 = sw128_desc(sIm + ib * kImBufSp);
                    const uint64_t al0 = sw128_desc(sIm + ib * kImBufSp + kImTileSp);
                    for (int pr = 0; pr < 2; ++pr) {
                        const int p = 2 * q + pr;
                        const int s = p % kSlotsSp;
                        if (p >= kSlotsSp &&
                            !wait_bounded(bar(kBFree + s), (uint32_t)(p / kSlotsSp - 1) & 1u, guard)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem + kSlotCol0Sp + (uint32_t)s * kPairNSp;
                        const uint64_t ah = ah0 + (uint64_t)((pr * 64) >> 4), al = al0 + (uint64_t)((pr * 64) >> 4);
                        constexpr uint64_t k16 = 32u >> 4;  // the second K16 step: 32 bytes further
                        mma_ss(d, ah, bh, idesc, 0u);
                        mma_ss(d, ah + k16, bh + k16, idesc, 1u);
                        mma_ss(d, ah, bl, idesc, 1u);
                        mma_ss(d, ah + k16, bl + k16, idesc, 1u);
                        mma_ss(d, al, bh, idesc, 1u);
                        mma_ss(d, al + k16, bh + k16, idesc, 1u);
                        mma_commit(bar(kBConv + s));
                    }
                    if (!ok) break;
                    mma_commit(bar(kBImFree + ib));
                }
            } else {
                constexpr uint32_t idesc = make_idesc(128, kN1, true);
                int segs_done = 0;  // accumulator segments handed to the epilogue
                int pt = 2 * qt0 - 1;
                for (int jj = 0; ok && jj < np; ++jj) {
                    pt = (pt + 1 == kPairsPerTile) ? 0 : pt + 1;
                    const bool first = (jj == 0) || (pt % kSegPairs == 0);
                    const bool last = (jj == np - 1) || (pt % kSegPairs == kSegPairs - 1);
                    const int wj = jj % kStagesSp;
                    const int s = jj % kSlotsSp;
                    if (!wait_bounded(bar(kBW1Full + wj), (uint32_t)(jj / kStagesSp) & 1u, guard) ||
                        !wait_bounded(bar(kBAct + s), (uint32_t)(jj / kSlotsSp) & 1u, guard)) {
                        ok = false;
                        break;
                    }
                    // a segment starts from zero once the epilogue has read the last one
                    if (first && segs_done > 0 &&
                        !wait_bounded(bar(kBAccEmpty), (uint32_t)(segs_done - 1) & 1u, guard)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t stage = sW1 + wj * kStageBytesSp;
                    const uint32_t a0 = tmem + kSlotCol0Sp + (uint32_t)s * kPairNSp;
#pragma unroll
                    for (int pos = 0; pos < 2; ++pos) {
#pragma unroll
                        for (int st = 0; st < 3; ++st) {
                            const int k = 48 * pos + 16 * st;  // first of the step's 16 inputs in the pair
                            const uint32_t woff = (uint32_t)((k >> 5) * kBoxBytesSp + (k & 31) * 2);
                            const uint32_t ah = a0 + 48u * pos + 8u * st, al = ah + 24u;
                            const uint64_t wh = sw64_desc(stage + woff), wl = sw64_desc(stage + kHalfStageSp + woff);
                            mma_ts(tmem + kAccColSp, ah, wh, idesc, (first && pos == 0 && st == 0) ? 0u : 1u);
                            mma_ts(tmem + kAccColSp, ah, wl, idesc, 1u);
                            mma_ts(tmem + kAccColSp, al, wh, idesc, 1u);
                        }
                    }
                    mma_commit(bar(kBFree + s));
                    mma_commit(bar(kBW1Empty + wj));
                    if (last) {
                        mma_commit(bar(kBAcc));
                        ++segs_done;
                    }
                }
            }
            // every MMA either thread issued completes before TMEM is released
            mma_commit(bar(kBDrain));
            const uint64_t t0 = global_timer_ns();
            while (!mbar_try_wait(bar(kBDrain), 0u) && (int64_t)(global_timer_ns() - t0) < (int64_t)timeout_ns) {
            }
        }
        __syncwarp();
    } else if (builder_of(warp) >= 0) {
        // ================================================ im2col builder
        // Row r of each im2col tile (hit r) is 128 bytes: pair (x, x+1) in
        // chunks 0-3, pair (x+2, x+3) in chunks 4-7, chunk c at c ^ (r & 7)
        // (128-byte swizzle).  Tap t = 6i + j of a pair at x is window pixel
        // (y + i, x + j); taps 30 and 31 are 1.0 in the heads tile (the bias)
        // and 0 in the tails tile.
        const int q4 = builder_of(warp);
        const int row = 32 * q4 + lane;
        constexpr uint32_t ones = 0x3C003C00u;  // two fp16 1.0
        pdl_wait();  // the images and window descriptors come from the kernel before
        uint8_t *my_hi = gbase + kOffImSp + row * 128;
        bool ok = true;
        const int t_first = tile0;
        const int t_last = nq > 0 ? (int)((u1 - 1) / kQuads) : t_first - 1;
        for (int tile = t_first; ok && tile <= t_last; ++tile) {
            const int j0 = tile == t_first ? qt0 : 0;
            const int j1 = tile == t_last ? (int)((u1 - 1) % kQuads) + 1 : kQuads;
            const int64_t k_base = (int64_t)tile * kQuads - u0;
            const int64_t hit = (int64_t)tile * 128 + row;
            const bool valid = hit < n;
            HitDesc hd;
            if (desc == nullptr) {
                hd.origin = valid ? hit * kPatchElems : 0;
                hd.pitch = kPatch;
                hd.inside = 1;
            } else if (valid) {
                hd = desc[hit];
            } else {
                hd.inside = 1;
            }
            // The window words of a quad at x0 lie in 16-byte chunks eb, eb+4 and, for
            // a window not aligned to 4 words (m > 0), eb+8 of each of its 5 rows
            // (eb = first word of the row + x0 - m).  Consecutive quads of an
            // output row share all but the last chunk, so `raw` carries them and
            // the new chunk of the next quad is loaded into `nxt` while this one
            // is built.
            const int m = (int)(hd.origin & 3);
            const bool fast = valid && hd.inside;
            uint32_t raw[kK][12], nxt[kK][4];
            for (int quad = j0; ok && quad < j1; ++quad) {
                const int y = quad / (kQ / 4), x0 = 4 * (quad % (kQ / 4));
                uint32_t W[kK][8];
                if (fast) {
                    const int64_t eb0 = hd.origin + (int64_t)y * hd.pitch + x0 - m;
                    if (quad == j0 || x0 == 0) {  // a new output row: load the chunks
#pragma unroll
                        for (int i = 0; i < kK; ++i) {
                            const uint4 *pc = reinterpret_cast<const uint4 *>(src + eb0 + (int64_t)i * hd.pitch);
                            const uint4 c0 = __ldg(pc), c1 = __ldg(pc + 1);
                            raw[i][0] = c0.x, raw[i][1] = c0.y, raw[i][2] = c0.z, raw[i][3] = c0.w;
                            raw[i][4] = c1.x, raw[i][5] = c1.y, raw[i][6] = c1.z, raw[i][7] = c1.w;
                            if (m != 0) {
                                const uint4 c2 = __ldg(pc + 2);
                                raw[i][8] = c2.x, raw[i][9] = c2.y, raw[i][10] = c2.z, raw[i][11] = c2.w;
                            }
                        }
                    } else {  // one chunk further: the prefetched one comes last
#pragma unroll
                        for (int i = 0; i < kK; ++i) {
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                raw[i][j] = raw[i][j + 4];
                                raw[i][j + 4] = m != 0 ? raw[i][j + 8] : nxt[i][j];
                                raw[i][j + 8] = nxt[i][j];
                            }
                        }
                    }
                    // the next quad of this output row: its new chunk, ahead of time
                    if (quad + 1 < j1 && x0 + 4 < kQ) {
                        const int64_t nc = eb0 + (m != 0 ? 12 : 8);
#pragma unroll
                        for (int i = 0; i < kK; ++i) {
                            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(src + nc + (int64_t)i * hd.pitch));
                            nxt[i][0] = v.x, nxt[i][1] = v.y, nxt[i][2] = v.z, nxt[i][3] = v.w;
                        }
                    }
                    // words m .. m+7 of each row: a shift made of selects
#pragma unroll
                    for (int i = 0; i < kK; ++i) {
                        uint32_t s2[10];
#pragma unroll
                        for (int j = 0; j < 10; ++j) s2[j] = (m & 2) ? raw[i][j + 2] : raw[i][j];
#pragma unroll
                        for (int j = 0; j < 8; ++j) W[i][j] = (m & 1) ? s2[j + 1] : s2[j];
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < kK; ++i) {
                        if (valid) {
                            load_words8_checked(src, hd, y + i, x0, W[i]);
                        } else {
#pragma unroll
                            for (int j = 0; j < 8; ++j) W[i][j] = 0u;
                        }
                    }
                }
                const int k = (int)(k_base + quad);
                const int ib = k % kImBufsSp;
                if (k >= kImBufsSp &&
                    !warp_wait(bar(kBImFree + ib), (uint32_t)(k / kImBufsSp - 1) & 1u, guard, lane)) {
                    ok = false;
                    break;
                }
                uint8_t *dh = my_hi + ib * kImBufSp;
                uint8_t *dl = dh + kImTileSp;
#pragma unroll
                for (int c = 0; c < 8; ++c) {  // chunk c: pair c / 4, taps 8 (c % 4) .. +7
                    const int xo = 2 * (c >> 2);
                    uint32_t hw[4], lw[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int kw = 4 * (c & 3) + e;  // word kw: taps 2 kw, 2 kw + 1
                        if (kw == 15) {
                            hw[e] = ones;
                            lw[e] = 0u;
                        } else {
                            const int i = kw / 3, jp = kw % 3;  // row i, columns x + 2 jp, x + 2 jp + 1
                            const uint32_t wa = W[i][xo + 2 * jp], wb = W[i][xo + 2 * jp + 1];
                            hw[e] = __byte_perm(wa, wb, 0x5410);
                            lw[e] = __byte_perm(wa, wb, 0x7632);
                        }
                    }
                    const int off = (c ^ (row & 7)) << 4;
                    *reinterpret_cast<uint4 *>(dh + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                    *reinterpret_cast<uint4 *>(dl + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBImFull + ib));
            }
        }
    } else {
        // ================================== epilogue + dense-1 partial sums
        const int q4 = warp & 3;
        const int row = 32 * q4 + lane;
        const uint32_t lane_tmem = tmem + ((uint32_t)(32 * q4) << 16);
        int segs_done = 0;
        int64_t last_tile = -1;  // tile whose partial row this CTA has started
        for (int pi = 0; pi < np; ++pi) {
            const int s = pi % kSlotsSp;
            if (!warp_wait(bar(kBConv + s), (uint32_t)(pi / kSlotsSp) & 1u, guard, lane)) break;
            tc_fence_after();
            const uint32_t d = lane_tmem + kSlotCol0Sp + (uint32_t)s * kPairNSp;
#pragma unroll
            for (int h = 0; h < 2; ++h) {  // position x, then x+1: 48 fp32 -> 24 head words + 24 tail words
                uint32_t f[48];
                tmem_ld16<0>(d + 48u * h, f);
                tmem_ld16<16>(d + 48u * h + 16u, f);
                tmem_ld16<32>(d + 48u * h + 32u, f);
                tmem_ld_wait();
                reg_fence(f);
                uint32_t oh[24], ol[24];
#pragma unroll
                for (int i = 0; i < 24; ++i) {
                    const float v0 = fmaxf(__uint_as_float(f[2 * i]), 0.0f) * act_mul;
                    const float v1 = fmaxf(__uint_as_float(f[2 * i + 1]), 0.0f) * act_mul;
                    split2(v0, v1, oh[i], ol[i]);
                }
                tmem_st16<0>(d + 48u * h, oh);
                tmem_st8<16>(d + 48u * h + 16u, oh);
                tmem_st16<0>(d + 48u * h + 24u, ol);
                tmem_st8<16>(d + 48u * h + 40u, ol);
            }
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBAct + s));
            const int64_t gp = 2 * u0 + pi;  // the pair's index in the launch
            const int pt = (int)(gp % kPairsPerTile);
            if (pi == np - 1 || pt % kSegPairs == kSegPairs - 1) {
                // a segment's sums: to (first segment of this CTA in the tile) or onto
                // this CTA's partial row of the tile
                if (!warp_wait(bar(kBAcc), (uint32_t)segs_done & 1u, guard, lane)) break;
                tc_fence_after();
                const int64_t tile = gp / kPairsPerTile;
                const bool start = tile != last_tile;
                last_tile = tile;
                const int krow = cta - cta_of_unit(tile * kQuads, units, G);
                const int64_t hit = tile * 128 + row;
                float *dst = partials + ((int64_t)krow * n_pad + hit) * kN1;
#pragma unroll
                for (int c = 0; c < kN1 / 32; ++c) {
                    uint32_t r[32];
                    tmem_ld16<0>(lane_tmem + kAccColSp + 32u * c, r);
                    tmem_ld16<16>(lane_tmem + kAccColSp + 32u * c + 16u, r);
                    tmem_ld_wait();
                    reg_fence(r);
                    if (hit < n) {
                        float4 *p4 = reinterpret_cast<float4 *>(dst + 32 * c);
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            float4 v = make_float4(__uint_as_float(r[4 * e]), __uint_as_float(r[4 * e + 1]),
                                                   __uint_as_float(r[4 * e + 2]), __uint_as_float(r[4 * e + 3]));
                            if (!start) {
                                const float4 o = p4[e];
                                v = make_float4(__fadd_rn(o.x, v.x), __fadd_rn(o.y, v.y), __fadd_rn(o.z, v.z),
                                                __fadd_rn(o.w, v.w));
                            }
                            p4[e] = v;
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBAccEmpty));
                // this CTA's last segment of the tile: its partial row is final, count it for the head
                if (tile_done != nullptr && (pi == np - 1 || pt == kPairsPerTile - 1)) {
                    __threadfence();
                    __syncwarp();
                    if (lane == 0) atomicAdd(tile_done + tile, 1);
                }
                ++segs_done;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kConvWarpSp) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemColsSp) : "memory");
    }
}

// The largest power of two 2^k with m 2^k <= cap (1 for m = 0 or not finite).
double pow2_scale(double m, double cap) {
    if (!(m > 0.0) || !std::isfinite(m)) return 1.0;
    int k = 0;
    while (k < 200 && m * std::ldexp(1.0, k + 1) <= cap) ++k;
    while (k > -200 && m * std::ldexp(1.0, k) > cap) --k;
    return std::ldexp(1.0, k);
}

uint16_t half_bits(float v) {
    const __half h = __float2half_rn(v);
    return __half_as_ushort(h);
}

// fp16 head and tail of v: v ~ head + tail.
void split_host(float v, uint16_t &head, uint16_t &tail) {
    head = half_bits(v);
    tail = half_bits(v - __half2float(__ushort_as_half(head)));
}

}  // namespace

cudaError_t init_split_kernel_attrs() {
    return cudaFuncSetAttribute(cnn_split_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytesSp);
}

cudaError_t prepare_split_weights(DeviceWeights &w, const emtk_weights &hw) {
    const size_t nw1 = (size_t)kFc1In * kN1;
    const int kKBlocks = kFc1In / 64;
    float mw = 0.0f, mc = 0.0f;
    for (size_t i = 0; i < nw1; ++i) mw = std::fmax(mw, std::fabs(hw.fc1_w[i]));
    for (int i = 0; i < kK * kK * kF; ++i) mc = std::fmax(mc, std::fabs(hw.conv_w[i]));
    for (int f = 0; f < kF; ++f) mc = std::fmax(mc, std::fabs(hw.conv_b[f]) * kSplitPatchScale);
    const float s_w = (float)pow2_scale(mw, 16384.0);
    const float s_c = (float)pow2_scale(mc, 16384.0);
    w.fc1_w_scale = s_w;
    w.fc1_scale = 1.0f / (kActScaleSp * s_w);
    w.act_mul = kActScaleSp / (kSplitPatchScale * s_c);
    // dense-1 heads and tails, each tiled [K/64][128][64] like the 16-bit weights
    std::vector<uint16_t> tiles(2 * nw1);
    for (int kb = 0; kb < kKBlocks; ++kb)
        for (int nn = 0; nn < kN1; ++nn)
            for (int kk = 0; kk < 64; ++kk) {
                const size_t t = ((size_t)kb * kN1 + nn) * 64 + kk;
                split_host(hw.fc1_w[(size_t)(kb * 64 + kk) * kN1 + nn] * s_w, tiles[t], tiles[nw1 + t]);
            }
    // conv B heads [96][32] then tails [96][32]: row f (< 48) is filter f at
    // position x, row 48 + f filter f at x + 1; tap t = 6i + j reads window
    // column j; taps 30 and 31 of the heads carry the bias's head and tail
    std::vector<uint16_t> cb(2 * kPairNSp * 32, 0);
    for (int f = 0; f < kF; ++f) {
        for (int i = 0; i < kK; ++i)
            for (int j = 0; j < kK; ++j) {
                uint16_t h, t;
                split_host(hw.conv_w[(i * kK + j) * kF + f] * s_c, h, t);
                for (int pos = 0; pos < 2; ++pos) {
                    const size_t r = (size_t)(pos * kF + f) * 32 + 6 * i + j + pos;
                    cb[r] = h;
                    cb[(size_t)kPairNSp * 32 + r] = t;
                }
            }
        uint16_t bh, bl;
        split_host(hw.conv_b[f] * kSplitPatchScale * s_c, bh, bl);
        for (int pos = 0; pos < 2; ++pos) {
            cb[(size_t)(pos * kF + f) * 32 + 30] = bh;
            cb[(size_t)(pos * kF + f) * 32 + 31] = bl;
        }
    }
    cudaError_t e = dev_alloc(&w.w1_tiles, 2 * nw1 * 2);
    if (e != cudaSuccess) return e;
    e = cudaMemcpy(w.w1_tiles, tiles.data(), 2 * nw1 * 2, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return e;
    void *cbp = nullptr;
    e = dev_alloc(&cbp, cb.size() * 2);
    w.convB = static_cast<uint16_t *>(cbp);
    if (e != cudaSuccess) return e;
    e = cudaMemcpy(w.convB, cb.data(), cb.size() * 2, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return e;

    void *fn = nullptr;
    cudaDriverEntryPointQueryResult qr;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qr);
    if (e != cudaSuccess || fn == nullptr || qr != cudaDriverEntryPointSuccess) return cudaErrorNotSupported;
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    CUtensorMap *maps = new CUtensorMap[2];
    for (int h = 0; h < 2; ++h) {
        cuuint64_t dims[3] = {64, (cuuint64_t)kN1, (cuuint64_t)kKBlocks};
        cuuint64_t strides[2] = {64 * 2, (cuuint64_t)64 * kN1 * 2};
        cuuint32_t box[3] = {(cuuint32_t)kBoxKSp, (cuuint32_t)kN1, 1u};  // 64-byte rows
        cuuint32_t estr[3] = {1u, 1u, 1u};
        CUresult r = encode(&maps[h], CU_TENSOR_MAP_DATA_TYPE_UINT16, 3,
                            static_cast<uint16_t *>(w.w1_tiles) + (size_t)h * nw1, dims, strides, box, estr,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            delete[] maps;
            return cudaErrorInvalidValue;
        }
    }
    w.w1_tmap = maps;
    return cudaSuccess;
}

cudaError_t launch_cnn_split(const DeviceWeights &w, const void *src, const HitDesc *desc, int32_t n, int G,
                             float *partials, int n_pad, int *status, int64_t timeout_ns, int debug_stall,
                             int *tile_done, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const CUtensorMap *maps = static_cast<const CUtensorMap *>(w.w1_tmap);
    const long long units = (long long)((n + 127) / 128) * kQuads;
    const uint32_t *src32 = static_cast<const uint32_t *>(src);
    const uint16_t *convB = w.convB;
    const float act_mul = w.act_mul;
    const long long tmo = (long long)timeout_ns;
    return launch_pdl(cnn_split_kernel, dim3(G), dim3(kThreadsSp), kSmemBytesSp, s, maps[0], maps[1], src32, desc, n,
                      convB, act_mul, partials, n_pad, units, status, tmo, debug_stall, tile_done);
}

}  // namespace emtk
