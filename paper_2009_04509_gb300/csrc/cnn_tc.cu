// Tensor-core network path on sm_103a (EMTK_BF16 / EMTK_FP16 / EMTK_FP8):
// the conv 5x5x48 + ReLU (Sec. 2.2) fused into dense-1 (92,928 -> 128), so
// the 92,928 conv activations of a hit never leave the SM.
//
// Work units are (tile of 128 hits, quad of 4 conv positions of one output
// row): 484 quads per tile, each supplying 192 consecutive dense-1 inputs
// (input index = position * 48 + filter, the channels-last flatten).  One
// persistent CTA per SM takes a contiguous range of units (stream-K), across
// tile boundaries; a quad is two position pairs (x, x+1):
//   builder warps   write, per hit, the 5 x 6 window of a pair (30 taps) and
//                   two bias taps of 1.0 as one 32-wide im2col row into a
//                   swizzled shared-memory tile (one 128-byte row per hit and
//                   quad), reading the window straight from the hit's plane
//                   image;
//   conv issuer     D[128 x 96] = A_smem[128 x 32] * Bpair[32 x 96] (16 bit):
//                   columns 0-47 are the 48 filters at x, 48-95 at x+1; the
//                   conv bias rides on the bias taps;
//   epilogue warps  ReLU + round the 128 x 96 conv tile (to 16 bit, or to
//                   e4m3: there the conv weights and bias are scaled by
//                   kFp8ActScale, a power of two, so the tile is already the
//                   scaled activation), written back into TMEM over it;
//   dense-1 issuer  ACC[128 x 128] += A_tmem[128 x 96] * W1[96 x 128], W1
//                   streamed by TMA through a 3-stage ring (one quad per
//                   stage: 48 KB of 16-bit or 24 KB of e4m3 weights);
//   at a tile's end the epilogue drains ACC to the CTA's partial-sum row.
// Every wait is bounded: on timeout the CTA raises an abort flag, sets bit 0
// of the status word, waits for its in-flight copies and MMAs, frees TMEM
// and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <vector>

#include "emtk_internal.h"
#include "tc_ptx.cuh"

namespace emtk {
namespace {

// Warp roles.  A warp runs on the SM sub-partition (scheduler) warp mod 4,
// and an epilogue warp may only touch TMEM lanes 32 (warp mod 4) .. +31, so
// the four epilogue warps sit on all four sub-partitions.  The dense-1
// issuer, whose every idle cycle between MMAs idles the tensor pipe, shares
// its sub-partition with one epilogue warp only; the builder warps take the
// other slots.
constexpr int kThreadsTC = 352;  // 11 warps
constexpr int kTmaWarp = 0;
constexpr int kConvWarp = 1;
constexpr int kFc1Warp = 3;      // warps 4-7: epilogue, TMEM lane quarter warp mod 4
__host__ __device__ constexpr int builder_index(int warp) {  // warps 2, 8, 9, 10 -> row blocks 0-3
    return warp == 2 ? 0 : warp >= 8 ? warp - 7 : -1;
}
constexpr int kW1Stages = 3;     // shared-memory stages of W1 (one quad each)
constexpr int kImBufs = 3;       // shared-memory im2col tiles (one quad each)
constexpr int kSlots = 4;        // TMEM conv/activation slots (one pair each)
constexpr int kPosPerW1 = 4;     // conv positions per W1 stage = per quad
constexpr int kW1Steps = kQuads;                             // 484 quads
constexpr int kW1Box = 64;                                   // K elements per TMA box (128 B)
constexpr int kW1BoxBytes = kW1Box * kN1 * 2;                // 16384
constexpr int kBoxesPerStage = kPosPerW1 * kF / kW1Box;      // 3
constexpr int kW1StageBytes = kBoxesPerStage * kW1BoxBytes;  // 49152
constexpr int kKBlocks = kFc1In / kW1Box;                    // 1452
constexpr int kPairN = 2 * kF;                               // 96 conv outputs per pair
constexpr int kConvK = 32;                                   // 30 window taps + 2 bias taps
constexpr int kImBytes = 128 * 128;                          // 128 hits x (2 pairs x 32 taps x 2 B)
constexpr int kConvBBytes = kPairN * 128;                    // 96 rows of one 128-byte swizzle span
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCol = 0;                              // dense-1 accumulator, 128 fp32 columns
constexpr uint32_t kSlotCol0 = 128;                          // conv fp32 tile of a pair, then its activations
constexpr uint32_t kSlotCols = kPairN;
// EMTK_FP8: dense-1 operands in e4m3.  A W1 box is 64 inputs x 128 outputs of
// one byte (64-byte swizzle), a stage 3 boxes; activations are scaled by
// kFp8ActScale (a power of two) before rounding.
constexpr int kW1BoxBytesF8 = kW1Box * kN1;                  // 8192
constexpr int kW1StageBytesF8 = kBoxesPerStage * kW1BoxBytesF8;  // 24576
constexpr float kFp8ActScale = 0.0625f;

constexpr int kOffW1 = 0;
constexpr int kOffIm = kOffW1 + kW1Stages * kW1StageBytes;
constexpr int kOffConvB = kOffIm + kImBufs * kImBytes;
constexpr int kOffBar = kOffConvB + kConvBBytes;
// barrier indices
constexpr int kBarW1Full = 0;
constexpr int kBarW1Empty = kBarW1Full + kW1Stages;
constexpr int kBarImFull = kBarW1Empty + kW1Stages;  // im2col tile written (4 builder warps)
constexpr int kBarImFree = kBarImFull + kImBufs;     // im2col tile read by its convs (MMA commit)
constexpr int kBarConv = kBarImFree + kImBufs;       // conv tile of a pair done (MMA commit)
constexpr int kBarAct = kBarConv + kSlots;           // activations written (4 epilogue warps)
constexpr int kBarFree = kBarAct + kSlots;           // dense-1 of the slot's pair done (MMA commit)
constexpr int kBarAcc = kBarFree + kSlots;             // a tile's dense-1 done (MMA commit)
constexpr int kBarAccEmpty = kBarAcc + 1;             // accumulator drained (4 epilogue warps)
constexpr int kBarStall = kBarAccEmpty + 1;
constexpr int kBarDrain = kBarStall + 1;
constexpr int kNumBars = kBarDrain + 1;
// accumulator drain: per epilogue warp, 32 rows x 32 outputs staged with a
// 36-float row pitch (conflict-free 16-byte writes and reads), so each global
// store of the warp writes four whole 128-byte row pieces
constexpr int kStagePitch = 36;
constexpr int kStageBytes = 32 * kStagePitch * 4;  // one epilogue warp
constexpr int kOffStage = kOffBar + kNumBars * 8 + 8;  // 16-byte aligned below
constexpr int kOffStageA = (kOffStage + 15) / 16 * 16;
constexpr int kOffTmemSlot = kOffStageA + 4 * kStageBytes;
constexpr int kOffAbort = kOffTmemSlot + 4;
constexpr int kSmemUsed = kOffAbort + 4;
constexpr int kSmemBytesTC = kSmemUsed + 1024;  // slack for 1024-byte alignment
static_assert(kSmemBytesTC <= 232448, "shared memory budget");
static_assert(kSlotCol0 + kSlots * kSlotCols <= kTmemCols, "TMEM budget");
static_assert(kQ % kPosPerW1 == 0, "quads do not straddle rows");

// One 48-wide row of a hit's window, 16-bit pixels packed two per word:
// element e0 of src and the 47 after it.  Seven aligned 16-byte loads cover
// it; the words are then moved down by e0 % 8 elements with selects and a
// funnel shift (no dynamic register indexing).  src must have 16 bytes of
// readable memory past the last window element.
__device__ __forceinline__ void load_window_row(const uint16_t *__restrict__ src, int64_t e0, uint32_t (&out)[24]) {
    const int m = (int)(e0 & 7);
    const uint4 *p = reinterpret_cast<const uint4 *>(src + (e0 - m));
    uint32_t w[28];
#pragma unroll
    for (int c = 0; c < 6; ++c) {
        const uint4 v = __ldg(p + c);
        w[4 * c] = v.x;
        w[4 * c + 1] = v.y;
        w[4 * c + 2] = v.z;
        w[4 * c + 3] = v.w;
    }
    if (m == 0) {
#pragma unroll
        for (int j = 0; j < 24; ++j) out[j] = w[j];
        return;
    }
    const uint4 v = __ldg(p + 6);
    w[24] = v.x;
    w[25] = v.y;
    w[26] = v.z;
    w[27] = v.w;
    const int s = m >> 1;
    uint32_t a[26];
#pragma unroll
    for (int j = 0; j < 26; ++j) a[j] = (s & 2) ? w[j + 2] : w[j];
    uint32_t b[25];
#pragma unroll
    for (int j = 0; j < 25; ++j) b[j] = (s & 1) ? a[j + 1] : a[j];
    if (m & 1) {
#pragma unroll
        for (int j = 0; j < 24; ++j) out[j] = __funnelshift_r(b[j], b[j + 1], 16);
    } else {
#pragma unroll
        for (int j = 0; j < 24; ++j) out[j] = b[j];
    }
}

// The first kK rows of a window at once (row r starts at element e0 + r * pitch,
// pitch a multiple of 8, so every row has the phase e0 % 8): all aligned
// 16-byte loads are issued before any row is shifted, so the rows cost one
// round trip to memory instead of kK.
__device__ __forceinline__ void load_window_rows5(const uint16_t *__restrict__ src, int64_t e0, int64_t pitch,
                                                  uint32_t (&R)[kK][24]) {
    const int m = (int)(e0 & 7);
    uint32_t X[kK][4];  // the seventh chunk of each row (needed when m != 0)
#pragma unroll
    for (int r = 0; r < kK; ++r) {
        const uint4 *p = reinterpret_cast<const uint4 *>(src + (e0 + r * pitch - m));
#pragma unroll
        for (int c = 0; c < 6; ++c) {
            const uint4 v = __ldg(p + c);
            R[r][4 * c] = v.x;
            R[r][4 * c + 1] = v.y;
            R[r][4 * c + 2] = v.z;
            R[r][4 * c + 3] = v.w;
        }
        if (m != 0) {
            const uint4 v = __ldg(p + 6);
            X[r][0] = v.x;
            X[r][1] = v.y;
            X[r][2] = v.z;
            X[r][3] = v.w;
        } else {
            X[r][0] = X[r][1] = X[r][2] = X[r][3] = 0u;
        }
    }
    if (m == 0) return;
    const int s = m >> 1;
#pragma unroll
    for (int r = 0; r < kK; ++r) {
        uint32_t w[28];
#pragma unroll
        for (int j = 0; j < 24; ++j) w[j] = R[r][j];
#pragma unroll
        for (int j = 0; j < 4; ++j) w[24 + j] = X[r][j];
        uint32_t a[26];
#pragma unroll
        for (int j = 0; j < 26; ++j) a[j] = (s & 2) ? w[j + 2] : w[j];
        uint32_t b[25];
#pragma unroll
        for (int j = 0; j < 25; ++j) b[j] = (s & 1) ? a[j + 1] : a[j];
        if (m & 1) {
#pragma unroll
            for (int j = 0; j < 24; ++j) R[r][j] = __funnelshift_r(b[j], b[j + 1], 16);
        } else {
#pragma unroll
            for (int j = 0; j < 24; ++j) R[r][j] = b[j];
        }
    }
}

// Two fp32 values rounded to nearest-even 16 bit (bf16, or fp16 if FP16) and
// packed, the first in the low half: the rounding of the patch conversion.
template <bool FP16>
__device__ __forceinline__ uint32_t pack_rn16(float lo, float hi) {
    if (FP16) {
        const __half2 h = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<const uint32_t *>(&h);
    }
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// One 48-value row of a pre-cut fp32 patch (element e0 of src, 16-byte
// aligned): twelve 16-byte loads, rounded to 16 bit, two pixels per word.
template <bool FP16>
__device__ __forceinline__ void load_patch_row_f32(const float *__restrict__ src, int64_t e0, uint32_t (&out)[24]) {
    const float4 *p = reinterpret_cast<const float4 *>(src + e0);
    float4 v[12];
#pragma unroll
    for (int c = 0; c < 12; ++c) v[c] = __ldg(p + c);
#pragma unroll
    for (int c = 0; c < 12; ++c) {
        out[2 * c] = pack_rn16<FP16>(v[c].x, v[c].y);
        out[2 * c + 1] = pack_rn16<FP16>(v[c].z, v[c].w);
    }
}

// The same row for a hit whose window leaves the haloed image (a hit outside
// its plane): every pixel checked against the plane, zero outside.
__device__ __forceinline__ void load_window_row_checked(const uint16_t *__restrict__ src, const HitDesc &hd, int r,
                                                     uint32_t (&out)[24]) {
    const int w = hd.wc - kHalf + r;
    const bool wok = w >= 0 && w < hd.nwires;
    const uint16_t *rowp = src + hd.d_off + (int64_t)(wok ? w + kHalo : 0) * hd.pitch + kHalo;
#pragma unroll
    for (int j = 0; j < 24; ++j) {
        const int64_t b0 = (int64_t)hd.bc - kHalf + 2 * j;
        const uint32_t lo = (wok && b0 >= 0 && b0 < hd.nint) ? rowp[b0] : 0u;
        const uint32_t hi = (wok && b0 + 1 >= 0 && b0 + 1 < hd.nint) ? rowp[b0 + 1] : 0u;
        out[j] = lo | (hi << 16);
    }
}

// ------------------------------------------------------------------ kernel
// MODE kTcBf16, kTcFp16, or kTcFp8 (bf16 conv, e4m3 dense-1).
template <int MODE>
__global__ void __launch_bounds__(kThreadsTC, 1)
    cnn_tc_kernel(const __grid_constant__ CUtensorMap tmap_w1, const uint16_t *__restrict__ src,
                  const HitDesc *__restrict__ desc, int n,
                  const uint16_t *__restrict__ convB_g, float *__restrict__ partials, int n_pad, long long units,
                  int *status, long long timeout_ns, int debug_stall, int *tile_done,
                  const float *__restrict__ src32) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t base = (raw_u32 + 1023u) & ~1023u;
    uint8_t *gbase = smem_raw + (base - raw_u32);
    const uint32_t sW1 = base + kOffW1;
    const uint32_t sIm = base + kOffIm;
    const uint32_t sConvB = base + kOffConvB;
    auto bar = [&](int i) -> uint32_t { return base + kOffBar + 8u * (uint32_t)i; };
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(gbase + kOffTmemSlot);
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(gbase + kOffAbort);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cta = blockIdx.x;
    const int G = gridDim.x;
    const int64_t u0 = unit_begin(cta, units, G);   // this CTA's units [u0, u1)
    const int64_t u1 = unit_begin(cta + 1, units, G);
    const int nq = (int)(u1 - u0);                  // quads, in order, across tile boundaries
    const int qt0 = (int)(u0 % kW1Steps);           // quad-in-tile and tile of the first unit
    const int tile0 = (int)(u0 / kW1Steps);
    const Guard guard{abort_flag, status, (int64_t)timeout_ns};
    constexpr bool FP16 = MODE == kTcFp16;  // 16-bit format of the conv operands
    constexpr bool F8 = MODE == kTcFp8;     // e4m3 dense-1
    constexpr int kStageTx = F8 ? kW1StageBytesF8 : kW1StageBytes;
    constexpr int kBoxTx = F8 ? kW1BoxBytesF8 : kW1BoxBytes;

    // the next kernel (the head) may be scheduled as SMs free up; it waits for this one
    pdl_trigger();
    // ---- set-up: pair conv B operand into swizzled smem, barriers, TMEM
    for (int idx = threadIdx.x; idx < kPairN * 8; idx += kThreadsTC) {
        const int row = idx >> 3, chunk = idx & 7;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (chunk < kConvK / 8) v = __ldg(reinterpret_cast<const uint4 *>(convB_g + row * kConvK) + chunk);
        *reinterpret_cast<uint4 *>(gbase + kOffConvB + row * 128 + ((chunk ^ (row & 7)) << 4)) = v;
    }
    if (threadIdx.x == 0) {
        for (int i = 0; i < kW1Stages; ++i) {
            mbar_init(bar(kBarW1Full + i), 1);
            mbar_init(bar(kBarW1Empty + i), 1);
        }
        for (int i = 0; i < kImBufs; ++i) {
            mbar_init(bar(kBarImFull + i), 4);
            mbar_init(bar(kBarImFree + i), 1);
        }
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(bar(kBarConv + i), 1);
            mbar_init(bar(kBarAct + i), 4);
            mbar_init(bar(kBarFree + i), 1);
        }
        mbar_init(bar(kBarAcc), 1);
        mbar_init(bar(kBarAccEmpty), 4);
        mbar_init(bar(kBarStall), 1);
        mbar_init(bar(kBarDrain), 2);
        *abort_flag = 0u;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (warp == kConvWarp) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(base + kOffTmemSlot),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == kTmaWarp) {
        // ================================================= TMA producer (W1)
        if (lane == 0) {
            int issued = 0;
            bool ok = true;
            int qt = qt0;
            for (int jj = 0; jj < nq; ++jj, qt = (qt + 1 == kW1Steps) ? 0 : qt + 1) {
                const int wj = jj % kW1Stages;
                const uint32_t use = (uint32_t)(jj / kW1Stages);
                if (jj >= kW1Stages && !wait_bounded(bar(kBarW1Empty + wj), (use - 1u) & 1u, guard)) {
                    ok = false;
                    break;
                }
                if (*abort_flag) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(bar(kBarW1Full + wj), kStageTx);
#pragma unroll
                for (int a = 0; a < kBoxesPerStage; ++a)
                    tma_load_3d(sW1 + wj * kW1StageBytes + a * kBoxTx, &tmap_w1, bar(kBarW1Full + wj), 0, 0,
                                kBoxesPerStage * qt + a);
                ++issued;
            }
            if (!ok) {  // let copies in flight land before the CTA's memory goes away
                for (int jj = issued > kW1Stages ? issued - kW1Stages : 0; jj < issued; ++jj) {
                    const uint32_t b = bar(kBarW1Full + jj % kW1Stages);
                    const uint32_t par = (uint32_t)(jj / kW1Stages) & 1u;
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(b, par) && (int64_t)(global_timer_ns() - t0) < (int64_t)timeout_ns) {
                    }
                }
            }
        }
    } else if (warp == kConvWarp || warp == kFc1Warp) {
        // ====================================================== MMA issuers
        // Two threads issue MMAs, lane 0 of warp kConvWarp (the convs) and lane 0 of
        // warp kFc1Warp (dense-1); each walks its own schedule alone, so that
        // nothing but its waits stands between its groups of MMAs (the tensor
        // pipe's queue is shallow: an issuing thread runs at the pace of
        // execution).  The conv thread issues a pair as soon as its im2col
        // tile and a free TMEM slot exist; the dense-1 thread issues a quad
        // (12 MMAs into the accumulator, the first pair's slot freed after
        // its 6) as soon as both pairs' activations and the W1 stage are in.
        // The slot-free barrier orders a slot's reuse after its dense-1; the
        // activation barrier orders dense-1 after its conv.  Each commit covers
        // all earlier MMAs of its thread.
        if (lane == 0) {
            bool ok = true;
            if (warp == kConvWarp) {
                constexpr uint32_t idesc_conv = make_idesc(128, kPairN, FP16);
                const uint64_t convb_desc = sw128_desc(sConvB);
                if (debug_stall) ok = wait_bounded(bar(kBarStall), 0u, guard);  // nothing arrives here
                for (int q = 0; ok && q < nq; ++q) {
                    const int ib = q % kImBufs;
                    if (!wait_bounded(bar(kBarImFull + ib), (uint32_t)(q / kImBufs) & 1u, guard)) {
                        ok = false;
                        break;
                    }
                    const uint64_t im_desc = sw128_desc(sIm + ib * kImBytes);
                    for (int pr = 0; pr < 2; ++pr) {
                        const int p = 2 * q + pr;
                        const int s = p % kSlots;
                        // the slot's previous pair (p - kSlots) has been read by its dense-1
                        if (p >= kSlots && !wait_bounded(bar(kBarFree + s), (uint32_t)(p / kSlots - 1) & 1u, guard)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem + kSlotCol0 + (uint32_t)s * kSlotCols;
                        const uint64_t ad = im_desc + (uint64_t)((pr * 64) >> 4);
                        mma_ss(d, ad, convb_desc, idesc_conv, 0u);
                        mma_ss(d, ad + (32u >> 4), convb_desc + (32u >> 4), idesc_conv, 1u);
                        mma_commit(bar(kBarConv + s));
                    }
                    if (!ok) break;
                    mma_commit(bar(kBarImFree + ib));
                }
            } else {
                constexpr uint32_t idesc_fc1 = make_idesc(128, kN1, FP16 || F8);
                int tiles_done = 0;  // tile segments whose accumulator was handed to the epilogue
                int qt = qt0 - 1;
                for (int q = 0; ok && q < nq; ++q) {
                    qt = (qt + 1 == kW1Steps) ? 0 : qt + 1;
                    const bool first = (q == 0) || (qt == 0);
                    const bool last = (q == nq - 1) || (qt == kW1Steps - 1);
                    const int wj = q % kW1Stages;
                    const int s0 = (2 * q) % kSlots, s1 = (2 * q + 1) % kSlots;
                    const uint32_t par = (uint32_t)((2 * q) / kSlots) & 1u;  // same use for both slots
                    if (!wait_bounded(bar(kBarW1Full + wj), (uint32_t)(q / kW1Stages) & 1u, guard) ||
                        !wait_bounded(bar(kBarAct + s0), par, guard)) {
                        ok = false;
                        break;
                    }
                    // a new tile starts from zero in the accumulator, once the epilogue drained the last one
                    if (first && tiles_done > 0 &&
                        !wait_bounded(bar(kBarAccEmpty), (uint32_t)(tiles_done - 1) & 1u, guard)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // K steps of 32 bytes per row: 16 inputs (16 bit) or 32 (e4m3); a pair's 96
                    // inputs are 6 or 3 steps, 8 TMEM columns each
                    constexpr int kSteps = F8 ? 6 : 12;
                    constexpr int kHalf = kSteps / 2;
                    constexpr int kStepsPerBox = kW1Box * (F8 ? 1 : 2) / 32;
                    const uint64_t wdesc = F8 ? sw64_desc(sW1 + wj * kW1StageBytes) : sw128_desc(sW1 + wj * kW1StageBytes);
#pragma unroll
                    for (int step = 0; step < kSteps; ++step) {
                        // the second pair's activations are waited for only when its half begins
                        if (step == kHalf) {
                            if (!wait_bounded(bar(kBarAct + s1), par, guard)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        }
                        const uint32_t a =
                            tmem + kSlotCol0 + (uint32_t)(step < kHalf ? s0 : s1) * kSlotCols + 8u * (step % kHalf);
                        const uint64_t bd = wdesc + (uint64_t)(((step / kStepsPerBox) * kBoxTx +
                                                                (step % kStepsPerBox) * 32) >> 4);
                        if (F8)
                            mma_ts_f8(tmem + kAccCol, a, bd, idesc_fc1, (first && step == 0) ? 0u : 1u);
                        else
                            mma_ts(tmem + kAccCol, a, bd, idesc_fc1, (first && step == 0) ? 0u : 1u);
                        if (step == kHalf - 1) mma_commit(bar(kBarFree + s0));
                    }
                    if (!ok) break;
                    mma_commit(bar(kBarFree + s1));
                    mma_commit(bar(kBarW1Empty + wj));
                    if (last) {
                        mma_commit(bar(kBarAcc));
                        ++tiles_done;
                    }
                }
            }
            // every MMA either thread issued completes before TMEM is released:
            // the drain barrier expects one commit from each issuer
            mma_commit(bar(kBarDrain));
            const uint64_t t0 = global_timer_ns();
            while (!mbar_try_wait(bar(kBarDrain), 0u) && (int64_t)(global_timer_ns() - t0) < (int64_t)timeout_ns) {
            }
        }
        __syncwarp();
    } else if (builder_index(warp) >= 0) {
        // ================================================ im2col builder
        // Row r of an im2col tile (hit r) is 128 bytes: pair (x, x+1) in
        // chunks 0-3, pair (x+2, x+3) in chunks 4-7; 16-byte chunk c sits at
        // chunk c ^ (r & 7) (128-byte swizzle).  Tap t = 6i + j of a pair at x
        // is patch pixel (y + i, x + j); taps 30 and 31 are 1.0.  Because x is
        // even, taps (2k, 2k+1) are one aligned pixel pair of the patch row.
        const int q4 = builder_index(warp);
        const int row = 32 * q4 + lane;
        const uint32_t one = FP16 ? 0x3C00u : 0x3F80u;
        pdl_wait();  // the images and window descriptors come from the kernel before
        const uint32_t ones = one | (one << 16);
        uint8_t *my_row = gbase + kOffIm + row * 128;
        bool ok = true;
        const int t_first = tile0;
        const int t_last = nq > 0 ? (int)((u1 - 1) / kW1Steps) : t_first - 1;
        for (int tile = t_first; ok && tile <= t_last; ++tile) {
        const int j0 = tile == t_first ? qt0 : 0;   // quads of this tile in [j0, j1)
        const int j1 = tile == t_last ? (int)((u1 - 1) % kW1Steps) + 1 : kW1Steps;
        const int64_t k_base = (int64_t)tile * kW1Steps - u0;        // running quad index = k_base + quad
        const int64_t hit = (int64_t)tile * 128 + row;
        const bool valid = hit < n;
        // the hit's window: a patch of the patch buffer, or a window of its plane's image
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
        const int y_first = j0 * kPosPerW1 / kQ;
        const int y_last = (j1 * kPosPerW1 - 1) / kQ;
        // window row r of this hit, 2 pixels per word
        auto load_row = [&](int r, uint32_t(&out)[24]) {
            if (!valid) {
#pragma unroll
                for (int j = 0; j < 24; ++j) out[j] = 0u;
            } else if (src32 != nullptr) {
                load_patch_row_f32<FP16>(src32, hd.origin + (int64_t)r * kPatch, out);
            } else if (hd.inside) {
                load_window_row(src, hd.origin + (int64_t)r * hd.pitch, out);
            } else {
                load_window_row_checked(src, hd, r, out);
            }
        };
        // rows y..y+4, slid down one row per y: each window row is loaded once
        uint32_t R[kK][24];
        if (valid && hd.inside && src32 == nullptr) {
            load_window_rows5(src, hd.origin + (int64_t)y_first * hd.pitch, hd.pitch, R);
        } else {
#pragma unroll
            for (int i = 0; i < kK; ++i) load_row(y_first + i, R[i]);
        }
        for (int y = y_first; ok && y <= y_last; ++y) {
            if (y > y_first) {
#pragma unroll
                for (int i = 0; i < kK - 1; ++i)
#pragma unroll
                    for (int j = 0; j < 24; ++j) R[i][j] = R[i + 1][j];
                load_row(y + kK - 1, R[kK - 1]);
            }
#pragma unroll
            for (int xq = 0; xq < kQ / kPosPerW1; ++xq) {
                const int quad = (y * kQ) / kPosPerW1 + xq;
                if (quad < j0 || quad >= j1) continue;
                const int k = (int)(k_base + quad);
                const int ib = k % kImBufs;
                if (k >= kImBufs &&
                    !warp_wait(bar(kBarImFree + ib), (uint32_t)(k / kImBufs - 1) & 1u, guard, lane)) {
                    ok = false;
                    break;
                }
                uint8_t *dst = my_row + ib * kImBytes;
#pragma unroll
                for (int c = 0; c < 8; ++c) {  // chunk c: pair c/4, taps 8(c%4) .. 8(c%4)+7
                    const int x = 4 * xq + 2 * (c >> 2);
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int kw = 4 * (c & 3) + e;  // word kw: taps 2kw, 2kw+1
                        if (kw == 15) {
                            w[e] = ones;
                        } else {
                            const int i = kw / 3, jp = kw % 3;  // row i, columns x + 2jp, x + 2jp + 1
                            w[e] = R[i][(x >> 1) + jp];
                        }
                    }
                    *reinterpret_cast<uint4 *>(dst + ((c ^ (row & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarImFull + ib));
            }
        }
        }
    } else {
        // ================================== conv epilogue + dense-1 store
        const int q4 = warp & 3;
        const uint32_t lane_tmem = tmem + ((uint32_t)(32 * q4) << 16);
        bool ok = true;
        int tiles_done = 0;
        int qt = qt0;       // quad-in-tile of pair pi
        for (int pi = 0; pi < 2 * nq; ++pi) {
            const int s = pi % kSlots;
            if (!warp_wait(bar(kBarConv + s), (uint32_t)(pi / kSlots) & 1u, guard, lane)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t d = lane_tmem + kSlotCol0 + (uint32_t)s * kSlotCols;
            if (F8) {  // both positions -> 96 e4m3 bytes = 24 words
                uint32_t o[24];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t f[48];
                    tmem_ld16<0>(d + 48u * h, f);
                    tmem_ld16<16>(d + 48u * h + 16u, f);
                    tmem_ld16<32>(d + 48u * h + 32u, f);
                    tmem_ld_wait();
                    reg_fence(f);
                    // the conv weights and bias carry kFp8ActScale, so f is already scaled
#pragma unroll
                    for (int i = 0; i < 12; ++i)
                        o[12 * h + i] = relu_e4m3x4(f[4 * i], f[4 * i + 1], f[4 * i + 2], f[4 * i + 3]);
                }
                tmem_st16<0>(d, o);
                tmem_st8<16>(d + 16u, o);
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h) {  // position x, then x+1: 48 fp32 -> 24 packed words
                    uint32_t f[48];
                    tmem_ld16<0>(d + 48u * h, f);
                    tmem_ld16<16>(d + 48u * h + 16u, f);
                    tmem_ld16<32>(d + 48u * h + 32u, f);
                    tmem_ld_wait();
                    reg_fence(f);
                    uint32_t o[24];
#pragma unroll
                    for (int i = 0; i < 24; ++i) o[i] = relu_pack<FP16>(f[2 * i], f[2 * i + 1]);
                    tmem_st16<0>(d + 24u * h, o);
                    tmem_st8<16>(d + 24u * h + 16u, o);
                }
            }
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarAct + s));
            // after a tile's last pair: drain its dense-1 accumulator to the partial-sum row
            const bool tile_end = (pi & 1) && ((pi >> 1) == nq - 1 || qt == kW1Steps - 1);
            if (pi & 1) qt = (qt + 1 == kW1Steps) ? 0 : qt + 1;
            if (tile_end) {
                if (!warp_wait(bar(kBarAcc), (uint32_t)tiles_done & 1u, guard, lane)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int64_t tile = tile0 + tiles_done;
                const int krow = cta - cta_of_unit(tile * kW1Steps, units, G);
                // this warp's 32 hits (rows 32 q4 ...) of the tile, 32 outputs at a time
                const int64_t hit0 = tile * 128 + 32 * q4;
                float *dst0 = partials + ((int64_t)krow * n_pad + hit0) * kN1;
                float *stage = reinterpret_cast<float *>(gbase + kOffStageA + q4 * kStageBytes);
#pragma unroll 1
                for (int c = 0; c < kN1 / 32; ++c) {
                    uint32_t r[32];
                    tmem_ld16<0>(lane_tmem + kAccCol + 32u * c, r);
                    tmem_ld16<16>(lane_tmem + kAccCol + 32u * c + 16u, r);
                    tmem_ld_wait();
                    reg_fence(r);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        *reinterpret_cast<uint4 *>(stage + lane * kStagePitch + 4 * e) =
                            make_uint4(r[4 * e], r[4 * e + 1], r[4 * e + 2], r[4 * e + 3]);
                    __syncwarp();
                    // lane l: row 4 k + l / 8, outputs 32 c + 4 (l % 8) ... + 3
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        const int i = 4 * k + (lane >> 3);
                        const float4 v = *reinterpret_cast<const float4 *>(stage + i * kStagePitch + 4 * (lane & 7));
                        if (hit0 + i < n)
                            *reinterpret_cast<float4 *>(dst0 + (int64_t)i * kN1 + 32 * c + 4 * (lane & 7)) = v;
                    }
                    __syncwarp();
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarAccEmpty));
                if (tile_done != nullptr) {  // this warp's rows of the tile are stored: count them for the head
                    __threadfence();
                    __syncwarp();
                    if (lane == 0) atomicAdd(tile_done + tile, 1);
                }
                ++tiles_done;
            }
        }
        (void)ok;
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kConvWarp) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

uint16_t to16(float v, bool fp16) {
    if (fp16) {
        __half h = __float2half_rn(v);
        return *reinterpret_cast<uint16_t *>(&h);
    }
    __nv_bfloat16 b = __float2bfloat16_rn(v);
    return *reinterpret_cast<uint16_t *>(&b);
}
float from16(uint16_t u, bool fp16) {
    if (fp16) {
        __half h;
        *reinterpret_cast<uint16_t *>(&h) = u;
        return __half2float(h);
    }
    __nv_bfloat16 b;
    *reinterpret_cast<uint16_t *>(&b) = u;
    return __bfloat162float(b);
}

}  // namespace

cudaError_t init_tc_kernel_attrs() {
    cudaError_t e = cudaFuncSetAttribute(cnn_tc_kernel<kTcBf16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytesTC);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(cnn_tc_kernel<kTcFp16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytesTC);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(cnn_tc_kernel<kTcFp8>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytesTC);
    return e;
}

double fp8_weight_scale(const float *fc1_w, size_t n) {
    float m = 0.0f;
    for (size_t i = 0; i < n; ++i) m = std::fmax(m, std::fabs(fc1_w[i]));
    if (!(m > 0.0f) || !std::isfinite(m)) return 1.0;
    // largest 2^k with m * 2^k <= 448, the largest finite e4m3 value
    int k = 0;
    while (k < 126 && (double)m * std::ldexp(1.0, k + 1) <= 448.0) ++k;
    while (k > -126 && (double)m * std::ldexp(1.0, k) > 448.0) --k;
    return std::ldexp(1.0, k);
}

cudaError_t prepare_tc_weights(DeviceWeights &w, const emtk_weights &hw, TcMode mode) {
    const bool fp16 = mode == kTcFp16;
    const bool f8 = mode == kTcFp8;
    const size_t nw1 = (size_t)kFc1In * kN1;
    // dense-1 weights, tiled [K/64][128][64] so that each TMA box is one
    // contiguous 16 KB (or 8 KB in e4m3): tile kb holds W1[kb*64 + kk][nn] at
    // [kb][nn][kk].
    std::vector<uint16_t> tiles(f8 ? 0 : nw1);
    std::vector<uint8_t> tiles8(f8 ? nw1 : 0);
    const float sw = f8 ? (float)fp8_weight_scale(hw.fc1_w, nw1) : 1.0f;
    for (int kb = 0; kb < kKBlocks; ++kb)
        for (int nn = 0; nn < kN1; ++nn)
            for (int kk = 0; kk < kW1Box; ++kk) {
                const size_t t = ((size_t)kb * kN1 + nn) * kW1Box + kk;
                const float v = hw.fc1_w[(size_t)(kb * kW1Box + kk) * kN1 + nn];
                if (f8)
                    tiles8[t] = (uint8_t)__nv_cvt_float_to_fp8(v * sw, __NV_SATFINITE, __NV_E4M3);
                else
                    tiles[t] = to16(v, fp16);
            }
    w.fc1_scale = f8 ? 1.0f / (kFp8ActScale * sw) : 1.0f;
    w.fc1_w_scale = sw;
    // pair conv B operand [96][32]: row f (< 48) is filter f at x, row 48 + f
    // filter f at x + 1; tap t = 6i + j reads window column j; taps 30 and 31
    // carry the bias split into a 16-bit head and a 16-bit remainder.  In
    // e4m3 mode weights and bias are multiplied by the activation scale (a
    // power of two: the rounding to bf16 and the fp32 sums scale exactly).
    const float cs = f8 ? kFp8ActScale : 1.0f;
    std::vector<uint16_t> cb((size_t)kPairN * kConvK, 0);
    for (int f = 0; f < kF; ++f) {
        for (int i = 0; i < kK; ++i)
            for (int j = 0; j < kK; ++j) {
                const uint16_t wv = to16(hw.conv_w[(i * kK + j) * kF + f] * cs, fp16);
                cb[(size_t)f * kConvK + 6 * i + j] = wv;              // position x: window columns 0..4
                cb[(size_t)(kF + f) * kConvK + 6 * i + j + 1] = wv;   // position x+1: window columns 1..5
            }
        const uint16_t hi = to16(hw.conv_b[f] * cs, fp16);
        const uint16_t lo = to16(hw.conv_b[f] * cs - from16(hi, fp16), fp16);
        for (int h = 0; h < 2; ++h) {
            cb[(size_t)(h * kF + f) * kConvK + 30] = hi;
            cb[(size_t)(h * kF + f) * kConvK + 31] = lo;
        }
    }
    const size_t w1_bytes = f8 ? nw1 : nw1 * 2;
    cudaError_t e = dev_alloc(&w.w1_tiles, w1_bytes);
    if (e != cudaSuccess) return e;
    e = cudaMemcpy(w.w1_tiles, f8 ? (const void *)tiles8.data() : (const void *)tiles.data(), w1_bytes,
                   cudaMemcpyHostToDevice);
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
    CUtensorMap *map = new CUtensorMap[1];
    cuuint64_t dims[3] = {(cuuint64_t)kW1Box, (cuuint64_t)kN1, (cuuint64_t)kKBlocks};
    const cuuint64_t esz = f8 ? 1 : 2;  // bytes per weight
    cuuint64_t strides[2] = {(cuuint64_t)kW1Box * esz, (cuuint64_t)kW1Box * kN1 * esz};
    cuuint32_t box[3] = {(cuuint32_t)kW1Box, (cuuint32_t)kN1, 1u};
    cuuint32_t estr[3] = {1u, 1u, 1u};
    // a box row is 128 bytes (16 bit) or 64 bytes (e4m3): the swizzle span matches it
    CUresult r = encode(map, f8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, w.w1_tiles,
                        dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        f8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        delete[] map;
        return cudaErrorInvalidValue;
    }
    w.w1_tmap = map;
    return cudaSuccess;
}

// Partial-sum rows a stream-K launch over G CTAs needs: the largest number
// of CTAs that share one tile.
int streamk_partial_rows(int32_t n, int G) {
    const int m_tiles = (n + 127) / 128;
    const int64_t units = (int64_t)m_tiles * kW1Steps;
    int rows = 1;
    for (int t = 0; t < m_tiles; ++t) {
        const int a = cta_of_unit((int64_t)t * kW1Steps, units, G);
        const int b = cta_of_unit((int64_t)t * kW1Steps + kW1Steps - 1, units, G);
        rows = b - a + 1 > rows ? b - a + 1 : rows;
    }
    return rows;
}

cudaError_t launch_cnn_tc(const DeviceWeights &w, const void *src, const HitDesc *desc, TcMode mode, int32_t n,
                          int G, float *partials, int n_pad, int *status, int64_t timeout_ns, int debug_stall,
                          int *tile_done, const float *src32, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const CUtensorMap &map = *static_cast<const CUtensorMap *>(w.w1_tmap);
    const long long units = (long long)((n + 127) / 128) * kW1Steps;
    const uint16_t *src16 = static_cast<const uint16_t *>(src);
    dim3 grid(G);
    if (mode == kTcSplit)
        return launch_cnn_split(w, src, desc, n, G, partials, n_pad, status, timeout_ns, debug_stall, tile_done, s);
    auto *kernel = mode == kTcFp16 ? cnn_tc_kernel<kTcFp16> : mode == kTcFp8 ? cnn_tc_kernel<kTcFp8>
                                                                              : cnn_tc_kernel<kTcBf16>;
    const uint16_t *convB = w.convB;
    const long long tmo = (long long)timeout_ns;
    return launch_pdl(kernel, grid, dim3(kThreadsTC), kSmemBytesTC, s, map, src16, desc, n, convB, partials, n_pad,
                      units, status, tmo, debug_stall, tile_done, src32);
}

}  // namespace emtk
