// Hit finding on the deconvolved waveforms (Sec. 2.1; the rule is stated in
// include/emtk.h): per wire, each maximal run of ticks above the threshold
// is one hit at the run's largest value.
//
// Work units are wire segments of kSegTicks ticks (a wire of 6000 ticks is 3
// units), in order: plane, wire, segment.  A run belongs to the segment that
// holds its first tick.  Three kernels per group of planes:
//   hf_find_kernel   one warp per unit: reads the segment in coalesced
//                    512-byte rows (lane l holds ticks 4l .. 4l+3 of each
//                    128-tick block) and finds the run starts, ticks above
//                    the threshold whose previous tick is not (the tick
//                    before the segment is read; before tick 0 counts as
//                    below).  The lane holding a start walks the run forward,
//                    past the segment's end if the run goes on (cached loads
//                    of rows just read), for its end, peak and fp32 charge,
//                    and keeps the unit's first kRunSlots runs in scratch
//                    slots; it writes the unit's run count;
//   hf_scan_kernel   one CTA per plane: exclusive scan of its units' counts
//                    (offsets within the plane) and the plane's total;
//   hf_place_kernel  one warp per unit: copies its runs from the slots to the
//                    output at the unit's offset; a unit with more runs than
//                    slots is scanned again and written directly.
// The plane is read once from HBM (plus units with more than kRunSlots
// runs).  Outputs are ordered by wire, then tick, whatever the launch shape.
#include <cmath>

#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kHfWarps = 8;     // warps (units) per CTA in the two passes
constexpr int kHfSub = 4;       // 128-tick blocks loaded per iteration (4 loads in flight per lane)
constexpr int kScanThreads = 1024;
constexpr int kRunSlots = 32;   // runs per unit kept by the first pass (more: the unit is scanned again)
constexpr unsigned kFull = 0xffffffffu;
static_assert(kSegTicks % (128 * kHfSub) == 0, "a segment is whole load blocks");

__device__ __forceinline__ int find_plane(const HfTable &t, int64_t u) {
    int r = 0;
    while (r + 1 < t.n && t.r[r + 1].unit0 <= u) ++r;
    return r;
}

// Ticks t0 .. t0+3 of a row; ticks at or past `lim` read as -inf (below any
// threshold).  row + t0 is 16-byte aligned (aligned base, ld % 4 == 0, t0 % 4 == 0).
__device__ __forceinline__ float4 load4(const float *__restrict__ row, int t0, int lim) {
    if (t0 + 3 < lim) return __ldg(reinterpret_cast<const float4 *>(row + t0));
    float4 v = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    if (t0 < lim) v.x = __ldg(row + t0);
    if (t0 + 1 < lim) v.y = __ldg(row + t0 + 1);
    if (t0 + 2 < lim) v.z = __ldg(row + t0 + 2);
    return v;
}

// Run starts among a lane's 4 ticks (bit j: tick 4*lane + j of the block);
// `prev` is whether the block's tick -1 is above (lane 0), updated to
// whether its last tick is above (for the next block).
__device__ __forceinline__ uint32_t starts4(const float4 v, float thr, int lane, bool &prev) {
    const bool a0 = v.x > thr, a1 = v.y > thr, a2 = v.z > thr, a3 = v.w > thr;
    const bool left = __shfl_up_sync(kFull, a3, 1);
    const bool p = lane == 0 ? prev : left;
    prev = __shfl_sync(kFull, a3, 31);
    return (uint32_t)(a0 && !p) | ((uint32_t)(a1 && !a0) << 1) | ((uint32_t)(a2 && !a1) << 2) |
           ((uint32_t)(a3 && !a2) << 3);
}

// A run found on a wire: its tick range, peak tick and value, fp32 charge.
struct Run {
    int32_t start, end, tick;
    float peak, charge;
};

// Walks the wire row from run start t0 (above the threshold) to the run's
// end: values in tick order, the first maximum kept.
__device__ __forceinline__ Run walk_run(const float *__restrict__ row, int t0, int nticks, float thr) {
    Run r{t0, t0, t0, -INFINITY, 0.0f};
    int tt = t0;
    while (tt < nticks) {
        const float x = __ldg(row + tt);
        if (!(x > thr)) break;
        if (x > r.peak) {
            r.peak = x;
            r.tick = tt;
        }
        r.charge += x;
        ++tt;
    }
    r.end = tt - 1;
    return r;
}

// The unit of a plane: its wire's row and tick range [t0, t1).
struct Unit {
    const float *row;
    int32_t wire, t0, t1;
};
__device__ __forceinline__ Unit unit_of(const HfDesc &d, int64_t u) {
    const int64_t local = u - d.unit0;
    const int32_t w = (int32_t)(local / d.nseg), seg = (int32_t)(local % d.nseg);
    const int32_t t0 = seg * kSegTicks;
    return Unit{d.adc + (int64_t)w * d.ld, w, t0, t0 + kSegTicks < d.nticks ? t0 + kSegTicks : d.nticks};
}

// All runs that start in the unit, in tick order: sink(k, run) for the k-th.
// Returns their number (the same in every lane).
template <class Sink>
__device__ __forceinline__ int32_t scan_unit(const Unit &un, int nticks, float thr, int lane, Sink sink) {
    int32_t next = 0;
    bool prev = un.t0 > 0 && __ldg(un.row + un.t0 - 1) > thr;
    for (int base = un.t0; base < un.t1; base += 128 * kHfSub) {
        float4 v[kHfSub];
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) v[k] = load4(un.row, base + 128 * k + 4 * lane, un.t1);
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) {
            uint32_t m = starts4(v[k], thr, lane, prev);
            const int c = __popc(m);
            int incl = c;  // inclusive scan of the lanes' start counts
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += y;
            }
            int32_t idx = next + incl - c;
            next += __shfl_sync(kFull, incl, 31);
            while (m) {
                const int j = __ffs(m) - 1;
                m &= m - 1;
                sink(idx++, walk_run(un.row, base + 128 * k + 4 * lane + j, nticks, thr));
            }
        }
    }
    return next;
}

__device__ __forceinline__ void put_hit(const HfDesc &d, int32_t w, int32_t idx, const Run &r) {
    if (idx >= d.capacity) return;
    d.hits[idx] = emtk_hit{w, r.tick};
    if (d.info) d.info[idx] = emtk_hit_info{r.start, r.end, r.peak, r.charge};
}

__global__ void __launch_bounds__(kHfWarps * 32) hf_find_kernel(const HfTable t, int64_t nunits,
                                                                int32_t *__restrict__ counts,
                                                                Run *__restrict__ slots) {
    const int lane = threadIdx.x & 31;
    const int64_t u = (int64_t)blockIdx.x * kHfWarps + (threadIdx.x >> 5);
    if (u >= nunits) return;  // the whole warp leaves together
    const HfDesc &d = t.r[find_plane(t, u)];
    const Unit un = unit_of(d, u);
    Run *my = slots + u * kRunSlots;
    const int32_t n = scan_unit(un, d.nticks, d.thr, lane, [&](int32_t k, const Run &r) {
        if (k < kRunSlots) my[k] = r;
    });
    if (lane == 0) counts[u] = n;
}

// Block r: offsets[u] = hits of plane r in its units before u; total[r] =
// the plane's hits.  Units in chunks of kScanThreads, one per thread.
__global__ void __launch_bounds__(kScanThreads) hf_scan_kernel(const HfTable t, int64_t nunits,
                                                               const int32_t *__restrict__ counts,
                                                               int32_t *__restrict__ offsets,
                                                               int32_t *__restrict__ total) {
    __shared__ int32_t warp_sum[kScanThreads / 32];
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t u0 = t.r[r].unit0, u1 = r + 1 < t.n ? t.r[r + 1].unit0 : nunits;
    int32_t carry = 0;  // fits: the host bounds a plane's runs by 2^31 - 1
    for (int64_t c0 = u0; c0 < u1; c0 += kScanThreads) {
        const int64_t u = c0 + tid;
        const int32_t v = u < u1 ? counts[u] : 0;
        int32_t incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) warp_sum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int32_t ws = warp_sum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(kFull, ws, o);
                if (lane >= o) ws += y;
            }
            warp_sum[lane] = ws;  // inclusive over warps
        }
        __syncthreads();
        const int32_t before = (warp > 0 ? warp_sum[warp - 1] : 0) + incl - v;
        if (u < u1) offsets[u] = carry + before;
        carry += warp_sum[kScanThreads / 32 - 1];
        __syncthreads();  // warp_sum is rewritten by the next chunk
    }
    if (tid == 0) total[r] = carry;
}

__global__ void __launch_bounds__(kHfWarps * 32) hf_place_kernel(const HfTable t, int64_t nunits,
                                                                 const int32_t *__restrict__ counts,
                                                                 const int32_t *__restrict__ offsets,
                                                                 const Run *__restrict__ slots) {
    const int lane = threadIdx.x & 31;
    const int64_t u = (int64_t)blockIdx.x * kHfWarps + (threadIdx.x >> 5);
    if (u >= nunits) return;
    const HfDesc &d = t.r[find_plane(t, u)];
    const Unit un = unit_of(d, u);
    const int32_t n = counts[u], off = offsets[u];
    if (n <= kRunSlots) {
        for (int k = lane; k < n; k += 32) put_hit(d, un.wire, off + k, slots[u * kRunSlots + k]);
    } else {  // more runs than slots: scan the unit again
        scan_unit(un, d.nticks, d.thr, lane, [&](int32_t k, const Run &r) { put_hit(d, un.wire, off + k, r); });
    }
}

}  // namespace

size_t find_hits_scratch_bytes(int64_t nunits) {
    return (size_t)nunits * (2 * sizeof(int32_t) + kRunSlots * sizeof(Run));
}

cudaError_t launch_find_hits(const HfTable &t, int64_t nunits, void *scratch, int32_t *totals, cudaStream_t s) {
    if (nunits <= 0) return cudaMemsetAsync(totals, 0, sizeof(int32_t) * kMaxHfPlanes, s);
    // scratch: run slots [units][kRunSlots], then counts [units] and offsets [units]
    Run *slots = static_cast<Run *>(scratch);
    int32_t *counts = reinterpret_cast<int32_t *>(slots + nunits * kRunSlots);
    int32_t *offsets = counts + nunits;
    const unsigned blocks = (unsigned)((nunits + kHfWarps - 1) / kHfWarps);
    hf_find_kernel<<<blocks, kHfWarps * 32, 0, s>>>(t, nunits, counts, slots);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    hf_scan_kernel<<<t.n, kScanThreads, 0, s>>>(t, nunits, counts, offsets, totals);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    hf_place_kernel<<<blocks, kHfWarps * 32, 0, s>>>(t, nunits, counts, offsets, slots);
    return cudaGetLastError();
}

}  // namespace emtk
