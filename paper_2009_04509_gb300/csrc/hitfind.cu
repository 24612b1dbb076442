// Hit finding on the deconvolved waveforms (Sec. 2.1; the rule is stated in
// include/emtk.h): per wire, each maximal run of ticks above the threshold
// is one hit at the run's largest value.
//
// Work units are wire segments of kSegTicks ticks (a wire of 6000 ticks is 3
// units), in order: plane, wire, segment.  A run belongs to the segment that
// holds its first tick.  Two kernels per group of planes:
//   hf_find_kernel   one warp per unit: reads the segment in coalesced
//                    512-byte rows (lane l holds ticks 4l .. 4l+3 of each
//                    128-tick block), four rows in flight; a 512-tick stretch
//                    with nothing above the threshold is passed over after
//                    one vote.  Otherwise each block finds its run starts (a
//                    tick above whose previous tick is not; the tick before
//                    the segment is read, before tick 0 counts as below).  A
//                    run that ends within its lane's 4 ticks is measured by
//                    that lane from registers; a run that goes past them is
//                    walked by the whole warp, 32 ticks per step, past the
//                    segment's end if it goes on (the stretch's samples from
//                    a shared-memory copy, later ticks from global memory).
//                    The warp keeps the unit's first kRunSlots runs in
//                    scratch slots, writes its run count and adds it to its
//                    chunk's sum (chunks: kHfChunk consecutive units of one
//                    plane);
//   hf_place_kernel  one CTA per chunk, a thread per unit: a unit's offset in
//                    its plane is the sum of the plane's earlier chunks plus
//                    a block scan of the chunk's counts.  The chunk's runs in
//                    the slots are then shared out evenly: thread i copies
//                    runs i, i + kHfChunk, ... of the chunk (its unit found by
//                    binary search of the scanned counts), so consecutive
//                    threads write consecutive hits.  A unit with more runs
//                    than slots is scanned again by a warp and written
//                    directly.  The plane's last unit writes its total.
// The chunk sums start at zero: the place kernel of the launch before cleared
// them (they alternate between two arrays of the context).  The plane is read
// once from HBM (plus units with more than kRunSlots runs).  No kernel waits
// on another CTA.  Outputs are ordered by wire, then tick, whatever the
// launch shape.  The samples are read with the streaming (evict-first) hint:
// each is used once, apart from walks of runs that go past a lane's 4 ticks,
// which read the stretch's shared-memory copy.
#include <cmath>

#include "emtk_internal.h"

namespace emtk {
namespace {

constexpr int kHfWarps = 4;     // warps (units) per CTA of the find kernel
constexpr int kHfSub = 4;       // 128-tick blocks loaded per step (4 loads in flight per lane)
constexpr int kRunSlots = 128;  // runs per unit kept in scratch (more: the unit is scanned again)
constexpr int kHfChunk = 128;   // units per chunk: threads per CTA of the place kernel
constexpr unsigned kFull = 0xffffffffu;
static_assert(kSegTicks % (128 * kHfSub) == 0, "a segment is whole load blocks");

// Scratch: per unit its run count and run slots.

__device__ __forceinline__ int find_plane(const HfTable &t, int64_t u) {
    int r = 0;
    while (r + 1 < t.n && t.r[r + 1].unit0 <= u) ++r;
    return r;
}

// Ticks t0 .. t0+3 of a row; ticks at or past `lim` read as -inf (below any
// threshold).  row + t0 is 16-byte aligned (aligned base, ld % 4 == 0, t0 % 4 == 0).
__device__ __forceinline__ float4 load4(const float *__restrict__ row, int t0, int lim) {
    if (t0 + 3 < lim) return __ldcs(reinterpret_cast<const float4 *>(row + t0));
    float4 v = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    if (t0 < lim) v.x = __ldg(row + t0);
    if (t0 + 1 < lim) v.y = __ldg(row + t0 + 1);
    if (t0 + 2 < lim) v.z = __ldg(row + t0 + 2);
    return v;
}

// A run found on a wire: its tick range, peak tick and value, fp32 charge.
struct Run {
    int32_t start, end, tick;
    float peak, charge;
};

// Orders floats as unsigned integers: x < y gives key(x) < key(y) for
// non-NaN x, y (-0 below +0), and key_value inverts it.
__device__ __forceinline__ uint32_t order_key(float x) {
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// The run that starts at tick ts (above the threshold), walked by the whole
// warp 32 ticks per step: each step's leading ticks above the threshold are
// the run's; the step's largest value (first lane among equals, float
// comparison, so -0 and +0 tie) replaces the peak only if strictly larger,
// which keeps the first maximum of the run; the charge adds each step's
// pairwise sum in step order.  Every lane returns the same run.
template <class Src>
__device__ __forceinline__ Run warp_walk(const Src &src, int ts, int nticks, float thr, int lane) {
    Run r{ts, ts, ts, -INFINITY, 0.0f};
    for (int t = ts;; t += 32) {
        const int tt = t + lane;
        const float x = tt < nticks ? src.tick(tt) : -INFINITY;
        const uint32_t below = __ballot_sync(kFull, !(x > thr));
        const int len = below ? __ffs(below) - 1 : 32;
        if (len == 0) break;  // the run ended on the previous step's last tick
        const bool in = lane < len;
        // run values are > thr, never NaN: key 0 (a NaN) is below all of them
        const float fm = key_value(__reduce_max_sync(kFull, in ? order_key(x) : 0u));
        const int first = __ffs(__ballot_sync(kFull, in && x == fm)) - 1;
        const float pk = __shfl_sync(kFull, x, first);
        if (pk > r.peak) {
            r.peak = pk;
            r.tick = t + first;
        }
        float c = in ? x : 0.0f;
#pragma unroll
        for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(kFull, c, o);  // same sum in every lane
        r.charge += c;
        r.end = t + len - 1;
        if (len < 32) break;
    }
    return r;
}

// The unit of a plane: its wire's row and tick range [t0, t1).
struct Unit {
    const float *row;
    int32_t wire, t0, t1;
};
__device__ __forceinline__ Unit unit_of(const HfDesc &d, int64_t u) {
    // a plane's units fit 32 bits (a plane in device memory holds < 2^31 x 2048 samples)
    const uint32_t local = (uint32_t)(u - d.unit0), nseg = (uint32_t)d.nseg;
    const int32_t w = (int32_t)(local / nseg), seg = (int32_t)(local % nseg);
    const int32_t t0 = seg * kSegTicks;
    return Unit{d.adc + (int64_t)w * d.ld, w, t0, t0 + kSegTicks < d.nticks ? t0 + kSegTicks : d.nticks};
}

// The samples of a unit's wire row.  A 512-tick stretch that holds a run
// start is also kept in the warp's shared-memory stash (ticks [sbase, send))
// for the walks; other ticks come from global memory.
struct Src {
    const float *row;
    int32_t t1;       // the unit's end
    float *stash;     // 512 floats of the warp
    int32_t sbase, send;
    // ticks t .. t+3 (t % 4 == 0): -inf at or past t1
    __device__ __forceinline__ float4 group(int t) const { return load4(row, t, t1); }
    // tick tt (tt < nticks)
    __device__ __forceinline__ float tick(int tt) const {
        return (tt >= sbase && tt < send) ? stash[tt - sbase] : __ldg(row + tt);
    }
};

// All runs that start in the unit, in tick order: sink(k, run) for the k-th,
// called by one lane per run.  Returns their number (the same in every lane).
template <class Sink>
__device__ __forceinline__ int32_t scan_unit(const Unit &un, Src src, int nticks, float thr, int lane, Sink sink) {
    int32_t next = 0;
    // the tick before the current block, as a value compared with thr: the
    // sample itself for the unit's first block, else +inf (above) or -inf
    float before = un.t0 > 0 ? __ldg(un.row + un.t0 - 1) : -INFINITY;
    const uint32_t lt = (1u << lane) - 1u;  // lanes below this one
    for (int base = un.t0; base < un.t1; base += 128 * kHfSub) {
        float4 v[kHfSub];
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) v[k] = src.group(base + 128 * k + 4 * lane);
        // fmaxf skips NaN, which is never above
        bool hot[kHfSub];
        bool any_hot = false;
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) {
            hot[k] = fmaxf(fmaxf(v[k].x, v[k].y), fmaxf(v[k].z, v[k].w)) > thr;
            any_hot = any_hot || hot[k];
        }
        if (!__any_sync(kFull, any_hot)) {
            before = -INFINITY;  // the stretch's last tick is below
            continue;
        }
        __syncwarp();  // the previous stretch's walks are done with the stash
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) reinterpret_cast<float4 *>(src.stash)[32 * k + lane] = v[k];
        __syncwarp();
        src.sbase = base;
        src.send = base + 128 * kHfSub < un.t1 ? base + 128 * kHfSub : un.t1;
#pragma unroll
        for (int k = 0; k < kHfSub; ++k) {
            if (!__any_sync(kFull, hot[k])) {  // no tick of the block is above: no start, no run end
                before = -INFINITY;
                continue;
            }
            const float x[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
            const bool a[4] = {x[0] > thr, x[1] > thr, x[2] > thr, x[3] > thr};
            const uint32_t b3 = __ballot_sync(kFull, a[3]);
            const bool left = lane == 0 ? before > thr : ((b3 >> (lane - 1)) & 1u) != 0;
            before = (b3 >> 31) ? INFINITY : -INFINITY;
            const uint32_t m = (uint32_t)(a[0] && !left) | ((uint32_t)(a[1] && !a[0]) << 1) |
                               ((uint32_t)(a[2] && !a[1]) << 2) | ((uint32_t)(a[3] && !a[2]) << 3);
            if (!__any_sync(kFull, m != 0)) continue;
            // the index of this lane's first start: the starts of the lanes below
            const uint32_t s0 = __ballot_sync(kFull, m & 1u), s1 = __ballot_sync(kFull, m & 2u),
                           s2 = __ballot_sync(kFull, m & 4u), s3 = __ballot_sync(kFull, m & 8u);
            int32_t idx = next + __popc(s0 & lt) + __popc(s1 & lt) + __popc(s2 & lt) + __popc(s3 & lt);
            next += __popc(s0) + __popc(s1) + __popc(s2) + __popc(s3);
            const int tb = base + 128 * k + 4 * lane;
            // the lane's last start begins a run past its last tick iff that tick is above
            const bool lng = a[3] && m != 0;
            const int hi = 31 - __clz(m | 1u);
            const uint32_t loc = lng ? m & ~(1u << hi) : m;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if ((loc >> j) & 1u) {  // ends within the lane: measured here, in tick order
                    Run r{tb + j, tb + j, tb + j, x[j], x[j]};
                    bool on = true;
#pragma unroll
                    for (int j2 = j + 1; j2 < 4; ++j2) {
                        on = on && a[j2];
                        if (on) {
                            if (x[j2] > r.peak) {
                                r.peak = x[j2];
                                r.tick = tb + j2;
                            }
                            r.charge += x[j2];
                            r.end = tb + j2;
                        }
                    }
                    sink(idx++, r);
                }
            }
            uint32_t longs = __ballot_sync(kFull, lng);
            while (longs) {  // in lane order, so in tick order
                const int owner = __ffs(longs) - 1;
                longs &= longs - 1;
                const int ts = __shfl_sync(kFull, tb + hi, owner);
                const int32_t kl = __shfl_sync(kFull, idx, owner);
                const Run r = warp_walk(src, ts, nticks, thr, lane);
                if (lane == 0) sink(kl, r);
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

__global__ void __launch_bounds__(kHfWarps * 32) hf_find_kernel(const __grid_constant__ HfTable t, int64_t nunits,
                                                                int32_t *__restrict__ chunk_sum,
                                                                int32_t *__restrict__ counts,
                                                                Run *__restrict__ slots) {
    __shared__ float4 stash[kHfWarps][32 * kHfSub];
    pdl_trigger();  // the place kernel may set up while this one runs; it waits for it
    const int lane = threadIdx.x & 31;
    const int64_t u = (int64_t)blockIdx.x * kHfWarps + (threadIdx.x >> 5);
    if (u >= nunits) return;  // the whole warp leaves together
    const HfDesc &d = t.r[find_plane(t, u)];
    const Unit unit = unit_of(d, u);
    Run *my = slots + u * kRunSlots;
    const Src src{unit.row, unit.t1, reinterpret_cast<float *>(stash[threadIdx.x >> 5]), 0, 0};
    const int32_t n = scan_unit(unit, src, d.nticks, d.thr, lane, [&](int32_t k, const Run &run) {
        if (k < kRunSlots) my[k] = run;
    });
    if (lane == 0) {
        counts[u] = n;
        if (n) atomicAdd(chunk_sum + d.chunk0 + (u - d.unit0) / kHfChunk, n);
    }
}

// One CTA per chunk (blockIdx.x = the chunk's index in the group).
__global__ void __launch_bounds__(kHfChunk) hf_place_kernel(const __grid_constant__ HfTable t, int64_t nunits,
                                                             const int32_t *__restrict__ chunk_sum,
                                                             const int32_t *__restrict__ counts,
                                                             const Run *__restrict__ slots,
                                                             int32_t *__restrict__ total,
                                                             int32_t *__restrict__ sums_next, int64_t cap) {
    constexpr int kWarps = kHfChunk / 32;
    __shared__ int32_t cum[kHfChunk + 1];  // runs copied from the slots before each unit
    __shared__ int32_t out[kHfChunk];      // each unit's offset in its plane
    __shared__ uint64_t warp_tot[kWarps];
    __shared__ int32_t base_sh, nover_sh;
    __shared__ int32_t over[kHfChunk];     // units with more runs than slots
    __shared__ float4 stash[kWarps][32 * kHfSub];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (blockIdx.x == 0 && tid < t.n) {  // planes without units
        const int64_t end = tid + 1 < t.n ? t.r[tid + 1].unit0 : nunits;
        if (t.r[tid].unit0 == end) total[tid] = 0;
    }
    // the next launch's chunk sums start at zero (this call's find kernel uses the
    // other array, and the last reader of this one finished before it started)
    for (int64_t i = (int64_t)blockIdx.x * kHfChunk + tid; i < cap; i += (int64_t)gridDim.x * kHfChunk)
        sums_next[i] = 0;
    int r = 0;  // the chunk's plane: the last with chunk0 <= blockIdx.x
    while (r + 1 < t.n && t.r[r + 1].chunk0 <= (int64_t)blockIdx.x) ++r;
    pdl_wait();  // counts, chunk sums and run slots come from the find kernel
    const HfDesc &d = t.r[r];
    const int64_t pend = r + 1 < t.n ? t.r[r + 1].unit0 : nunits;
    const int64_t c = (int64_t)blockIdx.x - d.chunk0;
    const int64_t first = d.unit0 + c * kHfChunk;
    const int64_t u = first + tid;
    const int32_t n = u < pend ? counts[u] : 0;
    const int32_t m = n <= kRunSlots ? n : 0;  // runs copied from the slots
    if (tid == 0) nover_sh = 0;
    if (warp == 0) {  // the plane's chunks before this one
        int32_t acc = 0;
        for (int64_t k = lane; k < c; k += 32) acc += chunk_sum[d.chunk0 + k];
        acc = (int32_t)__reduce_add_sync(kFull, (uint32_t)acc);
        if (lane == 0) base_sh = acc;
    }
    // block scan of (n, m) packed in 64 bits: both sums stay below 2^31
    uint64_t incl = ((uint64_t)(uint32_t)n << 32) | (uint32_t)m;
    const uint64_t own = incl;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint64_t y = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    uint64_t excl = incl - own;
    for (int w = 0; w < warp; ++w) excl += warp_tot[w];
    const int32_t off = base_sh + (int32_t)(excl >> 32);
    out[tid] = off;
    cum[tid] = (int32_t)(uint32_t)excl;
    if (tid == kHfChunk - 1) cum[kHfChunk] = (int32_t)(uint32_t)(excl + own);
    if (n > kRunSlots) over[atomicAdd(&nover_sh, 1)] = tid;
    if (u == pend - 1) total[r] = off + n;
    __syncthreads();
    // the slots' runs, shared out evenly
    const int32_t nrun = cum[kHfChunk];
    for (int32_t i = tid; i < nrun; i += kHfChunk) {
        int lo = 0, hi = kHfChunk - 1;  // the unit j with cum[j] <= i < cum[j + 1]
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (cum[mid] <= i)
                lo = mid;
            else
                hi = mid - 1;
        }
        const int32_t k = i - cum[lo];
        const int64_t uj = first + lo;
        put_hit(d, unit_of(d, uj).wire, out[lo] + k, slots[uj * kRunSlots + k]);
    }
    // units with more runs than slots: a warp each, scanned again
    for (int q = warp; q < nover_sh; q += kWarps) {
        const int j = over[q];
        const Unit unit = unit_of(d, first + j);
        const int32_t oj = out[j];
        const Src src{unit.row, unit.t1, reinterpret_cast<float *>(stash[warp]), 0, 0};
        scan_unit(unit, src, d.nticks, d.thr, lane, [&](int32_t k, const Run &run) { put_hit(d, unit.wire, oj + k, run); });
    }
}

}  // namespace

int64_t find_hits_unit_cap(size_t scratch_bytes) {
    return (int64_t)(scratch_bytes / (sizeof(int32_t) + kRunSlots * sizeof(Run)));
}

int64_t find_hits_chunks(const HfTable &t, int64_t nunits) {
    int64_t nchunks = 0;
    for (int r = 0; r < t.n; ++r) {
        const int64_t nu = (r + 1 < t.n ? t.r[r + 1].unit0 : nunits) - t.r[r].unit0;
        nchunks += (nu + kHfChunk - 1) / kHfChunk;
    }
    return nchunks;
}

cudaError_t launch_find_hits(const HfTable &t_in, int64_t nunits, void *scratch, int32_t *sums_cur, int32_t *sums_next,
                             int64_t cap, int32_t *totals, cudaStream_t s) {
    if (nunits <= 0) return cudaMemsetAsync(totals, 0, sizeof(int32_t) * kMaxHfPlanes, s);
    HfTable t = t_in;
    int64_t nchunks = 0;
    for (int r = 0; r < t.n; ++r) {
        const int64_t nu = (r + 1 < t.n ? t.r[r + 1].unit0 : nunits) - t.r[r].unit0;
        t.r[r].chunk0 = nchunks;
        nchunks += (nu + kHfChunk - 1) / kHfChunk;
    }
    if (nchunks > cap) return cudaErrorInvalidValue;
    int32_t *counts = static_cast<int32_t *>(scratch);
    Run *slots = reinterpret_cast<Run *>(counts + nunits);
    const unsigned blocks = (unsigned)((nunits + kHfWarps - 1) / kHfWarps);
    hf_find_kernel<<<blocks, kHfWarps * 32, 0, s>>>(t, nunits, sums_cur, counts, slots);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int32_t *cc = counts;
    const Run *cs = slots;
    return launch_pdl(hf_place_kernel, dim3((unsigned)nchunks), dim3(kHfChunk), 0, s, t, nunits,
                      static_cast<const int32_t *>(sums_cur), cc, cs, totals, sums_next, cap);
}

}  // namespace emtk
