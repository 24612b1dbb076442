// Request batcher (include/emtk.h): the dynamic batching of the paper's
// inference server (Sec. 2.3; measured under many client processes in
// Sec. 3.2), inside one process.  Client threads submit requests and wait on
// tickets; one dispatcher thread forms batches of whole requests in
// submission order and runs each with emtk_infer_batch on one of the
// batcher's streams (round robin), each stream with its own workspace; one
// completion thread waits for the batches in launch order and releases
// their tickets.
//
// Host threads only: no kernel of its own.  At most kMaxInflight batches are
// launched and not yet complete; the dispatcher waits for a free one, so the
// queue, not the GPU's launch queue, absorbs a burst of requests.
#include <chrono>
#include <condition_variable>
#include <deque>
#include <mutex>
#include <new>
#include <thread>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include "emtk_internal.h"

namespace {

using Clock = std::chrono::steady_clock;

constexpr int kMaxStreams = 16;
constexpr int kMaxInflight = 32;      // batches launched and not yet complete
constexpr int kMaxBatchRequests = 4096;

struct Lane {
    emtk_ctx *ctx = nullptr;
    cudaStream_t stream = nullptr;
};

struct Queued {
    emtk_request req;
    uint64_t ticket;
    Clock::time_point t;
};

struct Inflight {
    cudaEvent_t ev;
    std::vector<uint64_t> tickets;
    emtk_status st;
    int slot;  // pinned status word of the batch
};

}  // namespace

struct emtk_batcher {
    int device = 0;
    int32_t max_hits = 0;
    std::chrono::microseconds max_delay{0};
    std::vector<Lane> lanes;
    std::vector<cudaEvent_t> free_events;
    int *h_status = nullptr;  // pinned, kMaxInflight words: the device status after each batch

    std::mutex mu;
    std::condition_variable cv_dispatch;  // new request, stop, or a batch slot freed
    std::condition_variable cv_complete;  // new in-flight batch, or the dispatcher finished
    std::condition_variable cv_done;      // tickets finished
    std::deque<Queued> queue;
    int64_t queued_hits = 0;
    std::deque<Inflight> inflight;
    std::unordered_set<uint64_t> outstanding;          // submitted, not yet complete
    std::unordered_map<uint64_t, emtk_status> done;    // complete, not yet waited for
    uint64_t next_ticket = 1;
    uint64_t seq = 0;
    bool stop = false;
    bool dispatch_done = false;
    bool stalled = false;  // test knob (emtk_debug_batcher_stall): the dispatcher launches nothing
    int64_t n_batches = 0, n_requests = 0, n_hits = 0;

    std::thread dispatcher, completer;
};

namespace {

void dispatch_loop(emtk_batcher *b) {
    cudaSetDevice(b->device);
    std::unique_lock<std::mutex> lk(b->mu);
    for (;;) {
        if (b->queue.empty()) {
            if (b->stop) break;
            b->cv_dispatch.wait(lk);
            continue;
        }
        if (b->stalled && !b->stop) {  // a stalled dispatcher, until released or destroyed
            b->cv_dispatch.wait(lk);
            continue;
        }
        const Clock::time_point deadline = b->queue.front().t + b->max_delay;
        if (!b->stop && b->queued_hits < b->max_hits && Clock::now() < deadline) {
            b->cv_dispatch.wait_until(lk, deadline);
            continue;
        }
        if ((int)b->inflight.size() >= kMaxInflight || b->free_events.empty()) {
            b->cv_dispatch.wait(lk);
            continue;
        }
        std::vector<emtk_request> reqs;
        std::vector<uint64_t> tickets;
        int64_t hits = 0;
        while (!b->queue.empty() && (int)reqs.size() < kMaxBatchRequests) {
            const Queued &q = b->queue.front();
            if (!reqs.empty() && hits + q.req.nhits > b->max_hits) break;
            reqs.push_back(q.req);
            tickets.push_back(q.ticket);
            hits += q.req.nhits;
            b->queued_hits -= q.req.nhits;
            b->queue.pop_front();
        }
        const uint64_t seq = b->seq++;
        Lane &lane = b->lanes[seq % b->lanes.size()];
        const int slot = (int)(seq % kMaxInflight);
        cudaEvent_t ev = b->free_events.back();
        b->free_events.pop_back();
        lk.unlock();

        emtk_status st = emtk_infer_batch(lane.ctx, reqs.data(), (int32_t)reqs.size(),
                                          reinterpret_cast<emtk_stream>(lane.stream));
        if (st == EMTK_OK) {
            // the lane's device status word after this batch, then cleared for the next
            cudaError_t e = cudaMemcpyAsync(b->h_status + slot, lane.ctx->ws.status, sizeof(int),
                                            cudaMemcpyDeviceToHost, lane.stream);
            if (e == cudaSuccess) e = cudaMemsetAsync(lane.ctx->ws.status, 0, sizeof(int), lane.stream);
            if (e != cudaSuccess) st = EMTK_ERR_CUDA;
        }
        if (cudaEventRecord(ev, lane.stream) != cudaSuccess && st == EMTK_OK) st = EMTK_ERR_CUDA;

        lk.lock();
        b->inflight.push_back(Inflight{ev, std::move(tickets), st, slot});
        b->n_batches++;
        b->n_requests += (int64_t)reqs.size();
        b->n_hits += hits;
        b->cv_complete.notify_one();
    }
    b->dispatch_done = true;
    b->cv_complete.notify_all();
}

void complete_loop(emtk_batcher *b) {
    cudaSetDevice(b->device);
    std::unique_lock<std::mutex> lk(b->mu);
    for (;;) {
        while (b->inflight.empty() && !b->dispatch_done) b->cv_complete.wait(lk);
        if (b->inflight.empty()) break;
        Inflight &f = b->inflight.front();
        const cudaEvent_t ev = f.ev;
        lk.unlock();
        const cudaError_t e = cudaEventSynchronize(ev);
        lk.lock();
        emtk_status st = f.st;
        if (st == EMTK_OK) {
            if (e != cudaSuccess)
                st = EMTK_ERR_CUDA;
            else if (b->h_status[f.slot] & 1)
                st = EMTK_ERR_TIMEOUT;
        }
        for (uint64_t t : f.tickets) {
            b->outstanding.erase(t);
            b->done[t] = st;
        }
        b->free_events.push_back(ev);
        b->inflight.pop_front();
        b->cv_done.notify_all();
        b->cv_dispatch.notify_one();
    }
}

void free_batcher(emtk_batcher *b) {
    for (cudaEvent_t ev : b->free_events) cudaEventDestroy(ev);
    for (Lane &l : b->lanes) {
        if (l.stream) {
            cudaStreamSynchronize(l.stream);
            cudaStreamDestroy(l.stream);
        }
        emtk::destroy_lane_ctx(l.ctx);
    }
    emtk::host_free(b->h_status);
    delete b;
}

}  // namespace

extern "C" {

emtk_status emtk_batcher_create(emtk_ctx *ctx, int32_t nstreams, int32_t max_hits, int64_t max_delay_us,
                                emtk_batcher **out) {
    if (out) *out = nullptr;
    if (!ctx || !out || nstreams < 1 || nstreams > kMaxStreams || max_hits < 1 || max_delay_us < 0)
        return EMTK_ERR_ARG;
    emtk_batcher *b = new (std::nothrow) emtk_batcher;
    if (!b) return EMTK_ERR_OOM;
    b->device = ctx->device;
    b->max_hits = max_hits;
    b->max_delay = std::chrono::microseconds(max_delay_us);
    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    emtk_status st = cudaSetDevice(b->device) == cudaSuccess ? EMTK_OK : EMTK_ERR_CUDA;
    if (st == EMTK_OK) {
        void *h = nullptr;
        if (emtk::host_alloc(&h, kMaxInflight * sizeof(int)) != cudaSuccess)
            st = EMTK_ERR_OOM;
        else
            b->h_status = static_cast<int *>(h);
    }
    for (int i = 0; st == EMTK_OK && i < kMaxInflight; ++i) {
        cudaEvent_t ev;
        if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess)
            st = EMTK_ERR_CUDA;
        else
            b->free_events.push_back(ev);
    }
    for (int i = 0; st == EMTK_OK && i < nstreams; ++i) {
        Lane l;
        l.ctx = emtk::make_lane_ctx(ctx, &st);
        if (st == EMTK_OK && cudaStreamCreateWithFlags(&l.stream, cudaStreamNonBlocking) != cudaSuccess)
            st = EMTK_ERR_CUDA;
        b->lanes.push_back(l);
    }
    if (prev >= 0) cudaSetDevice(prev);
    if (st != EMTK_OK) {
        free_batcher(b);
        return st;
    }
    try {
        b->dispatcher = std::thread(dispatch_loop, b);
        b->completer = std::thread(complete_loop, b);
    } catch (...) {
        if (b->dispatcher.joinable()) {
            {
                std::lock_guard<std::mutex> lk(b->mu);
                b->stop = true;
                b->dispatch_done = true;
            }
            b->cv_dispatch.notify_all();
            b->dispatcher.join();
        }
        free_batcher(b);
        return EMTK_ERR_OOM;
    }
    *out = b;
    return EMTK_OK;
}

emtk_status emtk_batcher_submit(emtk_batcher *b, const emtk_request *req, uint64_t *ticket) {
    if (ticket) *ticket = 0;
    if (!b || !req || !ticket) return EMTK_ERR_ARG;
    const emtk_status st = emtk::validate_request(*req);
    if (st != EMTK_OK) return st;
    {
        std::lock_guard<std::mutex> lk(b->mu);
        if (b->stop) return EMTK_ERR_ARG;
        *ticket = b->next_ticket++;
        b->queue.push_back(Queued{*req, *ticket, Clock::now()});
        b->queued_hits += req->nhits;
        b->outstanding.insert(*ticket);
    }
    b->cv_dispatch.notify_one();
    return EMTK_OK;
}

emtk_status emtk_batcher_wait(emtk_batcher *b, uint64_t ticket, int64_t timeout_ms) {
    if (!b) return EMTK_ERR_ARG;
    std::unique_lock<std::mutex> lk(b->mu);
    if (!b->outstanding.count(ticket) && !b->done.count(ticket)) return EMTK_ERR_ARG;
    auto ready = [&] { return b->done.count(ticket) != 0; };
    if (timeout_ms < 0)
        b->cv_done.wait(lk, ready);
    else if (!b->cv_done.wait_for(lk, std::chrono::milliseconds(timeout_ms), ready))
        return EMTK_ERR_TIMEOUT;
    const emtk_status st = b->done[ticket];
    b->done.erase(ticket);
    return st;
}

emtk_status emtk_batcher_stats(emtk_batcher *b, int64_t *batches, int64_t *requests, int64_t *hits) {
    if (!b) return EMTK_ERR_ARG;
    std::lock_guard<std::mutex> lk(b->mu);
    if (batches) *batches = b->n_batches;
    if (requests) *requests = b->n_requests;
    if (hits) *hits = b->n_hits;
    return EMTK_OK;
}

emtk_status emtk_debug_batcher_stall(emtk_batcher *b, int32_t stall) {
    if (!b || (stall != 0 && stall != 1)) return EMTK_ERR_ARG;
    {
        std::lock_guard<std::mutex> lk(b->mu);
        b->stalled = stall != 0;
    }
    b->cv_dispatch.notify_all();
    return EMTK_OK;
}

emtk_status emtk_batcher_destroy(emtk_batcher *b) {
    if (!b) return EMTK_OK;
    {
        std::lock_guard<std::mutex> lk(b->mu);
        b->stop = true;
    }
    b->cv_dispatch.notify_all();
    if (b->dispatcher.joinable()) b->dispatcher.join();
    if (b->completer.joinable()) b->completer.join();
    free_batcher(b);
    return EMTK_OK;
}

}  // extern "C"
