// Stream-ordered page dependencies of a store.
//
// The store's pages are its only shared resource, so its calls are ordered
// by their data dependencies instead of by the order they were made in:
//   - a get (and a compaction, for the pages it moves out) waits for the
//     call that last wrote each page it reads (read after write);
//   - a put (and a compaction, for the pages it moves into) waits for the
//     calls that last wrote or read each page it reuses (write after read,
//     write after write: pages of freed or evicted objects).
// Waiting happens on the GPU (cudaStreamWaitEvent) and only across streams:
// work on one stream is already ordered. Per-call events are recorded only
// once a second stream has used the store, so that single-stream use keeps
// consecutive launches adjacent (programmatic dependent launch). Calls made
// before that have no event of their own; a dependency on one of them waits
// for everything its stream has been given so far.
//
// Streams given to a store must stay valid until the store is destroyed.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

namespace t2i {

class StreamDeps {
  public:
    struct Dep {
        uint32_t seq = 0;        // 0 = none; else the call's number on its stream
        uint16_t stream = 0;
    };
    struct PageDeps {
        Dep writer;
        Dep readers[2];
        uint8_t more_readers = 0;  // > 2 reading streams since the last write
    };
    static constexpr uint32_t kRing = 64;
    // a reader whose reads are not calls of the store (a view): later
    // writers wait for everything its stream has been given by then
    static constexpr uint32_t kOpen = 0xFFFFFFFFu;

    ~StreamDeps() { release(); }

    void resize_pages(uint64_t n) { pages_.assign(n, PageDeps{}); }

    // Index of `s`, registering it (and its events) on first use. -1 if the
    // events cannot be created.
    int stream_index(cudaStream_t s) {
        for (size_t i = 0; i < streams_.size(); ++i)
            if (streams_[i].s == s) return static_cast<int>(i);
        if (streams_.size() >= 0xFFFF) return -1;
        State st;
        st.s = s;
        if (cudaEventCreateWithFlags(&st.lazy, cudaEventDisableTiming) != cudaSuccess) return -1;
        for (uint32_t k = 0; k < kRing; ++k) {
            if (cudaEventCreateWithFlags(&st.ring[k], cudaEventDisableTiming) != cudaSuccess) {
                for (uint32_t j = 0; j < k; ++j) cudaEventDestroy(st.ring[j]);
                cudaEventDestroy(st.lazy);
                return -1;
            }
            st.ring_seq[k] = 0;
        }
        streams_.push_back(st);
        return static_cast<int>(streams_.size() - 1);
    }

    // --- one call on stream index `si`
    void begin(int si) {
        cur_ = si;
        need_.assign(streams_.size(), 0);
        wait_all_ = false;
    }
    void reads(uint32_t page) { note(pages_[page].writer); }
    void writes(uint32_t page) {
        const PageDeps& d = pages_[page];
        note(d.writer);
        note(d.readers[0]);
        note(d.readers[1]);
        if (d.more_readers) wait_all_ = true;
    }
    // Makes the call's stream wait for what it depends on.
    cudaError_t wait() {
        cudaStream_t s = streams_[cur_].s;
        for (size_t j = 0; j < streams_.size(); ++j) {
            const uint32_t q = wait_all_ ? streams_[j].seq : need_[j];
            if (int(j) == cur_ || q == 0) continue;
            cudaError_t e = wait_for(static_cast<int>(j), q, s);
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    }
    // After the call's work is enqueued: its number (and event, once more than
    // one stream has used the store).
    cudaError_t end(uint32_t* seq_out) {
        State& st = streams_[cur_];
        const uint32_t q = ++st.seq;
        *seq_out = q;
        if (streams_.size() > 1) {
            const uint32_t k = q % kRing;
            cudaError_t e = cudaEventRecord(st.ring[k], st.s);
            if (e != cudaSuccess) return e;
            st.ring_seq[k] = q;
        }
        return cudaSuccess;
    }
    void mark_write(uint32_t page, uint32_t seq) {
        PageDeps& d = pages_[page];
        d.writer = {seq, static_cast<uint16_t>(cur_)};
        d.readers[0] = d.readers[1] = Dep{};
        d.more_readers = 0;
    }
    void mark_read(uint32_t page, uint32_t seq) {
        PageDeps& d = pages_[page];
        const Dep me{seq, static_cast<uint16_t>(cur_)};
        for (Dep& r : d.readers) {
            if (r.seq == 0 || r.stream == me.stream) {
                r = me;
                return;
            }
        }
        d.more_readers = 1;
    }

    // Waits on the host for everything every known stream has been given.
    void synchronize_all() {
        for (State& st : streams_) {
            if (st.seq == 0) continue;
            if (cudaEventRecord(st.lazy, st.s) == cudaSuccess) cudaEventSynchronize(st.lazy);
        }
    }

    void release() {
        for (State& st : streams_) {
            cudaEventDestroy(st.lazy);
            for (uint32_t k = 0; k < kRing; ++k) cudaEventDestroy(st.ring[k]);
        }
        streams_.clear();
    }

    size_t n_streams() const { return streams_.size(); }

  private:
    struct State {
        cudaStream_t s = nullptr;
        uint32_t seq = 0;           // calls enqueued on this stream
        cudaEvent_t ring[kRing];    // call q's event lives in ring[q % kRing]
        uint32_t ring_seq[kRing];   // the call each ring event was last recorded for
        cudaEvent_t lazy = nullptr; // "everything so far" on this stream
        uint32_t lazy_seq = 0;
    };

    void note(const Dep& d) {
        if (d.seq == 0 || d.stream == cur_) return;
        if (need_[d.stream] < d.seq) need_[d.stream] = d.seq;
    }

    // Stream `s` waits until call q of stream j has run: on q's own event if
    // it has one (or on a later call's, which is later on the same stream),
    // else on an event recorded now after everything stream j was given.
    cudaError_t wait_for(int j, uint32_t q, cudaStream_t s) {
        State& st = streams_[j];
        const uint32_t k = q % kRing;
        if (st.ring_seq[k] >= q) return cudaStreamWaitEvent(s, st.ring[k], 0);
        if (st.lazy_seq < q) {
            cudaError_t e = cudaEventRecord(st.lazy, st.s);
            if (e != cudaSuccess) return e;
            st.lazy_seq = st.seq;
        }
        return cudaStreamWaitEvent(s, st.lazy, 0);
    }

    std::vector<State> streams_;
    std::vector<PageDeps> pages_;
    std::vector<uint32_t> need_;
    int cur_ = 0;
    bool wait_all_ = false;
};

}  // namespace t2i
