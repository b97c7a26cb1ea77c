// The store: host control core + pointer checks + kernel launches, and the
// t2i_store / t2i_put_batch / t2i_get_batch / t2i_free / t2i_compact C ABI.
#include <cuda.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "common.hpp"
#include "control.hpp"
#include "deps.hpp"
#include "kernels.cuh"

namespace t2i {
namespace {

// ------------------------------------------------------------------ driver
// Pointer attributes come from the driver API, fetched through the runtime
// so that the library does not link libcuda (it loads on machines without
// a driver, where only the t2i_ctl_* calls are usable).
using PFN_getAttrs = CUresult (*)(unsigned int, CUpointer_attribute*, void**, CUdeviceptr);

PFN_getAttrs driver_get_attrs() {
    static PFN_getAttrs fn = []() -> PFN_getAttrs {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuPointerGetAttributes", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<PFN_getAttrs>(p);
    }();
    return fn;
}

enum class MemKind { Unknown, Device, Host, Managed };

struct Range {
    uint64_t start = 0, end = 0;  // [start, end)
    MemKind kind = MemKind::Unknown;
    int device = -1;
    uint64_t dev_base = 0;  // device-visible address of `start` (host memory)
};

// Queries the allocation that holds p. false if the driver call failed.
bool query_range(const void* p, Range* r) {
    PFN_getAttrs fn = driver_get_attrs();
    if (!fn) return false;
    CUpointer_attribute attrs[6] = {CU_POINTER_ATTRIBUTE_MEMORY_TYPE,     CU_POINTER_ATTRIBUTE_DEVICE_ORDINAL,
                                    CU_POINTER_ATTRIBUTE_RANGE_START_ADDR, CU_POINTER_ATTRIBUTE_RANGE_SIZE,
                                    CU_POINTER_ATTRIBUTE_IS_MANAGED,       CU_POINTER_ATTRIBUTE_DEVICE_POINTER};
    unsigned int mtype = 0;
    int ordinal = -1;
    CUdeviceptr start = 0;
    size_t size = 0;
    int managed = 0;
    CUdeviceptr devptr = 0;
    void* data[6] = {&mtype, &ordinal, &start, &size, &managed, &devptr};
    if (fn(6, attrs, data, reinterpret_cast<CUdeviceptr>(p)) != CUDA_SUCCESS) return false;
    r->start = start;
    r->end = start + size;
    r->device = ordinal;
    if (managed)
        r->kind = MemKind::Managed;
    else if (mtype == CU_MEMORYTYPE_DEVICE)
        r->kind = MemKind::Device;
    else if (mtype == CU_MEMORYTYPE_HOST)
        r->kind = MemKind::Host;
    else
        r->kind = MemKind::Unknown;
    // device-visible address of the range start (same as the host address
    // under unified addressing)
    r->dev_base = devptr ? uint64_t(devptr) - (reinterpret_cast<uint64_t>(p) - start) : start;
    if (r->kind == MemKind::Unknown) r->start = r->end = 0;
    return true;
}

struct DeviceGuard {
    int prev = -1;
    bool switched = false;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) switched = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        if (switched) cudaSetDevice(prev);
    }
};

// One NVTX range per library call, named after it (profilers show the host
// control around the launches; without a tool attached it costs a branch).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

int log2_exact(uint64_t v) {
    int s = 0;
    while ((uint64_t(1) << s) < v) ++s;
    return (uint64_t(1) << s) == v ? s : -1;
}

}  // namespace

// -------------------------------------------------------------------- Store
class Store {
  public:
    Store(void* pool, const t2i_store_config& cfg, int device)
        : pool_(reinterpret_cast<uint64_t>(pool)), cfg_(cfg), device_(device),
          ctl_(cfg.pool_bytes / cfg.page_bytes, cfg.page_bytes, cfg.alloc_policy) {
        handle_.core = &ctl_;
        handle_.owned = false;
        handle_.mu = &mu;
        page_shift_ = log2_exact(cfg.page_bytes);
    }
    ~Store() {
        DeviceGuard g(device_);
        deps_.synchronize_all();
        deps_.release();
        if (work_) cudaFree(work_);
    }

    t2i_status init(std::string* err) {
        DeviceGuard g(device_);
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device_) != cudaSuccess || sms <= 0) {
            *err = "cannot query the device";
            return T2I_ERR_CUDA;
        }
        // resident CTAs on the device (SMs x CTAs per SM), per kernel
        const void* fns[4][2] = {
            {reinterpret_cast<const void*>(scatter_put_kernel<kBlobLarge, false>),
             reinterpret_cast<const void*>(scatter_put_kernel<kBlobLarge, true>)},
            {reinterpret_cast<const void*>(gather_get_kernel<kBlobLarge, false>),
             reinterpret_cast<const void*>(gather_get_kernel<kBlobLarge, true>)},
            {reinterpret_cast<const void*>(compact_move_kernel<kBlobLarge>),
             reinterpret_cast<const void*>(compact_move_kernel<kBlobLarge>)},
            {reinterpret_cast<const void*>(gather_copy_kernel<kBlobLarge, false>),
             reinterpret_cast<const void*>(gather_copy_kernel<kBlobLarge, true>)}};
        for (int m = 0; m < 4; ++m)
            for (int a = 0; a < 2; ++a) {
                int occ = 0;
                cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fns[m][a], kThreads, 0);
                max_ctas_[m][a] = sms * (occ > 0 ? occ : 1);
            }
        // one chunk counter per stream (the first kWorkStreams streams of
        // the store; later ones use equal static shares), zeroed once
        if (cudaMalloc(&work_, kWorkStreams * sizeof(WorkCounter)) != cudaSuccess) {
            work_ = nullptr;
            *err = "cannot allocate the work counters";
            return T2I_ERR_CUDA;
        }
        // cleared on a private non-blocking stream: waits for nothing else
        cudaStream_t zs = nullptr;
        bool zeroed = cudaStreamCreateWithFlags(&zs, cudaStreamNonBlocking) == cudaSuccess &&
                      cudaMemsetAsync(work_, 0, kWorkStreams * sizeof(WorkCounter), zs) == cudaSuccess &&
                      cudaStreamSynchronize(zs) == cudaSuccess;
        if (zs) cudaStreamDestroy(zs);
        if (!zeroed) {
            *err = "cannot clear the work counters";
            return T2I_ERR_CUDA;
        }
        deps_.resize_pages(ctl_.total_pages());
        return T2I_OK;
    }

    std::mutex mu;
    t2i_ctl* ctl_handle() { return &handle_; }
    Control& ctl() { return ctl_; }
    const std::string& error() const { return err_; }
    void set_error(std::string e) { err_ = std::move(e); }
    void inject_launch_failure(uint32_t countdown) { fail_countdown_ = countdown; }

    t2i_status put(const t2i_put_desc* descs, uint32_t n, t2i_id* ids, cudaStream_t stream);
    t2i_status get(const t2i_get_desc* descs, uint32_t n, t2i_status* per_item, cudaStream_t stream,
                   cudaEvent_t wait_event = nullptr);
    t2i_status free(const t2i_id* ids, uint32_t n) {
        t2i_status st = ctl_.free(ids, n);
        if (st != T2I_OK) err_ = ctl_.error();
        return st;
    }
    t2i_status compact(uint64_t limit_bytes, cudaStream_t stream, uint64_t* moved);
    t2i_status view(t2i_id id, cudaStream_t stream, void** ptr, uint64_t* nbytes);
    t2i_status pull_from(Store& src, const t2i_id* ids, uint32_t n, uint32_t consumers, t2i_id* out_ids,
                         t2i_status* per_item, cudaStream_t stream);
    t2i_status pull_pages(const void* src_pool, uint64_t src_pool_bytes, const t2i_paged_object* objs, uint32_t n,
                          uint32_t consumers, t2i_id* out_ids, cudaStream_t stream);

  private:
    // ---- pointer checks (per call cache of the last allocation seen)
    t2i_status check_user(const void* p, uint64_t n, bool want_write, bool is_host_flag, uint64_t* dev_addr,
                          bool* needs_copy_engine, Range* cache);
    bool overlaps_pool(uint64_t a, uint64_t n) const {
        const uint64_t pend = pool_ + cfg_.pool_bytes;
        return n && a < pend && pool_ < a + n;
    }

    // ---- launch building
    struct Seg {
        uint64_t user;
        uint64_t nbytes_flags;
        const uint32_t* pages;
        uint32_t n_pages;
    };
    template <Mode M>
    t2i_status launch_segments(const std::vector<Seg>& segs, cudaStream_t stream);
    template <Mode M, bool GENERAL>
    t2i_status launch_group(const std::vector<Seg>& segs, cudaStream_t stream);
    template <Mode M, bool GENERAL, int BLOB>
    t2i_status launch_one(const std::vector<SegDesc>& sd, const std::vector<uint32_t>& pages, uint32_t n_granules,
                          cudaStream_t stream);
    // the call's stream in the dependency tracker (creating its events), and
    // the work counter its launches use
    t2i_status stream_slot(cudaStream_t s, int* si) {
        *si = deps_.stream_index(s);
        if (*si < 0) {
            err_ = "cannot create the events for a new stream";
            return T2I_ERR_CUDA;
        }
        cur_work_ = *si < int(kWorkStreams) ? reinterpret_cast<uint64_t>(work_) + uint64_t(*si) * sizeof(WorkCounter)
                                             : 0;
        return T2I_OK;
    }
    t2i_status cuda_fail(const char* what, cudaError_t e) {
        err_ = std::string(what) + ": " + cudaGetErrorString(e);
        return T2I_ERR_CUDA;
    }

    uint64_t pool_;
    t2i_store_config cfg_;
    int device_;
    Control ctl_;
    t2i_ctl handle_{};
    uint32_t page_shift_ = 0;
    int max_ctas_[4][2] = {{1, 1}, {1, 1}, {1, 1}, {1, 1}};  // [mode][any alignment]: resident CTAs on the device
    uint32_t fail_countdown_ = 0;  // > 0: that many launches from now, report a failure (testing)
    // Work counters, one per stream index: launches on one stream run one
    // after another (each waits for the previous grid before touching its
    // counter), launches on different streams use different counters.
    static constexpr uint32_t kWorkStreams = 64;
    WorkCounter* work_ = nullptr;
    uint64_t cur_work_ = 0;  // the current call's counter (0: static shares)
    // LaunchHeader::flags of the current call's launches with static
    // shares: kPrefetchSources unless a put reads host or managed memory
    uint32_t launch_flags_ = kPrefetchSources;
    std::vector<Seg> aligned_, general_;
    StreamDeps deps_;
    std::string err_;
    std::vector<const Object*> objs_;
    std::vector<Seg> segs_;
    std::vector<t2i_move> batch_;  // the moves of one compaction launch
    // moves per compaction launch: one 24-byte descriptor and one page each
    static constexpr size_t kMovesPerLaunch = 1024;
#ifndef T2I_TUNE_COMPACT_FIRST
#define T2I_TUNE_COMPACT_FIRST 64
#endif
    static constexpr size_t kCompactFirstBatch = T2I_TUNE_COMPACT_FIRST;  // moves in the first launch
    static_assert(kMovesPerLaunch * (sizeof(SegDesc) + sizeof(uint32_t)) <= size_t(kBlobLarge), "moves per launch");
    std::vector<SegDesc> sd_;
    std::vector<uint32_t> lp_;
    alignas(16) unsigned char param_buf_[sizeof(LaunchParams<kBlobLarge>)];
};

t2i_status Store::check_user(const void* p, uint64_t n, bool want_write, bool is_host_flag, uint64_t* dev_addr,
                             bool* needs_copy_engine, Range* cache) {
    const uint64_t a = reinterpret_cast<uint64_t>(p);
    *needs_copy_engine = false;
    *dev_addr = a;
    if (n == 0) return T2I_OK;
    if (!p) {
        err_ = "null buffer";
        return T2I_ERR_INVALID;
    }
    if (a + n < a) {
        err_ = "buffer range wraps around";
        return T2I_ERR_INVALID;
    }
    if (overlaps_pool(a, n)) {
        err_ = "a user buffer overlaps the store's pool";
        return T2I_ERR_INVALID;
    }
    if (!cfg_.check_pointers) {
        *needs_copy_engine = is_host_flag && cfg_.h2d_mode == 1;
        return T2I_OK;
    }
    if (!(cache->kind != MemKind::Unknown && a >= cache->start && a + n <= cache->end)) {
        if (!query_range(p, cache)) {
            err_ = "the CUDA driver cannot describe a buffer pointer";
            return T2I_ERR_INVALID;
        }
    }
    const Range& r = *cache;
    switch (r.kind) {
        case MemKind::Device:
            if (is_host_flag) {
                err_ = "src_is_host = 1 but the buffer is device memory";
                return T2I_ERR_INVALID;
            }
            if (r.device != device_) {
                err_ = "a buffer lives on another device";
                return T2I_ERR_INVALID;
            }
            break;
        case MemKind::Managed:
            break;
        case MemKind::Host:
            if (!is_host_flag && !want_write) {
                err_ = "host memory passed as a device source (set src_is_host)";
                return T2I_ERR_INVALID;
            }
            *dev_addr = r.dev_base + (a - r.start);
            *needs_copy_engine = want_write ? cfg_.d2h_mode == 1 : cfg_.h2d_mode == 1;
            break;
        case MemKind::Unknown:
            // pageable host memory: only a host source, through the copy engine
            if (is_host_flag && !want_write) {
                *needs_copy_engine = true;
                return T2I_OK;
            }
            err_ = want_write ? "a get destination must be device memory or pinned host memory"
                              : "unknown source pointer (not device memory; set src_is_host for host memory)";
            return T2I_ERR_INVALID;
    }
    if (a + n > r.end) {
        err_ = "a buffer range runs past the end of its allocation";
        return T2I_ERR_INVALID;
    }
    return T2I_OK;
}

#include "launch.cuh"

t2i_status Store::put(const t2i_put_desc* descs, uint32_t n, t2i_id* ids, cudaStream_t stream) {
    if (n == 0) return T2I_OK;
    if (!descs || !ids) {
        err_ = "put: null descriptor or id array";
        return T2I_ERR_INVALID;
    }
    // 1. check every source before touching the directory
    std::vector<uint64_t> dev_src(n);
    std::vector<uint8_t> use_ce(n);
    Range cache;
    bool device_sources = true;  // every source the kernel reads is device memory
    for (uint32_t i = 0; i < n; ++i) {
        const t2i_put_desc& d = descs[i];
        if (d.src_is_host > 1 || d.evictable > 1) {
            err_ = "put: src_is_host and evictable must be 0 or 1";
            return T2I_ERR_INVALID;
        }
        bool ce = false;
        if (d.src) {
            t2i_status st = check_user(d.src, d.nbytes, false, d.src_is_host != 0, &dev_src[i], &ce, &cache);
            if (st != T2I_OK) {
                err_ = "put: item " + std::to_string(i) + ": " + err_;
                return st;
            }
            // (without pointer checks the kind of memory is unknown: no prefetch)
            if (!ce && d.nbytes)
                device_sources = device_sources && !d.src_is_host && cfg_.check_pointers &&
                                 cache.kind == MemKind::Device;
        }
        use_ce[i] = ce;
    }
    // 2. plan and commit pages (evicting if needed)
    t2i_status st = ctl_.put(descs, n, ids, &objs_);
    if (st != T2I_OK) {
        err_ = ctl_.error();
        return st;
    }
    // 3. copies, after the earlier users of the pages they overwrite
    DeviceGuard g(device_);
    int si = 0;
    if ((st = stream_slot(stream, &si)) != T2I_OK) {
        ctl_.rollback_put(ids, n);
        return st;
    }
    deps_.begin(si);
    bool any = false;
    for (uint32_t i = 0; i < n; ++i) {
        if (!descs[i].src) continue;  // reserved: nothing is written
        for (uint32_t pg : objs_[i]->pages) deps_.writes(pg);
        any = any || !objs_[i]->pages.empty();
    }
    if (!any) return T2I_OK;
    cudaError_t we = deps_.wait();
    if (we != cudaSuccess) {
        ctl_.rollback_put(ids, n);
        return cuda_fail("put: cannot order after earlier calls", we);
    }
    // The call's number goes on every page it writes once its copies are
    // enqueued, and also when it fails part-way: copies enqueued before the
    // failure may still be writing the pages it hands back.
    auto mark_writes = [&]() {
        uint32_t q = 0;
        cudaError_t ee = deps_.end(&q);
        for (uint32_t i = 0; i < n; ++i)
            if (descs[i].src)
                for (uint32_t pg : objs_[i]->pages) deps_.mark_write(pg, q);
        return ee;
    };
    segs_.clear();
    const uint64_t P = uint64_t(1) << page_shift_;
    for (uint32_t i = 0; i < n; ++i) {
        const Object* o = objs_[i];
        if (!descs[i].src || o->nbytes == 0) continue;
        if (use_ce[i]) {
            // one copy per run of consecutive pages
            const char* src = static_cast<const char*>(descs[i].src);
            size_t j = 0;
            while (j < o->pages.size()) {
                size_t k = j + 1;
                while (k < o->pages.size() && o->pages[k] == o->pages[k - 1] + 1) ++k;
                const uint64_t off = j * P;
                const uint64_t bytes = std::min<uint64_t>(o->nbytes - off, (k - j) * P);
                cudaError_t e = cudaMemcpyAsync(reinterpret_cast<void*>(pool_ + uint64_t(o->pages[j]) * P), src + off,
                                                bytes, cudaMemcpyHostToDevice, stream);
                if (e != cudaSuccess) {
                    err_ = std::string("put: host copy failed: ") + cudaGetErrorString(e);
                    mark_writes();
                    ctl_.rollback_put(ids, n);
                    return T2I_ERR_CUDA;
                }
                ctl_.counters().h2d_copies++;
                j = k;
            }
        } else {
            segs_.push_back({dev_src[i], o->nbytes, o->pages.data(), uint32_t(o->pages.size())});
        }
    }
    if (!segs_.empty()) {
        launch_flags_ = device_sources ? kPrefetchSources : 0;
        st = launch_segments<Mode::Put>(segs_, stream);
        launch_flags_ = kPrefetchSources;
        if (st != T2I_OK) {
            mark_writes();
            ctl_.rollback_put(ids, n);
            return st;
        }
    }
    cudaError_t ee = mark_writes();
    if (ee != cudaSuccess) return cuda_fail("put: cannot record its event", ee);
    return T2I_OK;
}

t2i_status Store::get(const t2i_get_desc* descs, uint32_t n, t2i_status* per_item, cudaStream_t stream,
                      cudaEvent_t wait_event) {
    if (n == 0) return T2I_OK;
    if (!descs) {
        err_ = "get: null descriptor array";
        return T2I_ERR_INVALID;
    }
    // 1. directory (ids, evictions, cast rules) without touching the LRU
    std::vector<t2i_status> per(n, T2I_OK);
    std::vector<uint64_t> dev_dst(n, 0);
    std::vector<uint8_t> use_ce(n, 0);
    t2i_status first = T2I_OK;
    uint32_t first_i = 0;
    Range cache;
    for (uint32_t i = 0; i < n; ++i) {
        const t2i_get_desc& d = descs[i];
        t2i_status s = T2I_OK;
        const Object* o = ctl_.find(d.id);
        if (d.cast > 1 || d.reserved != 0) {
            s = T2I_ERR_INVALID;
        } else if (!o) {
            s = ctl_.is_evicted(d.id) ? T2I_ERR_EVICTED : T2I_ERR_NOT_FOUND;
        } else {
            const uint64_t out_bytes = d.cast ? o->nbytes / 2 : o->nbytes;
            if ((d.cast && (o->nbytes % 4 != 0 || (reinterpret_cast<uint64_t>(d.dst) & 1))) ||
                d.dst_bytes < out_bytes) {
                s = T2I_ERR_INVALID;
            } else {
                bool ce = false;
                if (check_user(d.dst, out_bytes, true, false, &dev_dst[i], &ce, &cache) != T2I_OK) s = T2I_ERR_INVALID;
                use_ce[i] = ce && !d.cast;  // the cast runs in the kernel
            }
        }
        per[i] = s;
        if (s != T2I_OK && first == T2I_OK) {
            first = s;
            first_i = i;
        }
    }
    if (first != T2I_OK) {
        // nothing is written and the LRU is not touched; misses still count
        std::string why = err_;
        for (t2i_status s : per) ctl_.counters().misses += s == T2I_ERR_EVICTED;
        if (per_item) std::copy(per.begin(), per.end(), per_item);
        static const char* what[] = {"ok", "invalid", "no space", "id not found", "id was evicted", "cuda"};
        err_ = "get: item " + std::to_string(first_i) + ": " + what[first] +
               (first == T2I_ERR_INVALID && !why.empty() ? " (" + why + ")" : "");
        return first;
    }
    // 2. one gather launch for the batch (copies and casts together), after
    //    the calls that wrote its pages and after the caller's event
    objs_.resize(n);
    for (uint32_t i = 0; i < n; ++i) objs_[i] = ctl_.find(descs[i].id);
    DeviceGuard g(device_);
    int si = 0;
    t2i_status st = stream_slot(stream, &si);
    if (st != T2I_OK) return st;
    if (wait_event) {
        cudaError_t e = cudaStreamWaitEvent(stream, wait_event, 0);
        if (e != cudaSuccess) return cuda_fail("get: cannot wait for the event", e);
    }
    segs_.clear();
    deps_.begin(si);
    bool any = false;
    for (uint32_t i = 0; i < n; ++i) {
        const Object* o = objs_[i];
        if (o->nbytes == 0) continue;
        for (uint32_t pg : o->pages) deps_.reads(pg);
        any = true;
        if (use_ce[i]) continue;
        segs_.push_back({dev_dst[i], o->nbytes | (descs[i].cast ? kCastFlag : 0), o->pages.data(),
                         uint32_t(o->pages.size())});
    }
    if (any) {
        cudaError_t we = deps_.wait();
        if (we != cudaSuccess) return cuda_fail("get: cannot order after earlier calls", we);
        st = segs_.empty() ? T2I_OK : launch_segments<Mode::Get>(segs_, stream);
        // items for the copy engine (pinned host destinations, d2h_mode = 1):
        // one copy per run of consecutive pages
        const uint64_t P = uint64_t(1) << page_shift_;
        for (uint32_t i = 0; i < n && st == T2I_OK; ++i) {
            const Object* o = objs_[i];
            if (!use_ce[i] || o->nbytes == 0) continue;
            char* dst = static_cast<char*>(descs[i].dst);
            size_t j = 0;
            while (j < o->pages.size()) {
                size_t k = j + 1;
                while (k < o->pages.size() && o->pages[k] == o->pages[k - 1] + 1) ++k;
                const uint64_t off = j * P;
                const uint64_t bytes = std::min<uint64_t>(o->nbytes - off, (k - j) * P);
                const void* src = reinterpret_cast<const void*>(pool_ + uint64_t(o->pages[j]) * P);
                cudaError_t e = cudaMemcpyAsync(dst + off, src, bytes, cudaMemcpyDeviceToHost, stream);
                if (e != cudaSuccess) {
                    st = cuda_fail("get: host copy failed", e);
                    break;
                }
                ctl_.counters().d2h_copies++;
                j = k;
            }
        }
        // every page of the batch carries this call as a reader, even when it
        // failed part-way (copies enqueued before the failure may still be
        // reading them)
        uint32_t q = 0;
        cudaError_t ee = deps_.end(&q);
        for (uint32_t i = 0; i < n; ++i)
            for (uint32_t pg : objs_[i]->pages) deps_.mark_read(pg, q);
        if (st != T2I_OK) return st;  // nothing was counted: the get did not happen
        if (ee != cudaSuccess) st = cuda_fail("get: cannot record its event", ee);
    }
    // 3. LRU stamps and consumer counts, now that the copies are enqueued;
    //    objects consumed to zero are freed (their pages carry this call as
    //    a reader, so reuse waits for it)
    if (per_item) std::fill(per_item, per_item + n, T2I_OK);
    ctl_.account_get(&descs[0].id, n, sizeof(t2i_get_desc));
    ctl_.release_pending();
    return st;
}

t2i_status Store::view(t2i_id id, cudaStream_t stream, void** ptr, uint64_t* nbytes) {
    if (!ptr) {
        err_ = "view: null output";
        return T2I_ERR_INVALID;
    }
    *ptr = nullptr;
    if (nbytes) *nbytes = 0;
    const Object* o = nullptr;
    t2i_status st = ctl_.view(id, &o);
    if (st != T2I_OK) {
        err_ = ctl_.error();
        return st;
    }
    if (nbytes) *nbytes = o->nbytes;
    if (o->pages.empty()) return T2I_OK;
    DeviceGuard g(device_);
    int si = 0;
    if ((st = stream_slot(stream, &si)) != T2I_OK) return st;
    deps_.begin(si);
    for (uint32_t pg : o->pages) deps_.reads(pg);
    cudaError_t we = deps_.wait();
    if (we != cudaSuccess) return cuda_fail("view: cannot order after the object's writer", we);
    for (uint32_t pg : o->pages) deps_.mark_read(pg, StreamDeps::kOpen);
    *ptr = reinterpret_cast<void*>(pool_ + (uint64_t(o->pages[0]) << page_shift_));
    return T2I_OK;
}

// The consumer's store (this) allocates pages for the producer's objects and
// copies them page to page with the move kernel: source = the producer's
// pages, destination = the new pages (§5.2: the consumer allocates a block in
// its own arena and pulls the producer's bytes into it).
t2i_status Store::pull_from(Store& src, const t2i_id* ids, uint32_t n, uint32_t consumers, t2i_id* out_ids,
                            t2i_status* per_item, cudaStream_t stream) {
    if (n == 0) return T2I_OK;
    if (!ids || !out_ids) {
        err_ = "pull: null id array";
        return T2I_ERR_INVALID;
    }
    if (&src == this || src.device_ != device_ || src.page_shift_ != page_shift_) {
        err_ = "pull: the stores must differ, share a device and have the same page size";
        return T2I_ERR_INVALID;
    }
    // 1. every source id first (a failed pull changes nothing)
    std::vector<const Object*> so(n);
    t2i_status first = T2I_OK;
    for (uint32_t i = 0; i < n; ++i) {
        so[i] = src.ctl_.find(ids[i]);
        t2i_status s = so[i] ? T2I_OK : (src.ctl_.is_evicted(ids[i]) ? T2I_ERR_EVICTED : T2I_ERR_NOT_FOUND);
        if (s == T2I_ERR_EVICTED) src.ctl_.counters().misses++;
        if (per_item) per_item[i] = s;
        if (s != T2I_OK && first == T2I_OK) first = s;
    }
    if (first != T2I_OK) {
        err_ = "pull: a source id is not in the producer's store";
        return first;
    }
    // 2. room in this store, as intermediates
    std::vector<t2i_put_desc> pd(n);
    for (uint32_t i = 0; i < n; ++i)
        pd[i] = t2i_put_desc{nullptr, so[i]->nbytes, 0, so[i]->dtype_tag, 0, 0, 0, consumers, 0};
    t2i_status st = ctl_.put(pd.data(), n, out_ids, &objs_);
    if (st != T2I_OK) {
        err_ = ctl_.error();
        return st;
    }
    const std::vector<const Object*>& src_objs = so;
    // 3. page-to-page copies, after the producer's writer and this store's
    //    earlier users of the new pages
    DeviceGuard g(device_);
    int sd = 0, ss = 0;
    if ((st = stream_slot(stream, &sd)) != T2I_OK || (st = src.stream_slot(stream, &ss)) != T2I_OK) {
        ctl_.rollback_put(out_ids, n);
        return st;
    }
    const uint64_t P = uint64_t(1) << page_shift_;
    deps_.begin(sd);
    src.deps_.begin(ss);
    segs_.clear();
    for (uint32_t i = 0; i < n; ++i) {
        const Object* s_o = src_objs[i];
        const Object* d_o = objs_[i];
        for (size_t j = 0; j < s_o->pages.size(); ++j) {
            src.deps_.reads(s_o->pages[j]);
            deps_.writes(d_o->pages[j]);
            segs_.push_back({src.pool_ + uint64_t(s_o->pages[j]) * P, std::min<uint64_t>(P, s_o->nbytes - j * P),
                             &d_o->pages[j], 1u});
        }
    }
    cudaError_t we = deps_.wait();
    if (we == cudaSuccess) we = src.deps_.wait();
    if (we != cudaSuccess) {
        ctl_.rollback_put(out_ids, n);
        return cuda_fail("pull: cannot order after earlier calls", we);
    }
    if (!segs_.empty()) {
        st = launch_segments<Mode::Move>(segs_, stream);
        // marked even after a failure part-way: launches before it may still
        // be reading the sources and writing the pages handed back
        uint32_t qd = 0, qs = 0;
        cudaError_t e1 = deps_.end(&qd);
        cudaError_t e2 = src.deps_.end(&qs);
        for (uint32_t i = 0; i < n; ++i) {
            for (uint32_t pg : objs_[i]->pages) deps_.mark_write(pg, qd);
            for (uint32_t pg : src_objs[i]->pages) src.deps_.mark_read(pg, qs);
        }
        if (st != T2I_OK) {
            ctl_.rollback_put(out_ids, n);  // nothing counted on the sources
            return st;
        }
        if (e1 != cudaSuccess || e2 != cudaSuccess)
            st = cuda_fail("pull: cannot record its event", e1 != cudaSuccess ? e1 : e2);
    }
    // 4. the sources are read like a get (stamps, consumer counts)
    src.ctl_.account_get(ids, n, sizeof(t2i_id));
    src.ctl_.release_pending();
    return st;
}

// The consumer's half of a pull whose producer is not a store of this
// process: the source pages are given as a pool address and page lists.
t2i_status Store::pull_pages(const void* src_pool, uint64_t src_pool_bytes, const t2i_paged_object* objs, uint32_t n,
                             uint32_t consumers, t2i_id* out_ids, cudaStream_t stream) {
    if (n == 0) return T2I_OK;
    if (!src_pool || !objs || !out_ids) {
        err_ = "pull_pages: null pool, object or id array";
        return T2I_ERR_INVALID;
    }
    const uint64_t P = uint64_t(1) << page_shift_;
    const uint64_t sp = reinterpret_cast<uint64_t>(src_pool);
    if (src_pool_bytes < P || sp % 256 != 0 || sp + src_pool_bytes < sp) {
        err_ = "pull_pages: the source pool must be 256-byte aligned and hold at least one page";
        return T2I_ERR_INVALID;
    }
    if (overlaps_pool(sp, src_pool_bytes)) {
        err_ = "pull_pages: the source pool overlaps this store's pool";
        return T2I_ERR_INVALID;
    }
    Range r;
    if (!query_range(src_pool, &r) || r.kind != MemKind::Device || r.device != device_ || sp + src_pool_bytes > r.end) {
        err_ = "pull_pages: the source pool must be device memory of this store's device covering src_pool_bytes";
        return T2I_ERR_INVALID;
    }
    // 1. every object's page list first (a failed pull changes nothing)
    const uint64_t src_pages = src_pool_bytes / P;
    for (uint32_t i = 0; i < n; ++i) {
        const t2i_paged_object& o = objs[i];
        if (o.n_pages != o.nbytes / P + (o.nbytes % P != 0) || (o.n_pages && !o.pages)) {
            err_ = "pull_pages: object " + std::to_string(i) + ": n_pages must be nbytes / page_bytes rounded up";
            return T2I_ERR_INVALID;
        }
        for (uint32_t j = 0; j < o.n_pages; ++j)
            if (o.pages[j] >= src_pages) {
                err_ = "pull_pages: object " + std::to_string(i) + ": a page lies outside the source pool";
                return T2I_ERR_INVALID;
            }
    }
    // 2. room in this store, as intermediates
    std::vector<t2i_put_desc> pd(n);
    for (uint32_t i = 0; i < n; ++i) pd[i] = t2i_put_desc{nullptr, objs[i].nbytes, 0, objs[i].dtype_tag, 0, 0, 0, consumers, 0};
    t2i_status st = ctl_.put(pd.data(), n, out_ids, &objs_);
    if (st != T2I_OK) {
        err_ = ctl_.error();
        return st;
    }
    // 3. page-to-page copies, after this store's earlier users of the new pages
    DeviceGuard g(device_);
    int si = 0;
    if ((st = stream_slot(stream, &si)) != T2I_OK) {
        ctl_.rollback_put(out_ids, n);
        return st;
    }
    deps_.begin(si);
    segs_.clear();
    for (uint32_t i = 0; i < n; ++i) {
        const Object* d_o = objs_[i];
        for (uint32_t j = 0; j < objs[i].n_pages; ++j) {
            deps_.writes(d_o->pages[j]);
            segs_.push_back({sp + uint64_t(objs[i].pages[j]) * P, std::min<uint64_t>(P, objs[i].nbytes - uint64_t(j) * P),
                             &d_o->pages[j], 1u});
        }
    }
    if (segs_.empty()) return T2I_OK;
    cudaError_t we = deps_.wait();
    if (we != cudaSuccess) {
        ctl_.rollback_put(out_ids, n);
        return cuda_fail("pull_pages: cannot order after earlier calls", we);
    }
    st = launch_segments<Mode::Move>(segs_, stream);
    // marked even after a failure part-way: launches before it may still be
    // writing the pages handed back
    uint32_t q = 0;
    cudaError_t ee = deps_.end(&q);
    for (uint32_t i = 0; i < n; ++i)
        for (uint32_t pg : objs_[i]->pages) deps_.mark_write(pg, q);
    if (st != T2I_OK) {
        ctl_.rollback_put(out_ids, n);
        return st;
    }
    if (ee != cudaSuccess) return cuda_fail("pull_pages: cannot record its event", ee);
    return T2I_OK;
}

t2i_status Store::compact(uint64_t limit_bytes, cudaStream_t stream, uint64_t* moved) {
    if (moved) *moved = 0;
    t2i_status st = ctl_.begin_compact(limit_bytes);
    if (st != T2I_OK) {
        err_ = ctl_.error();
        return st;
    }
    DeviceGuard g(device_);
    int si = 0;
    if ((st = stream_slot(stream, &si)) != T2I_OK) {
        ctl_.rollback_compact();
        return st;
    }
    // Planned and launched a batch of moves at a time, so that the first moves
    // run while the rest is planned. The first batch is small, so that the GPU
    // starts early; each later one is 4x larger, up to one launch's worth
    // (planning a move takes ~50 ns on the host, copying a 2 MiB page
    // ~0.6 us on the GPU, so the plan stays ahead).
    const uint64_t P = uint64_t(1) << page_shift_;
    uint64_t total = 0;
    cudaError_t event_error = cudaSuccess;
    bool more = true;
    size_t batch = std::min<size_t>(kCompactFirstBatch, kMovesPerLaunch);
    while (more) {
        batch_.clear();
        more = ctl_.plan_more(batch, &batch_);
        batch = std::min<size_t>(batch * 4, kMovesPerLaunch);
        if (batch_.empty()) break;
        deps_.begin(si);
        if (deps_.n_streams() > 1) {  // with one stream there is nothing to wait for
            for (const t2i_move& m : batch_) {
                deps_.reads(m.src_page);
                deps_.writes(m.dst_page);
            }
        }
        cudaError_t we = deps_.wait();
        if (we != cudaSuccess) {
            ctl_.rollback_compact();
            return cuda_fail("compact: cannot order after earlier calls", we);
        }
        segs_.clear();
        // each move is a one-page segment whose source is the old page
        for (const t2i_move& m : batch_)
            segs_.push_back({pool_ + uint64_t(m.src_page) * P, m.valid_bytes, &m.dst_page, 1u});
        st = launch_segments<Mode::Move>(segs_, stream);
        // marked even after a failure: launches before it may still be
        // reading the old pages and writing the new ones
        uint32_t q = 0;
        cudaError_t ee = deps_.end(&q);
        for (const t2i_move& m : batch_) {
            deps_.mark_read(m.src_page, q);
            deps_.mark_write(m.dst_page, q);
        }
        if (st != T2I_OK) {
            // the old pages still hold every byte: point the page tables back
            ctl_.rollback_compact();
            return st;
        }
        if (ee != cudaSuccess && event_error == cudaSuccess) event_error = ee;
        total += batch_.size();
    }
    ctl_.finish_compact();  // the free pages are rebuilt while the moves run
    if (moved) *moved = total;
    if (event_error != cudaSuccess) return cuda_fail("compact: cannot record its event", event_error);
    return T2I_OK;
}

}  // namespace t2i

// ======================================================================= C ABI
using t2i::Store;

struct t2i_store {
    Store* s;
};

extern "C" {

t2i_status t2i_store_create(void* pool_dev, const t2i_store_config* cfg, int device, t2i_store** out) {
    if (!out) {
        t2i::set_thread_error("t2i_store_create: null out");
        return T2I_ERR_INVALID;
    }
    *out = nullptr;
    if (!cfg || !pool_dev) {
        t2i::set_thread_error("t2i_store_create: null pool or config");
        return T2I_ERR_INVALID;
    }
    const int shift = t2i::log2_exact(cfg->page_bytes);
    if (shift < 8 || shift > 30) {
        t2i::set_thread_error("t2i_store_create: page_bytes must be a power of two in [256 B, 1 GiB]");
        return T2I_ERR_INVALID;
    }
    if (cfg->pool_bytes / cfg->page_bytes > 0xFFFFFFFFull || cfg->h2d_mode > 1 || cfg->check_pointers > 1 ||
        cfg->alloc_policy > 1 || cfg->d2h_mode > 1) {
        t2i::set_thread_error("t2i_store_create: too many pages or a bad flag");
        return T2I_ERR_INVALID;
    }
    if (reinterpret_cast<uint64_t>(pool_dev) & 255) {
        t2i::set_thread_error("t2i_store_create: the pool must be 256-byte aligned");
        return T2I_ERR_INVALID;
    }
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
        cudaGetLastError();
        t2i::set_thread_error("t2i_store_create: no such CUDA device");
        return T2I_ERR_CUDA;
    }
    t2i::Range r;
    if (!t2i::query_range(pool_dev, &r) || r.kind != t2i::MemKind::Device || r.device != device ||
        reinterpret_cast<uint64_t>(pool_dev) + cfg->pool_bytes > r.end) {
        t2i::set_thread_error("t2i_store_create: the pool must be device memory of `device` covering pool_bytes");
        return T2I_ERR_INVALID;
    }
    Store* s = nullptr;
    try {
        s = new Store(pool_dev, *cfg, device);
    } catch (const std::exception& e) {
        t2i::set_thread_error(std::string("t2i_store_create: host error: ") + e.what());
        return T2I_ERR_INVALID;
    }
    std::string err;
    t2i_status st = s->init(&err);
    if (st != T2I_OK) {
        delete s;
        t2i::set_thread_error("t2i_store_create: " + err);
        return st;
    }
    *out = new t2i_store{s};
    return T2I_OK;
}

t2i_status t2i_store_destroy(t2i_store* store) {
    if (!store) return T2I_OK;
    delete store->s;
    delete store;
    return T2I_OK;
}

// Every store call: an NVTX range, the store's lock, and no C++ exception
// past the C boundary (host memory exhaustion and the like become INVALID
// with a message).
#define T2I_STORE_CALL(store, expr)                                   \
    do {                                                              \
        if (!(store)) return T2I_ERR_INVALID;                         \
        t2i::NvtxRange nvtx_range(__func__);                          \
        std::lock_guard<std::mutex> lock((store)->s->mu);             \
        try {                                                         \
            return (expr);                                            \
        } catch (const std::exception& e) {                           \
            (store)->s->set_error(std::string("host error: ") + e.what()); \
            return T2I_ERR_INVALID;                                   \
        }                                                             \
    } while (0)

t2i_status t2i_put_batch(t2i_store* store, const t2i_put_desc* descs, uint32_t n, t2i_id* out_ids,
                         void* cuda_stream) {
    T2I_STORE_CALL(store, store->s->put(descs, n, out_ids, static_cast<cudaStream_t>(cuda_stream)));
}

t2i_status t2i_get_batch(t2i_store* store, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item,
                         void* cuda_stream) {
    T2I_STORE_CALL(store, store->s->get(descs, n, per_item, static_cast<cudaStream_t>(cuda_stream)));
}

t2i_status t2i_get_batch_after(t2i_store* store, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item,
                               void* cuda_stream, void* wait_event) {
    T2I_STORE_CALL(store, store->s->get(descs, n, per_item, static_cast<cudaStream_t>(cuda_stream),
                                        static_cast<cudaEvent_t>(wait_event)));
}

t2i_status t2i_free(t2i_store* store, const t2i_id* ids, uint32_t n) {
    T2I_STORE_CALL(store, store->s->free(ids, n));
}

t2i_status t2i_put_layers(t2i_store* store, const t2i_put_desc* descs, const uint32_t* layer_off, uint32_t n_layers,
                          uint32_t first, t2i_id* out_ids, void* cuda_stream, void* const* events) {
    if (!store || !layer_off || first > n_layers || (n_layers > first && (!descs || !out_ids))) {
        if (store) store->s->set_error("put_layers: bad arguments");
        return T2I_ERR_INVALID;
    }
    for (uint32_t l = first; l < n_layers; ++l) {
        if (layer_off[l + 1] < layer_off[l]) {
            store->s->set_error("put_layers: layer offsets must not decrease");
            return T2I_ERR_INVALID;
        }
    }
    t2i::NvtxRange nvtx_range("t2i_put_layers");
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    for (uint32_t l = first; l < n_layers; ++l) {
        t2i_status st;
        {
            std::lock_guard<std::mutex> lock(store->s->mu);
            try {
                st = store->s->put(descs + layer_off[l], layer_off[l + 1] - layer_off[l], out_ids + layer_off[l],
                                   stream);
            } catch (const std::exception& e) {
                store->s->set_error(std::string("host error: ") + e.what());
                st = T2I_ERR_INVALID;
            }
        }
        if (st != T2I_OK) return st;
        if (events && events[l]) {
            cudaError_t e = cudaEventRecord(static_cast<cudaEvent_t>(events[l]), stream);
            if (e != cudaSuccess) {
                store->s->set_error(std::string("put_layers: event record failed: ") + cudaGetErrorString(e));
                return T2I_ERR_CUDA;
            }
        }
    }
    return T2I_OK;
}

t2i_status t2i_view(t2i_store* store, t2i_id id, void* cuda_stream, void** dev_ptr, uint64_t* nbytes) {
    T2I_STORE_CALL(store, store->s->view(id, static_cast<cudaStream_t>(cuda_stream), dev_ptr, nbytes));
}

t2i_status t2i_pull(t2i_store* dst, t2i_store* src, const t2i_id* src_ids, uint32_t n, uint32_t consumers,
                    t2i_id* out_ids, t2i_status* per_item, void* cuda_stream) {
    if (!dst || !src) return T2I_ERR_INVALID;
    if (dst == src) {
        dst->s->set_error("pull: a store cannot pull from itself");
        return T2I_ERR_INVALID;
    }
    t2i::NvtxRange nvtx_range("t2i_pull");
    std::scoped_lock lock(dst->s->mu, src->s->mu);
    try {
        return dst->s->pull_from(*src->s, src_ids, n, consumers, out_ids, per_item,
                                 static_cast<cudaStream_t>(cuda_stream));
    } catch (const std::exception& e) {
        dst->s->set_error(std::string("host error: ") + e.what());
        return T2I_ERR_INVALID;
    }
}

t2i_status t2i_pull_pages(t2i_store* dst, const void* src_pool, uint64_t src_pool_bytes,
                          const t2i_paged_object* objs, uint32_t n, uint32_t consumers, t2i_id* out_ids,
                          void* cuda_stream) {
    T2I_STORE_CALL(dst, dst->s->pull_pages(src_pool, src_pool_bytes, objs, n, consumers, out_ids,
                                          static_cast<cudaStream_t>(cuda_stream)));
}

t2i_status t2i_compact(t2i_store* store, uint64_t limit_bytes, void* cuda_stream, uint64_t* pages_moved) {
    T2I_STORE_CALL(store, store->s->compact(limit_bytes, static_cast<cudaStream_t>(cuda_stream), pages_moved));
}

t2i_status t2i_inject_launch_failure(t2i_store* store, uint32_t countdown) {
    if (!store) return T2I_ERR_INVALID;
    std::lock_guard<std::mutex> lock(store->s->mu);
    store->s->inject_launch_failure(countdown);
    return T2I_OK;
}

t2i_status t2i_store_stats(const t2i_store* store, t2i_stats* out) {
    if (!store || !out) return T2I_ERR_INVALID;
    std::lock_guard<std::mutex> lock(store->s->mu);
    store->s->ctl().stats(out);
    return T2I_OK;
}

const t2i_ctl* t2i_store_ctl(const t2i_store* store) { return store ? store->s->ctl_handle() : nullptr; }

const char* t2i_last_error(const t2i_store* store) {
    if (!store) return t2i::thread_error();
    return store->s->error().c_str();
}

}  // extern "C"

// ================================================= gather without allocation
// t2i_gather_noalloc: the chunked gather of one object's pages for callers
// that cannot allocate device memory (see include/t2istore.h). Its chunk
// counters live in a file-scope array that is part of the library's device
// image, so the call allocates nothing. The paper has no counterpart.
namespace t2i {
namespace {
constexpr uint32_t kNoAllocCounters = 64;  // one per launch of a call: 2 KiB in all
constexpr uint64_t kNoAllocMaxPagesPerLaunch = (kBlobLarge - sizeof(SegDesc)) / sizeof(uint32_t);
// pages per launch: the page list fits the parameters and the bytes fit
// 32-bit granule offsets
uint64_t noalloc_pages_per_launch(uint64_t page_bytes) {
    return std::min<uint64_t>(kNoAllocMaxPagesPerLaunch, std::max<uint64_t>(1, kMaxSegBytes / page_bytes));
}
constexpr int kNoAllocMaxDevices = 64;
}  // namespace
}  // namespace t2i

// Every GPU that loads the library holds this array until the process exits.
static __device__ __align__(256) t2i::WorkCounter t2i_noalloc_scratch[t2i::kNoAllocCounters];

namespace t2i {
namespace {

// The kernels a call can run, as a store's chunked get picks them: the
// cast-capable gather for 16-byte aligned destinations and for casts, the
// copy-only gather for other destinations without a cast.
enum NoAllocKernel { kNoAllocGetAligned = 0, kNoAllocGetAny = 1, kNoAllocCopyAny = 2 };

// Per-device set-up, done once by the first call on that device: the
// device address of the scratch array (host code sees only a stand-in for
// the symbol) and the resident CTAs of the gather kernels (its grid size).
struct NoAllocDevice {
    bool ready = false;
    WorkCounter* scratch = nullptr;
    int max_ctas[3] = {1, 1, 1};  // [NoAllocKernel]
};

const void* noalloc_kernel(int k) {
    return k == kNoAllocGetAligned ? reinterpret_cast<const void*>(gather_get_kernel<kBlobLarge, false>)
           : k == kNoAllocGetAny   ? reinterpret_cast<const void*>(gather_get_kernel<kBlobLarge, true>)
                                   : reinterpret_cast<const void*>(gather_copy_kernel<kBlobLarge, true>);
}

std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_dev[kNoAllocMaxDevices];

t2i_status noalloc_setup(int device, NoAllocDevice** out) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocDevice& d = g_noalloc_dev[device];
    if (!d.ready) {
        DeviceGuard g(device);
        void* ptr = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&ptr, t2i_noalloc_scratch);
        if (e != cudaSuccess || !ptr) {
            set_thread_error(std::string("t2i_gather_noalloc: cannot get the scratch array's device address: ") +
                             cudaGetErrorString(e));
            return T2I_ERR_CUDA;
        }
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess || sms <= 0) {
            set_thread_error("t2i_gather_noalloc: cannot query the device");
            return T2I_ERR_CUDA;
        }
        for (int k = 0; k < 3; ++k) {
            int occ = 0;
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, noalloc_kernel(k), kThreads, 0);
            d.max_ctas[k] = sms * (occ > 0 ? occ : 1);
        }
        d.scratch = static_cast<WorkCounter*>(ptr);
        d.ready = true;
    }
    *out = &d;
    return T2I_OK;
}

// One launch of kernel `kern`: `np` pages of the object starting at page
// index `p0`.
t2i_status noalloc_one(const NoAllocDevice& d, int kern, uint32_t k, const void* pool, int shift,
                       const uint32_t* pages, uint64_t p0, uint64_t np, uint64_t nbytes, unsigned char* dst, bool cast,
                       cudaStream_t stream) {
    thread_local LaunchParams<kBlobLarge> p;  // host-side parameter staging (no device memory)
    const uint64_t P = uint64_t(1) << shift;
    const uint64_t off = p0 * P;
    const uint64_t seg_bytes = std::min<uint64_t>(nbytes - off, np * P);
    p.h.pool = reinterpret_cast<uint64_t>(pool);
    p.h.work = reinterpret_cast<uint64_t>(d.scratch + k);
    p.h.n_seg = 1;
    p.h.n_granules = static_cast<uint32_t>((seg_bytes + kGranule - 1) / kGranule);
    p.h.page_shift = static_cast<uint32_t>(shift);
    p.h.piece_bytes = static_cast<uint32_t>(std::min<uint64_t>(kPieceBytes, P));
    p.h.pages_offset = sizeof(SegDesc);
    p.h.chunk_granules = kChunkGranules;
    p.h.flags = 0;
    p.h.prefetch_ctas = 0;
    SegDesc s;
    s.user = reinterpret_cast<uint64_t>(dst) + (cast ? off / 2 : off);
    s.nbytes_flags = seg_bytes | (cast ? kCastFlag : 0);
    s.start = 0;
    s.page_begin = 0;
    std::memcpy(p.blob, &s, sizeof(s));
    std::memcpy(p.blob + sizeof(SegDesc), pages + p0, np * sizeof(uint32_t));
    const uint64_t want = (seg_bytes + kMinCtaBytes - 1) / kMinCtaBytes;
    const unsigned grid = static_cast<unsigned>(std::max<uint64_t>(1, std::min<uint64_t>(want, uint64_t(d.max_ctas[kern]))));
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(kThreads);
    lc.stream = stream;
    void* args[] = {&p};
    cudaError_t e = cudaLaunchKernelExC(&lc, noalloc_kernel(kern), args);
    if (e != cudaSuccess) {
        set_thread_error(std::string("t2i_gather_noalloc: kernel launch failed: ") + cudaGetErrorString(e));
        return T2I_ERR_CUDA;
    }
    return T2I_OK;
}

}  // namespace
}  // namespace t2i

extern "C" t2i_status t2i_gather_noalloc(const void* pool_dev, uint64_t pool_bytes, uint64_t page_bytes,
                                         const uint32_t* pages, uint32_t n_pages, uint64_t nbytes, void* dst_dev,
                                         uint64_t dst_bytes, uint32_t cast, int device, void* cuda_stream) {
    using namespace t2i;
    NvtxRange nvtx_range(__func__);
    try {
        const int shift = log2_exact(page_bytes);
        if (!pool_dev || shift < 8 || shift > 30 || pool_bytes < page_bytes || pool_bytes % page_bytes != 0 ||
            cast > 1) {
            set_thread_error("t2i_gather_noalloc: null pool, page_bytes not a power of two in [256 B, 1 GiB], "
                             "pool_bytes not a positive multiple of page_bytes, or cast not 0/1");
            return T2I_ERR_INVALID;
        }
        const uint64_t need = nbytes / page_bytes + (nbytes % page_bytes != 0);
        if (n_pages != need) {
            set_thread_error("t2i_gather_noalloc: n_pages must be nbytes / page_bytes rounded up");
            return T2I_ERR_INVALID;
        }
        const uint64_t per_launch = noalloc_pages_per_launch(page_bytes);
        const uint64_t max_pages = uint64_t(kNoAllocCounters) * per_launch;
        if (n_pages > max_pages) {
            set_thread_error("t2i_gather_noalloc: " + std::to_string(n_pages) + " pages exceed the maximum of " +
                             std::to_string(max_pages) + " (" + std::to_string(kNoAllocCounters) +
                             " launches of " + std::to_string(per_launch) + " pages, one scratch counter each)");
            return T2I_ERR_INVALID;
        }
        if (nbytes == 0) return T2I_OK;
        if (!pages || !dst_dev) {
            set_thread_error("t2i_gather_noalloc: null page list or destination");
            return T2I_ERR_INVALID;
        }
        if (cast ? (nbytes % 4 != 0 || dst_bytes < nbytes / 2 || (reinterpret_cast<uint64_t>(dst_dev) & 1))
                 : dst_bytes < nbytes) {
            set_thread_error("t2i_gather_noalloc: dst_bytes too small, or a cast with nbytes % 4 != 0 or an odd "
                             "destination address");
            return T2I_ERR_INVALID;
        }
        const uint64_t total_pages = pool_bytes / page_bytes;
        for (uint32_t i = 0; i < n_pages; ++i)
            if (pages[i] >= total_pages) {
                set_thread_error("t2i_gather_noalloc: a page index is outside the pool");
                return T2I_ERR_INVALID;
            }
        int n_dev = 0;
        if (cudaGetDeviceCount(&n_dev) != cudaSuccess || device < 0 || device >= n_dev ||
            device >= kNoAllocMaxDevices) {
            set_thread_error("t2i_gather_noalloc: no such CUDA device");
            return T2I_ERR_INVALID;
        }
        // both ranges must lie in device memory of `device`, and not overlap
        const uint64_t pa = reinterpret_cast<uint64_t>(pool_dev), da = reinterpret_cast<uint64_t>(dst_dev);
        const uint64_t dn = cast ? nbytes / 2 : nbytes;
        Range rp, rd;
        if (!query_range(pool_dev, &rp) || rp.kind != MemKind::Device || rp.device != device ||
            pa + pool_bytes > rp.end || !query_range(dst_dev, &rd) || rd.kind != MemKind::Device ||
            rd.device != device || da + dn > rd.end || da + dn < da) {
            set_thread_error("t2i_gather_noalloc: the pool and the destination must be device memory of `device` "
                             "covering their sizes");
            return T2I_ERR_INVALID;
        }
        if (da < pa + pool_bytes && pa < da + dn) {
            set_thread_error("t2i_gather_noalloc: the destination overlaps the pool");
            return T2I_ERR_INVALID;
        }
        NoAllocDevice* d = nullptr;
        t2i_status st = noalloc_setup(device, &d);
        if (st != T2I_OK) return st;
        DeviceGuard g(device);
        cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
        const uint64_t n_launch = (n_pages + per_launch - 1) / per_launch;
        // the counters this call uses start at zero whatever an earlier call left
        cudaError_t e = cudaMemsetAsync(d->scratch, 0, n_launch * sizeof(WorkCounter), stream);
        if (e != cudaSuccess) {
            set_thread_error(std::string("t2i_gather_noalloc: cannot clear the scratch counters: ") +
                             cudaGetErrorString(e));
            return T2I_ERR_CUDA;
        }
        const int kern = (da & 15u) == 0 ? kNoAllocGetAligned : cast ? kNoAllocGetAny : kNoAllocCopyAny;
        unsigned char* dst = static_cast<unsigned char*>(dst_dev);
        for (uint64_t k = 0; k < n_launch; ++k) {
            const uint64_t p0 = k * per_launch;
            const uint64_t np = std::min<uint64_t>(per_launch, n_pages - p0);
            st = noalloc_one(*d, kern, uint32_t(k), pool_dev, shift, pages, p0, np, nbytes, dst, cast != 0, stream);
            if (st != T2I_OK) return st;
        }
        return T2I_OK;
    } catch (const std::exception& ex) {
        set_thread_error(std::string("t2i_gather_noalloc: host error: ") + ex.what());
        return T2I_ERR_INVALID;
    }
}
