// C ABI of the host control core (t2i_ctl_*). No CUDA here.
#include <new>
#include <string>

#include "common.hpp"
#include "control.hpp"

namespace t2i {
namespace {
thread_local std::string g_thread_error;
}
void set_thread_error(const std::string& e) { g_thread_error = e; }
const char* thread_error() { return g_thread_error.c_str(); }
}  // namespace t2i

using t2i::Control;

#define T2I_GUARD_BEGIN try {
#define T2I_GUARD_END(ctl)                                               \
    }                                                                    \
    catch (const std::exception& e) {                                    \
        (ctl)->core->set_error(std::string("host error: ") + e.what());  \
        return T2I_ERR_INVALID;                                          \
    }

namespace {
// Queries of a store's control core take the store's lock.
struct QueryLock {
    std::unique_lock<std::mutex> lk;
    explicit QueryLock(const t2i_ctl* c) {
        if (c->mu) lk = std::unique_lock<std::mutex>(*c->mu);
    }
};
}  // namespace

extern "C" {

t2i_status t2i_ctl_create(uint64_t total_pages, uint64_t page_bytes, uint32_t alloc_policy, t2i_ctl** out) {
    if (!out) {
        t2i::set_thread_error("t2i_ctl_create: null out");
        return T2I_ERR_INVALID;
    }
    *out = nullptr;
    if (page_bytes == 0 || total_pages > 0xFFFFFFFFull || alloc_policy > 1) {
        t2i::set_thread_error("t2i_ctl_create: page_bytes must be > 0, total_pages < 2^32, alloc_policy 0 or 1");
        return T2I_ERR_INVALID;
    }
    try {
        t2i_ctl* c = new t2i_ctl{new Control(total_pages, page_bytes, alloc_policy), true, nullptr};
        *out = c;
    } catch (const std::exception& e) {
        t2i::set_thread_error(std::string("t2i_ctl_create: host error: ") + e.what());
        return T2I_ERR_INVALID;
    }
    return T2I_OK;
}

t2i_status t2i_ctl_destroy(t2i_ctl* ctl) {
    if (!ctl) return T2I_OK;
    if (!ctl->owned) return T2I_ERR_INVALID;
    delete ctl->core;
    delete ctl;
    return T2I_OK;
}

t2i_status t2i_ctl_put(t2i_ctl* ctl, const t2i_put_desc* descs, uint32_t n, t2i_id* out_ids) {
    if (!ctl || !ctl->owned) return T2I_ERR_INVALID;
    T2I_GUARD_BEGIN
    return ctl->core->put(descs, n, out_ids, nullptr);
    T2I_GUARD_END(ctl)
}

t2i_status t2i_ctl_get(t2i_ctl* ctl, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item) {
    if (!ctl || !ctl->owned) return T2I_ERR_INVALID;
    T2I_GUARD_BEGIN
    return ctl->core->get(descs, n, per_item, nullptr);
    T2I_GUARD_END(ctl)
}

t2i_status t2i_ctl_free(t2i_ctl* ctl, const t2i_id* ids, uint32_t n) {
    if (!ctl || !ctl->owned) return T2I_ERR_INVALID;
    T2I_GUARD_BEGIN
    return ctl->core->free(ids, n);
    T2I_GUARD_END(ctl)
}

t2i_status t2i_ctl_compact(t2i_ctl* ctl, uint64_t limit_bytes, t2i_move* moves, uint64_t cap, uint64_t* n_moves) {
    if (!ctl || !ctl->owned) return T2I_ERR_INVALID;
    T2I_GUARD_BEGIN
    Control& c = *ctl->core;
    // a short moves buffer must change nothing: count the moves first
    if (moves && limit_bytes % c.page_bytes() == 0 && limit_bytes / c.page_bytes() <= c.total_pages() &&
        c.used_pages() <= limit_bytes / c.page_bytes()) {
        const uint64_t need = c.live_pages_at_or_above(limit_bytes / c.page_bytes());
        if (need > cap) {
            if (n_moves) *n_moves = need;
            c.set_error("compact: the moves buffer is too small");
            return T2I_ERR_INVALID;
        }
    }
    std::vector<t2i_move> mv;
    t2i_status st = c.compact(limit_bytes, &mv);
    if (n_moves) *n_moves = mv.size();
    if (st != T2I_OK) return st;
    if (moves)
        for (size_t i = 0; i < mv.size(); ++i) moves[i] = mv[i];
    return T2I_OK;
    T2I_GUARD_END(ctl)
}

t2i_status t2i_ctl_object(const t2i_ctl* ctl, t2i_id id, t2i_object_info* info, uint32_t* pages, uint64_t cap) {
    if (!ctl) return T2I_ERR_INVALID;
    QueryLock ql(ctl);
    const t2i::Object* o = ctl->core->find(id);
    if (!o) return ctl->core->is_evicted(id) ? T2I_ERR_EVICTED : T2I_ERR_NOT_FOUND;
    if (info) {
        info->nbytes = o->nbytes;
        info->group = o->group->key;
        info->dtype_tag = o->dtype_tag;
        info->order = o->order;
        info->evictable = o->evictable ? 1u : 0u;
        info->n_pages = static_cast<uint32_t>(o->pages.size());
        info->consumers_left = o->consumers_left;
        info->reserved = 0;
    }
    if (pages) {
        const uint64_t k = o->pages.size() < cap ? o->pages.size() : cap;
        for (uint64_t i = 0; i < k; ++i) pages[i] = o->pages[i];
    }
    return T2I_OK;
}

t2i_status t2i_ctl_free_pages(const t2i_ctl* ctl, uint32_t* out, uint64_t cap, uint64_t* n) {
    if (!ctl) return T2I_ERR_INVALID;
    QueryLock ql(ctl);
    const std::vector<uint32_t> f = ctl->core->free_list();
    if (n) *n = f.size();
    if (out) {
        const uint64_t k = f.size() < cap ? f.size() : cap;
        for (uint64_t i = 0; i < k; ++i) out[i] = f[i];
    }
    return T2I_OK;
}

t2i_status t2i_ctl_last_evictions(const t2i_ctl* ctl, t2i_id* out, uint64_t cap, uint64_t* n) {
    if (!ctl) return T2I_ERR_INVALID;
    QueryLock ql(ctl);
    const auto& e = ctl->core->last_evictions();
    if (n) *n = e.size();
    if (out) {
        const uint64_t k = e.size() < cap ? e.size() : cap;
        for (uint64_t i = 0; i < k; ++i) out[i] = e[i];
    }
    return T2I_OK;
}

t2i_status t2i_ctl_stats(const t2i_ctl* ctl, t2i_stats* out) {
    if (!ctl || !out) return T2I_ERR_INVALID;
    QueryLock ql(ctl);
    ctl->core->stats(out);
    return T2I_OK;
}

const char* t2i_ctl_last_error(const t2i_ctl* ctl) {
    if (!ctl) return t2i::thread_error();
    return ctl->core->error().c_str();
}

}  // extern "C"
