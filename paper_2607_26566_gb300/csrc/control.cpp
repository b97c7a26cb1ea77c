// Host control core: see control.hpp for the rules it implements.
#include "control.hpp"

#include <cstdint>

#include <algorithm>
#include <string>

namespace t2i {

// ---------------------------------------------------------------- IdTable
uintptr_t IdTable::get(uint64_t id) const {
    const uint64_t leaf = id >> kLeafBits;
    if (leaf >= leaves_.size() || !leaves_[leaf]) return 0;
    return leaves_[leaf]->slot[id & (kLeafSize - 1)];
}

void IdTable::set(uint64_t id, uintptr_t v, uint64_t /*next_id*/) {
    const uint64_t leaf = id >> kLeafBits;
    if (leaf >= leaves_.size()) leaves_.resize(leaf + 1);
    if (!leaves_[leaf]) leaves_[leaf].reset(new Leaf());
    Leaf* L = leaves_[leaf].get();
    uintptr_t& s = L->slot[id & (kLeafSize - 1)];
    if (s == 0) L->used++;
    s = v;
}

void IdTable::clear(uint64_t id, uint64_t next_id) {
    const uint64_t leaf = id >> kLeafBits;
    if (leaf >= leaves_.size() || !leaves_[leaf]) return;
    Leaf* L = leaves_[leaf].get();
    uintptr_t& s = L->slot[id & (kLeafSize - 1)];
    if (s != 0) {
        s = 0;
        L->used--;
    }
    // every id of the leaf has been issued and none is live or evicted: no
    // lookup can find anything in it any more
    if (L->used == 0 && (leaf + 1) * kLeafSize <= next_id) leaves_[leaf].reset();
}

// ---------------------------------------------------------------- FreePages
FreePages::FreePages(uint64_t total_pages, uint32_t policy) : policy_(policy), count_(total_pages) {
    if (policy_ == 0) {
        stack_.reserve(total_pages);
        for (uint64_t p = total_pages; p-- > 0;) stack_.push_back(static_cast<uint32_t>(p));
    } else if (total_pages) {
        runs_[0] = static_cast<uint32_t>(total_pages);
    }
}

void FreePages::take(uint64_t k, std::vector<uint32_t>* out) {
    out->resize(k);
    count_ -= k;
    if (policy_ == 0) {
        for (uint64_t j = 0; j < k; ++j) {
            (*out)[j] = stack_.back();
            stack_.pop_back();
        }
        return;
    }
    if (k == 0) return;
    for (auto it = runs_.begin(); it != runs_.end(); ++it) {  // first fit
        if (it->second >= k) {
            const uint32_t start = it->first, len = it->second;
            runs_.erase(it);
            if (len > k) runs_[start + uint32_t(k)] = len - uint32_t(k);
            for (uint64_t j = 0; j < k; ++j) (*out)[j] = start + uint32_t(j);
            return;
        }
    }
    uint64_t j = 0;  // no run is long enough: the lowest pages
    while (j < k) {
        auto it = runs_.begin();
        const uint32_t start = it->first, len = it->second;
        const uint32_t m = uint32_t(std::min<uint64_t>(len, k - j));
        runs_.erase(it);
        if (len > m) runs_[start + m] = len - m;
        for (uint32_t t = 0; t < m; ++t) (*out)[j++] = start + t;
    }
}

void FreePages::insert_page(uint32_t p) {
    auto next = runs_.lower_bound(p);
    if (next != runs_.begin()) {
        auto prev = std::prev(next);
        if (prev->first + prev->second == p) {
            prev->second++;
            if (next != runs_.end() && next->first == p + 1) {
                prev->second += next->second;
                runs_.erase(next);
            }
            return;
        }
    }
    if (next != runs_.end() && next->first == p + 1) {
        const uint32_t len = next->second + 1;
        runs_.erase(next);
        runs_[p] = len;
    } else {
        runs_[p] = 1;
    }
}

void FreePages::give(const std::vector<uint32_t>& pages, bool undo) {
    count_ += pages.size();
    if (policy_ == 0) {
        if (undo)
            for (size_t j = pages.size(); j-- > 0;) stack_.push_back(pages[j]);
        else
            for (uint32_t p : pages) stack_.push_back(p);
        return;
    }
    for (uint32_t p : pages) insert_page(p);
}

std::vector<uint32_t> FreePages::list() const {
    if (policy_ == 0) return stack_;
    std::vector<uint32_t> out;
    out.reserve(count_);
    for (const auto& r : runs_)
        for (uint32_t t = 0; t < r.second; ++t) out.push_back(r.first + t);
    return out;
}

// ---------------------------------------------------------------- Control
Control::Control(uint64_t total_pages, uint64_t page_bytes, uint32_t policy)
    : P_(page_bytes),
      total_pages_(total_pages),
      limit_pages_(total_pages),
      free_(total_pages, policy),
      page_obj_(total_pages, nullptr),
      page_idx_(total_pages, 0) {}

void Control::own(const Object* o) {
    for (uint32_t j = 0; j < o->pages.size(); ++j) {
        page_obj_[o->pages[j]] = const_cast<Object*>(o);
        page_idx_[o->pages[j]] = j;
    }
}

void Control::disown(const Object* o) {
    for (uint32_t p : o->pages) page_obj_[p] = nullptr;
}

Control::~Control() {
    for (Object* o : live_) delete o;
}

Group* Control::group_for(uint64_t key) {
    auto it = groups_.find(key);
    if (it != groups_.end()) return it->second.get();
    auto g = std::make_unique<Group>();
    g->key = key;
    Group* raw = g.get();
    groups_.emplace(key, std::move(g));
    return raw;
}

void Control::maybe_drop_group(Group* g) {
    if (g->n_objects == 0 && g->victims.empty() && g->rec_key == 0 && g->epoch != epoch_) groups_.erase(g->key);
}

void Control::touch(Object* o) {
    Group* g = o->group;
    g->last = ++clock_;
    if (g->epoch != epoch_) {
        g->epoch = epoch_;
        touched_.push_back(g);
    }
}

void Control::flush_touches() {
    for (Group* g : touched_) {
        if (g->victims.empty()) continue;
        if (g->rec_key) recency_.erase({g->rec_key, g});
        recency_.insert({g->last, g});
        g->rec_key = g->last;
    }
    touched_.clear();
    ++epoch_;
}

void Control::release(Object* o, bool evicted) {
    const uint64_t np = o->pages.size();
    disown(o);
    free_.give(o->pages);
    used_pages_ -= np;
    Group* g = o->group;
    g->n_objects--;
    if (o->evictable) {
        g->victims.erase({o->order, o->id});
        g->evictable_pages -= np;
        evictable_pages_ -= np;
        if (g->victims.empty() && g->rec_key) {
            recency_.erase({g->rec_key, g});
            g->rec_key = 0;
        }
    }
    const size_t i = o->live_index;
    live_[i] = live_.back();
    live_[i]->live_index = i;
    live_.pop_back();
    if (evicted)
        ids_.set(o->id, IdTable::kEvicted, next_id_);
    else
        ids_.clear(o->id, next_id_);
    delete o;
    maybe_drop_group(g);
}

uint64_t Control::live_pages_at_or_above(uint64_t limit) const {
    uint64_t k = 0;
    for (uint64_t p = limit; p < limit_pages_; ++p) k += page_obj_[p] != nullptr;
    return k;
}

t2i_status Control::view(uint64_t id, const Object** out) {
    *out = nullptr;
    const uintptr_t v = ids_.get(id);
    if (v == 0) {
        err_ = "view: id " + std::to_string(id) + " not found";
        return T2I_ERR_NOT_FOUND;
    }
    if (v == IdTable::kEvicted) {
        err_ = "view: id " + std::to_string(id) + " was evicted";
        return T2I_ERR_EVICTED;
    }
    Object* o = reinterpret_cast<Object*>(v);
    for (size_t j = 1; j < o->pages.size(); ++j) {
        if (o->pages[j] != o->pages[0] + j) {
            err_ = "view: the object's pages are not consecutive";
            return T2I_ERR_NOT_CONTIGUOUS;
        }
    }
    touch(o);
    flush_touches();
    counters_.views++;
    *out = o;
    return T2I_OK;
}

void Control::rollback_compact() {
    // the free pages and the limit change only in finish_compact: the page
    // tables and the counters are all there is to undo
    for (const Remap& r : last_remap_) {
        page_obj_[r.o->pages[r.idx]] = nullptr;
        r.o->pages[r.idx] = r.old_page;
        page_obj_[r.old_page] = r.o;
        page_idx_[r.old_page] = r.idx;
    }
    last_remap_.clear();
    counters_.pages_moved = last_compact_counters_.pages_moved;
    counters_.bytes_moved = last_compact_counters_.bytes_moved;
}

const Object* Control::find(uint64_t id) const {
    const uintptr_t v = ids_.get(id);
    return v > IdTable::kEvicted ? reinterpret_cast<const Object*>(v) : nullptr;
}

t2i_status Control::put(const t2i_put_desc* descs, uint32_t n, t2i_id* ids, std::vector<const Object*>* created) {
    last_evictions_.clear();
    if (created) created->clear();
    if (n == 0) return T2I_OK;
    if (!descs || !ids) {
        err_ = "put: null descriptor or id array";
        return T2I_ERR_INVALID;
    }
    uint64_t demand = 0;
    std::vector<uint64_t> pinned;
    pinned.reserve(n);
    for (uint32_t i = 0; i < n; ++i) {
        if (descs[i].reserved != 0) {
            err_ = "put: reserved field must be 0";
            return T2I_ERR_INVALID;
        }
    }
    for (uint32_t i = 0; i < n; ++i) {
        const uint64_t np = pages_for(descs[i].nbytes);
        if (np > limit_pages_ || demand + np > limit_pages_) {
            err_ = "put: the batch needs more pages than the store has";
            return T2I_ERR_NOSPACE;
        }
        demand += np;
        pinned.push_back(descs[i].group);
    }
    std::sort(pinned.begin(), pinned.end());
    pinned.erase(std::unique(pinned.begin(), pinned.end()), pinned.end());

    if (demand > free_.size()) {
        uint64_t avail = evictable_pages_;
        for (uint64_t key : pinned) {
            auto it = groups_.find(key);
            if (it != groups_.end()) avail -= it->second->evictable_pages;
        }
        if (free_.size() + avail < demand) {
            err_ = "put: not enough free pages even after evicting every allowed object";
            return T2I_ERR_NOSPACE;
        }
        auto it = recency_.begin();
        while (free_.size() < demand && it != recency_.end()) {
            Group* g = it->second;
            auto next = std::next(it);
            if (!std::binary_search(pinned.begin(), pinned.end(), g->key)) {
                while (free_.size() < demand) {
                    auto v = g->victims.begin();
                    const bool last = std::next(v) == g->victims.end();
                    Object* o = reinterpret_cast<Object*>(ids_.get(v->second));
                    last_evictions_.push_back(o->id);
                    counters_.evictions++;
                    release(o, true);  // may drop g once its last victim is gone
                    if (last) break;
                }
            }
            it = next;
        }
    }

    for (uint32_t i = 0; i < n; ++i) {
        const t2i_put_desc& d = descs[i];
        Object* o = new Object();
        o->id = next_id_++;
        o->nbytes = d.nbytes;
        o->dtype_tag = d.dtype_tag;
        o->order = d.order;
        o->evictable = d.evictable != 0;
        o->consumers_left = d.consumers;
        o->group = group_for(d.group);
        const uint64_t np = pages_for(d.nbytes);
        free_.take(np, &o->pages);
        own(o);
        used_pages_ += np;
        Group* g = o->group;
        g->n_objects++;
        if (o->evictable) {
            g->victims.insert({o->order, o->id});
            g->evictable_pages += np;
            evictable_pages_ += np;
        }
        o->live_index = live_.size();
        live_.push_back(o);
        ids_.set(o->id, reinterpret_cast<uintptr_t>(o), next_id_);
        touch(o);
        counters_.puts++;
        counters_.bytes_put += d.nbytes;
        ids[i] = o->id;
        if (created) created->push_back(o);
    }
    flush_touches();
    return T2I_OK;
}

void Control::rollback_put(const t2i_id* ids, uint32_t n) {
    // last object first, each object's pages in reverse: the exact undo of
    // the pops that placed them
    for (uint32_t i = n; i-- > 0;) {
        Object* o = const_cast<Object*>(find(ids[i]));
        if (!o) continue;
        counters_.puts--;
        counters_.bytes_put -= o->nbytes;
        const uint64_t np = o->pages.size();
        disown(o);
        free_.give(o->pages, /*undo=*/true);
        used_pages_ -= np;
        Group* g = o->group;
        g->n_objects--;
        if (o->evictable) {
            g->victims.erase({o->order, o->id});
            g->evictable_pages -= np;
            evictable_pages_ -= np;
            if (g->victims.empty() && g->rec_key) {
                recency_.erase({g->rec_key, g});
                g->rec_key = 0;
            }
        }
        const size_t li = o->live_index;
        live_[li] = live_.back();
        live_[li]->live_index = li;
        live_.pop_back();
        ids_.clear(o->id, next_id_);
        if (o->id + 1 == next_id_) next_id_ = o->id;  // never handed out: issue again
        delete o;
        maybe_drop_group(g);
    }
}

void Control::account_get(const t2i_id* ids, uint32_t n, size_t stride) {
    const char* base = reinterpret_cast<const char*>(ids);
    for (uint32_t i = 0; i < n; ++i) {
        const t2i_id id = *reinterpret_cast<const t2i_id*>(base + i * stride);
        Object* o = reinterpret_cast<Object*>(ids_.get(id));
        touch(o);
        counters_.gets++;
        counters_.bytes_got += o->nbytes;
        if (o->consumers_left > 0 && --o->consumers_left == 0) pending_release_.push_back(o);
    }
    flush_touches();
}

t2i_status Control::get(const t2i_get_desc* descs, uint32_t n, t2i_status* per_item,
                        std::vector<const Object*>* objs, bool defer_release) {
    if (objs) objs->assign(n, nullptr);
    if (n == 0) return T2I_OK;
    if (!descs) {
        err_ = "get: null descriptor array";
        return T2I_ERR_INVALID;
    }
    t2i_status first = T2I_OK;
    uint32_t first_i = 0;
    for (uint32_t i = 0; i < n; ++i) {
        const t2i_get_desc& d = descs[i];
        t2i_status st = T2I_OK;
        if (d.cast > 1 || d.reserved != 0) {
            st = T2I_ERR_INVALID;
        } else {
            const uintptr_t v = ids_.get(d.id);
            if (v == 0) {
                st = T2I_ERR_NOT_FOUND;
            } else if (v == IdTable::kEvicted) {
                st = T2I_ERR_EVICTED;
                counters_.misses++;
            } else {
                const Object* o = reinterpret_cast<const Object*>(v);
                if (d.cast == 1 && (o->nbytes % 4) != 0) st = T2I_ERR_INVALID;
                if (objs) (*objs)[i] = o;
            }
        }
        if (per_item) per_item[i] = st;
        if (st != T2I_OK && first == T2I_OK) {
            first = st;
            first_i = i;
        }
    }
    if (first != T2I_OK) {
        static const char* what[] = {"ok", "invalid descriptor (cast needs nbytes % 4 == 0)", "no space",
                                     "id not found", "id was evicted", "cuda"};
        err_ = "get: item " + std::to_string(first_i) + ": " + what[first];
        return first;
    }
    if (objs) {
        for (uint32_t i = 0; i < n; ++i) (*objs)[i] = reinterpret_cast<const Object*>(ids_.get(descs[i].id));
    }
    account_get(&descs[0].id, n, sizeof(t2i_get_desc));
    if (!defer_release) release_pending();
    return T2I_OK;
}

void Control::release_pending() {
    for (Object* o : pending_release_) {
        counters_.reclaimed++;
        release(o, false);
    }
    pending_release_.clear();
}

t2i_status Control::free(const t2i_id* ids, uint32_t n) {
    if (n == 0) return T2I_OK;
    if (!ids) {
        err_ = "free: null id array";
        return T2I_ERR_INVALID;
    }
    std::vector<uint64_t> sorted(ids, ids + n);
    std::sort(sorted.begin(), sorted.end());
    if (std::adjacent_find(sorted.begin(), sorted.end()) != sorted.end()) {
        err_ = "free: an id appears twice";
        return T2I_ERR_INVALID;
    }
    for (uint32_t i = 0; i < n; ++i) {
        if (ids_.get(ids[i]) == 0) {
            err_ = "free: id " + std::to_string(ids[i]) + " not found";
            return T2I_ERR_NOT_FOUND;
        }
    }
    for (uint32_t i = 0; i < n; ++i) {
        const uintptr_t v = ids_.get(ids[i]);
        if (v == IdTable::kEvicted)
            ids_.clear(ids[i], next_id_);
        else
            release(reinterpret_cast<Object*>(v), false);
    }
    return T2I_OK;
}

t2i_status Control::compact(uint64_t limit_bytes, std::vector<t2i_move>* moves) {
    const t2i_status st = plan_compact(limit_bytes, moves);
    if (st == T2I_OK) finish_compact();
    return st;
}

t2i_status Control::plan_compact(uint64_t limit_bytes, std::vector<t2i_move>* moves) {
    moves->clear();
    const t2i_status st = begin_compact(limit_bytes);
    if (st != T2I_OK) return st;
    moves->reserve(last_remap_.capacity());
    plan_more(SIZE_MAX, moves);
    return T2I_OK;
}

t2i_status Control::begin_compact(uint64_t limit_bytes) {
    if (limit_bytes % P_ != 0 || limit_bytes / P_ > total_pages_) {
        err_ = "compact: the limit must be a multiple of the page size and at most the pool";
        return T2I_ERR_INVALID;
    }
    const uint64_t limit = limit_bytes / P_;
    if (used_pages_ > limit) {
        err_ = "compact: more pages are in use than the limit holds";
        return T2I_ERR_NOSPACE;
    }
    last_remap_.clear();
    last_remap_.reserve(live_pages_at_or_above(limit));
    last_compact_counters_ = counters_;
    planned_limit_ = limit;
    plan_p_ = limit;
    plan_scan_ = 0;
    return T2I_OK;
}

bool Control::plan_more(size_t max, std::vector<t2i_move>* moves) {
    // live pages at or above the limit, ascending (pages at or above the
    // current limit are all free), each to the lowest free page below it
    size_t n = 0;
    uint64_t moved_bytes = 0;
    for (; plan_p_ < limit_pages_ && n < max; ++plan_p_) {
        const uint64_t p = plan_p_;
        Object* o = page_obj_[p];
        if (!o) continue;
        while (page_obj_[plan_scan_]) ++plan_scan_;  // used_pages_ <= limit guarantees a free page
        const uint32_t dst = static_cast<uint32_t>(plan_scan_);
        const uint32_t idx = page_idx_[p];
        const uint64_t valid = std::min<uint64_t>(P_, o->nbytes - uint64_t(idx) * P_);
        o->pages[idx] = dst;
        page_obj_[dst] = o;
        page_idx_[dst] = idx;
        page_obj_[p] = nullptr;
        last_remap_.push_back({o, idx, static_cast<uint32_t>(p)});
        moves->push_back({static_cast<uint32_t>(p), dst, valid});
        moved_bytes += valid;
        ++n;
    }
    counters_.pages_moved += n;
    counters_.bytes_moved += moved_bytes;
    // more to plan if a live page may remain at or above the limit
    for (; plan_p_ < limit_pages_; ++plan_p_)
        if (page_obj_[plan_p_]) return true;
    return false;
}

void Control::finish_compact() {
    free_.rebuild(planned_limit_, [this](uint64_t q) { return page_obj_[q] != nullptr; });
    limit_pages_ = planned_limit_;
}

void Control::stats(t2i_stats* out) const {
    *out = counters_;
    out->total_pages = total_pages_;
    out->limit_pages = limit_pages_;
    out->used_pages = used_pages_;
    out->free_pages = free_.size();
    out->live_objects = live_.size();
}

}  // namespace t2i
