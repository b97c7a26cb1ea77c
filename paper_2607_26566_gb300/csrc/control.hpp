// Host control core of the paged tensor store: page allocator, object
// directory, per-group LRU and compaction planner. Plain C++17, no CUDA.
//
// The paper's data plane keeps a fixed-size arena per executor managed by a
// buddy allocator (§5.2) and a Layer Lookup Table that maps a model's logical
// layers to tensor objects and their physical memory (§5.3, "How does it
// work?"). Here the arena is cut into fixed pages and the lookup table is the
// directory id -> {size, tags, page list}. Eviction follows §5.3: least
// recently used model first, its layers in reverse order, until the demand is
// met. Where the paper is silent the rules are:
//   - placement policy 0 (LIFO): free pages form a stack; page 0 pops first
//     on a new store; a put pops its pages one at a time, objects in
//     descriptor order; a free pushes an object's pages back in page-list
//     order;
//   - placement policy 1 (extent): free pages form a set of runs; an object
//     of k pages takes the lowest-numbered run of k consecutive free pages,
//     else the k lowest-numbered free pages (objects stay contiguous, so they
//     can be used in place);
//   - ids are 1, 2, 3, ... in descriptor order and never reused;
//   - recency is per group, stamped once per object put or got, in
//     descriptor order; victims: least recent group first, then the highest
//     `order`, then the highest id; groups named by the put are exempt, so are
//     non-evictable objects; a put that cannot be satisfied evicts nothing;
//   - an object put with k > 0 consumers is freed after its k-th successful
//     get item (§5.3: reclaimed once no downstream consumer needs it); the
//     objects a get brings to zero are freed at the end of that get, in the
//     order of the items that brought them there;
//   - compaction to `limit` pages moves the live pages numbered >= limit, in
//     ascending order, to the lowest free pages below limit, then rebuilds the
//     free stack from the free pages below limit so the lowest pops first.
#pragma once

#include <cstdint>
#include <map>
#include <memory>
#include <mutex>
#include <set>
#include <string>
#include <unordered_map>
#include <utility>
#include <vector>

#include "t2istore.h"

namespace t2i {

struct Group;

struct Object {
    uint64_t id = 0;
    uint64_t nbytes = 0;
    uint32_t dtype_tag = 0;
    uint32_t order = 0;
    bool evictable = false;
    uint32_t consumers_left = 0;    // gets still expected before the store frees it (0 = none)
    Group* group = nullptr;
    size_t live_index = 0;          // position in Control::live_
    std::vector<uint32_t> pages;    // page list, in object byte order
};

struct Group {
    uint64_t key = 0;
    uint64_t last = 0;              // recency stamp of the last touch
    uint64_t rec_key = 0;           // stamp under which it sits in the recency set; 0 = absent
    uint64_t n_objects = 0;
    uint64_t evictable_pages = 0;
    uint64_t epoch = 0;             // batch marker for de-duplicating touches
    // evictable objects, eviction order first: highest order, then highest id
    std::set<std::pair<uint32_t, uint64_t>, std::greater<std::pair<uint32_t, uint64_t>>> victims;
};

// The free pages under either placement policy.
class FreePages {
  public:
    FreePages(uint64_t total_pages, uint32_t policy);
    uint64_t size() const { return count_; }
    uint32_t policy() const { return policy_; }
    // k pages for one object, in page-list order (requires k <= size())
    void take(uint64_t k, std::vector<uint32_t>* out);
    // an object's pages back, in page-list order (or, undoing a take, in
    // reverse, which restores a LIFO stack exactly)
    void give(const std::vector<uint32_t>& pages, bool undo = false);
    // after a compaction: every page below limit for which used(p) is false
    template <class Used>
    void rebuild(uint64_t limit, Used used) {
        stack_.clear();
        runs_.clear();
        count_ = 0;
        if (policy_ == 0) {
            for (uint64_t p = limit; p-- > 0;)
                if (!used(p)) stack_.push_back(static_cast<uint32_t>(p));
            count_ = stack_.size();
            return;
        }
        uint64_t p = 0;
        while (p < limit) {
            if (used(p)) {
                ++p;
                continue;
            }
            const uint64_t start = p;
            while (p < limit && !used(p)) ++p;
            runs_.emplace_hint(runs_.end(), uint32_t(start), uint32_t(p - start));
            count_ += p - start;
        }
    }
    // policy 0: the stack from bottom to top; policy 1: ascending
    std::vector<uint32_t> list() const;

  private:
    void insert_page(uint32_t p);
    uint32_t policy_;
    uint64_t count_ = 0;
    std::vector<uint32_t> stack_;          // policy 0; back() is the top
    std::map<uint32_t, uint32_t> runs_;    // policy 1: first page -> run length
};

// id -> object, or the "evicted" tombstone; two-level table over the dense
// id space whose leaves are released once every id in them is gone.
class IdTable {
  public:
    static constexpr uintptr_t kEvicted = 1;
    uintptr_t get(uint64_t id) const;
    void set(uint64_t id, uintptr_t v, uint64_t next_id);
    void clear(uint64_t id, uint64_t next_id);

  private:
    static constexpr int kLeafBits = 12;
    static constexpr uint64_t kLeafSize = uint64_t(1) << kLeafBits;
    struct Leaf {
        uintptr_t slot[kLeafSize] = {};
        uint64_t used = 0;
    };
    std::vector<std::unique_ptr<Leaf>> leaves_;
};


class Control {
  public:
    Control(uint64_t total_pages, uint64_t page_bytes, uint32_t policy = 0);
    ~Control();
    Control(const Control&) = delete;
    Control& operator=(const Control&) = delete;

    uint64_t page_bytes() const { return P_; }
    uint64_t total_pages() const { return total_pages_; }
    uint64_t limit_pages() const { return limit_pages_; }
    uint64_t used_pages() const { return used_pages_; }
    uint64_t pages_for(uint64_t nbytes) const { return nbytes / P_ + (nbytes % P_ != 0); }

    // put: validates, evicts, allocates and commits. On success ids[i] and
    // created[i] (if non-null) describe descs[i].
    t2i_status put(const t2i_put_desc* descs, uint32_t n, t2i_id* ids, std::vector<const Object*>* created);
    // Undo the put of freshly created objects (after a failed launch):
    // pages, ids and counters return to their state before the put;
    // evictions it made and recency stamps stand.
    void rollback_put(const t2i_id* ids, uint32_t n);
    // The accounting half of a get (recency stamps, consumer counts) for
    // items already validated; objects consumed to zero wait for
    // release_pending(). Called after the get's copies are enqueued.
    void account_get(const t2i_id* ids, uint32_t n, size_t stride);
    // get: validates every item (per_item nullable), then stamps recency and
    // counts consumers. objs[i] receives the object of descs[i] on success.
    // dst fields are not looked at here. Objects whose last consumer this was
    // are freed at the end of the call, or, with defer_release, kept until
    // release_pending() (the store frees them after packing its launches).
    t2i_status get(const t2i_get_desc* descs, uint32_t n, t2i_status* per_item, std::vector<const Object*>* objs,
                   bool defer_release = false);
    void release_pending();
    t2i_status free(const t2i_id* ids, uint32_t n);
    // compact: plans, remaps and returns the moves (always filled).
    t2i_status compact(uint64_t limit_bytes, std::vector<t2i_move>* moves);
    // The same in steps, so that moves can run while the rest is planned
    // and the free pages are rebuilt while the moves run:
    //   begin_compact validates the limit and starts a plan;
    //   plan_more remaps up to `max` more live pages and appends their moves
    //     (true while live pages remain at or above the limit);
    //   finish_compact (after a complete plan, before any other call)
    //     rebuilds the free pages and applies the new limit;
    //   rollback_compact (instead of finish_compact, after a failed launch)
    //     puts every page list planned since begin_compact back.
    // plan_compact is begin_compact + plan_more until done.
    t2i_status plan_compact(uint64_t limit_bytes, std::vector<t2i_move>* moves);
    t2i_status begin_compact(uint64_t limit_bytes);
    bool plan_more(size_t max, std::vector<t2i_move>* moves);
    void finish_compact();
    void rollback_compact();

    uint64_t live_pages_at_or_above(uint64_t limit) const;
    const Object* find(uint64_t id) const;
    bool is_evicted(uint64_t id) const { return ids_.get(id) == IdTable::kEvicted; }
    std::vector<uint32_t> free_list() const { return free_.list(); }
    // A view: the object's first page if its pages are consecutive (stamps
    // recency like a get, counts no consumer). NOT_FOUND / EVICTED /
    // NOT_CONTIGUOUS otherwise.
    t2i_status view(uint64_t id, const Object** out);
    const std::vector<t2i_id>& last_evictions() const { return last_evictions_; }
    void stats(t2i_stats* out) const;
    t2i_stats& counters() { return counters_; }

    const std::string& error() const { return err_; }
    void set_error(std::string e) { err_ = std::move(e); }

  private:
    Group* group_for(uint64_t key);
    void maybe_drop_group(Group* g);
    void touch(Object* o);
    void flush_touches();
    void release(Object* o, bool evicted);

    uint64_t P_;
    uint64_t total_pages_;
    uint64_t limit_pages_;
    uint64_t used_pages_ = 0;
    uint64_t evictable_pages_ = 0;
    uint64_t next_id_ = 1;
    uint64_t clock_ = 0;
    uint64_t epoch_ = 1;            // groups start at epoch 0, so the first batch is new
    FreePages free_;
    IdTable ids_;
    std::vector<Object*> live_;
    std::unordered_map<uint64_t, std::unique_ptr<Group>> groups_;
    std::set<std::pair<uint64_t, Group*>> recency_;   // groups holding evictable objects
    std::vector<Group*> touched_;
    std::vector<t2i_id> last_evictions_;
    std::vector<Object*> pending_release_;   // consumed to zero by the last get
    struct Remap {
        Object* o;
        uint32_t idx;
        uint32_t old_page;
    };
    // page -> (object, index in its page list); null for a free page. Kept
    // on every put, release and move, so a compaction visits only the pages
    // at or above its limit.
    void own(const Object* o);
    void disown(const Object* o);
    std::vector<Object*> page_obj_;
    std::vector<uint32_t> page_idx_;
    std::vector<Remap> last_remap_;          // the last compaction, for rollback_compact
    uint64_t planned_limit_ = 0;
    uint64_t plan_p_ = 0;      // next page at or above the limit to look at
    uint64_t plan_scan_ = 0;   // lowest page below the limit that may be free
    t2i_stats last_compact_counters_{};
    t2i_stats counters_{};
    std::string err_;
};

}  // namespace t2i

// The opaque C handle around a control core.
struct t2i_ctl {
    t2i::Control* core;
    bool owned;                 // false: borrowed from a store (queries only)
    std::mutex* mu = nullptr;   // the store's lock, for queries of a borrowed core
};
