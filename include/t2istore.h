/*
 * t2istore.h -- a paged tensor store in the spare HBM of one GPU (GB300, sm_103a).
 *
 * The store is the GPU-resident data plane of a serverless text-to-image
 * system (arxiv 2607.26566, §5): model functions put intermediate tensors
 * (text embeddings, latents, decoded images) and cached model or adapter
 * weights into it, and get them back into their own buffers. The pool is one
 * block of device memory that the caller owns (typically a PyTorch
 * allocation); the store divides it into fixed pages and keeps the page
 * tables, the object directory and the LRU order on the host. Bytes move only
 * through the library's own CUDA kernels (and, for host sources on request,
 * the copy engine), stream-ordered on the caller's stream.
 *
 * Conventions shared by every call:
 *  - Every call returns a t2i_status; nothing aborts or prints.
 *  - The caller owns the pool, every source and destination buffer and every
 *    descriptor array. Descriptor arrays are read only during the call.
 *  - Calls are asynchronous like cudaMemcpyAsync: a put's sources must stay
 *    unchanged until the stream has passed the put; a get's destinations hold
 *    the bytes once the stream has passed the get.
 *  - Calls are ordered by the pages they share, on the GPU: a get waits for
 *    the call that wrote each page it reads; a put waits for the calls that
 *    last wrote or read each page it reuses (pages of freed or evicted
 *    objects); a compaction waits for both. Calls on one stream are ordered
 *    by the stream; across streams the store inserts event waits only where
 *    pages are shared, so independent calls on different streams overlap.
 *    Streams given to a store must stay valid until the store is destroyed.
 *  - Pointers are checked on the host before any launch (when
 *    check_pointers = 1): a pointer the CUDA driver does not know, on another
 *    device, or a range that runs past its allocation returns
 *    T2I_ERR_INVALID, so a bad argument never reaches the GPU.
 *  - A store may be used from several host threads; calls are serialised by
 *    a lock inside the store.
 */
#ifndef T2ISTORE_H
#define T2ISTORE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
typedef int32_t t2i_status;
#define T2I_OK 0
#define T2I_ERR_INVALID 1   /* bad argument; nothing changed                     */
#define T2I_ERR_NOSPACE 2   /* not enough pages even after eviction; nothing changed */
#define T2I_ERR_NOT_FOUND 3 /* id never issued, or already freed                 */
#define T2I_ERR_EVICTED 4   /* id was evicted to make room (put it again)        */
#define T2I_ERR_CUDA 5      /* a CUDA call failed; see t2i_last_error            */
#define T2I_ERR_NOT_CONTIGUOUS 6 /* t2i_view: the object's pages are not consecutive */

/* Object ids: 1, 2, 3, ... in descriptor order, never reused; 0 is never an id. */
typedef uint64_t t2i_id;

typedef struct t2i_store t2i_store; /* opaque: a store over one pool          */
typedef struct t2i_ctl t2i_ctl;     /* opaque: the host control core alone     */

/* ---- configuration ------------------------------------------------------- */
typedef struct t2i_store_config {
    uint64_t pool_bytes;     /* bytes at pool_dev; the store uses floor(pool_bytes / page_bytes) pages */
    uint64_t page_bytes;     /* power of two, 256 B ... 1 GiB                                   */
    uint32_t h2d_mode;       /* puts from host memory: 0 = the put kernel reads pinned host memory
                                directly (zero-copy over the host link); 1 = one copy-engine
                                cudaMemcpyAsync per run of consecutive pages. Pageable (not
                                pinned) host memory always takes the copy engine.               */
    uint32_t check_pointers; /* 1 = check every user pointer range with the driver before launch
                                (recommended); 0 = trust the caller                             */
    uint32_t alloc_policy;   /* page placement: 0 = LIFO stack of free pages (page 0 first on a
                                new store; a free pushes pages back in page-list order);
                                1 = extent: the lowest run of enough consecutive free pages,
                                else the lowest free pages (objects stay contiguous and can be
                                used in place, see t2i_view)                                  */
    uint32_t d2h_mode;       /* gets into pinned host memory: 0 = the get kernel writes host memory
                                directly (zero-copy over the host link); 1 = items without the
                                cast take one copy-engine cudaMemcpyAsync per run of consecutive
                                pages, which leaves the SMs free for work in the other direction
                                (a put from host on another stream); items with the cast always
                                run in the kernel. Needs check_pointers = 1 (the store must see
                                that a destination is host memory).                           */
} t2i_store_config;

/* ---- put ------------------------------------------------------------------
 * One object to store. Ids are returned in descriptor order.
 * §5.2: a producer writes its output into the store; §5.3: cached weights are
 * evictable, least recently used model first, higher layers first.        */
typedef struct t2i_put_desc {
    const void* src;      /* nbytes to copy: device memory of the store's device, or host memory
                             when src_is_host = 1. NULL reserves pages and copies nothing: the
                             object takes capacity and its bytes are undefined.              */
    uint64_t nbytes;      /* object size; 0 is allowed (no pages)                            */
    uint32_t src_is_host; /* 1 = src is host memory (pinned or pageable)                      */
    uint32_t dtype_tag;   /* opaque tag kept in the directory                                 */
    uint64_t group;       /* LRU group: one model or one adapter set                          */
    uint32_t order;       /* layer index inside the group; the highest is evicted first        */
    uint32_t evictable;   /* 1 = cached weights (may be evicted); 0 = intermediate (never)      */
    uint32_t consumers;   /* > 0: the object is freed by the store after this many successful
                             gets of it (each occurrence in a get batch counts once): an
                             intermediate reclaimed when no downstream consumer needs it any
                             more (§5.3). 0 = freed only by t2i_free (or evicted).           */
    uint32_t reserved;    /* must be 0                                                        */
} t2i_put_desc;

/* ---- get ------------------------------------------------------------------
 * Copies an object into a consumer buffer (§5.2: the consumer pulls a
 * produced tensor into its own memory), optionally casting fp32 -> bf16.  */
typedef struct t2i_get_desc {
    t2i_id id;
    void* dst;            /* device memory of the store's device, or pinned host memory (written
                             by the kernel, or by the copy engine under d2h_mode = 1)         */
    uint64_t dst_bytes;   /* capacity at dst: >= nbytes, or >= nbytes / 2 with cast = 1       */
    uint32_t cast;        /* 0 = bytes as stored; 1 = the object is little-endian fp32 and dst
                             receives bf16, round to nearest even (NaN -> quiet NaN with the
                             sign kept: 0x7FC0 | sign << 15); needs nbytes % 4 == 0 and a
                             2-byte aligned dst                                               */
    uint32_t reserved;    /* must be 0                                                        */
} t2i_get_desc;

/* ---- compaction moves ------------------------------------------------------ */
typedef struct t2i_move {
    uint32_t src_page;    /* live page at or above the limit                                  */
    uint32_t dst_page;    /* lowest free page below the limit                                 */
    uint64_t valid_bytes; /* bytes of the object in that page (only these are copied)          */
} t2i_move;

/* ---- introspection ----------------------------------------------------------- */
typedef struct t2i_stats {
    uint64_t total_pages, limit_pages, used_pages, free_pages, live_objects;
    uint64_t bytes_put, bytes_got, puts, gets, misses, evictions;
    uint64_t pages_moved, bytes_moved;
    uint64_t launches;   /* kernels launched by the store                                    */
    uint64_t h2d_copies; /* copy-engine copies issued for host sources                        */
    uint64_t reclaimed;  /* objects freed by the store after their last declared consumer    */
    uint64_t views;      /* successful t2i_view calls                                         */
    uint64_t d2h_copies; /* copy-engine copies issued for host destinations (d2h_mode = 1)       */
} t2i_stats;

typedef struct t2i_object_info {
    uint64_t nbytes;
    uint64_t group;
    uint32_t dtype_tag;
    uint32_t order;
    uint32_t evictable;
    uint32_t n_pages;
    uint32_t consumers_left; /* gets still expected before the store frees it (0 = none)   */
    uint32_t reserved;
} t2i_object_info;

/* =========================================================================
 * Store: the pool, the host control core and the CUDA kernels.
 * ========================================================================= */

/* Creates a store over [pool_dev, pool_dev + pool_bytes) on CUDA device
 * `device`. pool_dev must be device memory of that device, 256-byte aligned.
 * The store never frees pool_dev. It allocates 2 KiB of device memory of its
 * own (cudaMalloc, cleared on a private stream before this returns): the
 * chunk counters through which the CTAs of a large launch share out its
 * work, one for each of the first 64 streams the store is given (launches
 * on later streams split their work statically). t2i_store_destroy frees it.
 * Errors: INVALID (geometry, pointer), CUDA (device query or allocation
 * failed). On error *out is NULL and t2i_last_error(NULL) describes it.     */
t2i_status t2i_store_create(void* pool_dev, const t2i_store_config* cfg, int device, t2i_store** out);

/* Frees the store's host state, events and chunk counters after waiting for
 * the work of every stream it was given.
 * Does not free the pool. NULL is accepted.                                 */
t2i_status t2i_store_destroy(t2i_store* store);

/* Stores n objects (paper §5.2 "producer writes its output", §5.3 eviction).
 * All-or-nothing: pages for the whole batch are taken from the free stack,
 * evicting least-recently-used evictable objects of groups not named in this
 * batch (highest `order`, then highest id, first) until the batch fits.
 * Returns NOSPACE (and evicts nothing) if even that is not enough, INVALID
 * for a bad descriptor; out_ids[i] receives the id of descs[i] (n ids).
 * The copy is one kernel launch per batch (more only when the descriptors
 * exceed one launch's parameter space). On CUDA the batch is not stored
 * (pages, ids and counters as before the call); evictions it made stand.     */
t2i_status t2i_put_batch(t2i_store* store, const t2i_put_desc* descs, uint32_t n, t2i_id* out_ids,
                         void* cuda_stream);

/* Copies n objects into their destinations (paper §5.2 "consumer pulls").
 * The copies are one kernel launch per batch (more only when the
 * descriptors exceed one launch's parameter space), plus, under d2h_mode =
 * 1, one copy-engine copy per run of consecutive pages of each item without
 * the cast whose destination is pinned host memory. Every item is validated first; per_item (nullable, n entries) receives
 * OK / NOT_FOUND / EVICTED / INVALID per item. If any item fails, the call
 * returns the first failing status in descriptor order and writes nothing.
 * The same id may appear more than once. Objects reserved with src = NULL
 * return whatever their pages hold. Objects put with consumers > 0 count one
 * consumer per successful item; those that reach zero are freed once the
 * call's copies are enqueued (stream order keeps their pages intact until
 * the copies have run).                                                      */
t2i_status t2i_get_batch(t2i_store* store, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item,
                         void* cuda_stream);

/* As t2i_get_batch, but the copies start only after `wait_event` (a
 * cudaEvent_t recorded by the producer, e.g. on another stream) has
 * completed: the consumer issues the fetch where its execution needs the
 * tensor, and the store orders it after the producer (§5.2, callback-based
 * fetching). wait_event = NULL behaves as t2i_get_batch. The wait is a
 * cudaStreamWaitEvent on cuda_stream: the host never blocks.               */
t2i_status t2i_get_batch_after(t2i_store* store, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item,
                               void* cuda_stream, void* wait_event);

/* A zero-copy view of one object (§5.3: the paper wraps arena memory as a
 * tensor with torch::from_blob and rebinds the model's parameters to it).
 * If the object's pages are consecutive, *dev_ptr = the device address of
 * its first byte and *nbytes = its size; else T2I_ERR_NOT_CONTIGUOUS
 * (alloc_policy 1 keeps objects contiguous whenever a long enough run of
 * free pages exists). cuda_stream becomes ordered after the call that wrote
 * the object, so work enqueued on it afterwards may read the bytes in place.
 * The view stamps recency like a get but counts no consumer. The address is
 * valid until the object is freed, evicted or moved by a compaction; a later
 * put that reuses its pages waits for everything enqueued on cuda_stream up
 * to that put. Reads through the view must not outlive those events.
 * NOT_FOUND / EVICTED for unknown or evicted ids.                             */
t2i_status t2i_view(t2i_store* store, t2i_id id, void* cuda_stream, void** dev_ptr, uint64_t* nbytes);

/* Pulls n objects of the producer's store `src` into the consumer's store
 * `dst` (§5.2: the consumer allocates a block in its own arena and pulls the
 * producer's bytes into it), page to page on the GPU, without a staging
 * buffer. out_ids[i] receives the new id in dst of src_ids[i]; the new
 * objects are intermediates (evictable = 0, group 0, order 0) with the
 * source's dtype_tag and `consumers`. The sources are read like a get
 * (recency stamped, one consumer counted). Every source id is checked first
 * (per_item, nullable: OK / NOT_FOUND / EVICTED); NOSPACE in dst changes
 * nothing. Both stores must be distinct, on the same device and have the
 * same page size (INVALID otherwise). The copy is ordered after the
 * producer's write of the source pages and after the consumer store's
 * earlier users of the new pages.                                            */
t2i_status t2i_pull(t2i_store* dst, t2i_store* src, const t2i_id* src_ids, uint32_t n, uint32_t consumers,
                    t2i_id* out_ids, t2i_status* per_item, void* cuda_stream);

/* One object laid out in pages of a pool that the pulling store does not
 * own (t2i_pull_pages).                                                     */
typedef struct {
    uint64_t nbytes;        /* the object's size in bytes                      */
    const uint32_t* pages;  /* its page list in byte order: page indices into
                               the source pool (host array, read during the
                               call)                                           */
    uint32_t n_pages;       /* ceil(nbytes / page_bytes)                       */
    uint32_t dtype_tag;     /* kept on the new object                          */
} t2i_paged_object;

/* Pulls n objects laid out in pages of another pool into `dst` (§5.2: the
 * consumer allocates a block in its own arena and pulls the producer's bytes
 * into it), page to page on the GPU. The source pool is usually a producer
 * store's pool in another process on the same GPU, mapped into this one with
 * cudaIpcOpenMemHandle (torch shares CUDA tensors between processes this
 * way); the page lists come from the producer (t2i_ctl_object).
 * src_pool: device memory of dst's device covering src_pool_bytes, laid out
 * in pages of dst's page size, not overlapping dst's pool. Each object's
 * pages must lie in the source pool and number ceil(nbytes / page_bytes).
 * out_ids[i] receives the new id of objs[i]: an intermediate (evictable = 0,
 * group 0, order 0) with objs[i].dtype_tag and `consumers`. NOSPACE in dst
 * changes nothing. The source is not a store of this process: the caller
 * orders its bytes before this call (the producer synchronizes, or its event
 * is waited on), and keeps them until the copy has run on cuda_stream. The
 * copy is ordered after dst's earlier users of the new pages.               */
t2i_status t2i_pull_pages(t2i_store* dst, const void* src_pool, uint64_t src_pool_bytes,
                          const t2i_paged_object* objs, uint32_t n, uint32_t consumers, t2i_id* out_ids,
                          void* cuda_stream);

/* Returns the pages of n objects to the free stack (paper §5.3: data is
 * reclaimed when no consumer needs it). Host-only: stream order makes reuse
 * safe. A repeated id is INVALID; an unknown id is NOT_FOUND; in both cases
 * nothing is freed. An evicted id is accepted and forgotten.                 */
t2i_status t2i_free(t2i_store* store, const t2i_id* ids, uint32_t n);

/* Shrinks (or regrows) the usable pool to limit_bytes (a multiple of
 * page_bytes, at most the pool): live pages at or above the limit move, in
 * ascending order, to the lowest free pages below it (one kernel; only the
 * valid bytes of each page are copied) and the page tables are remapped.
 * NOSPACE if more than limit_bytes / page_bytes pages are in use. After the
 * stream has passed this call, [pool + limit_bytes, pool + pool_bytes) is
 * not touched by the store until a larger limit is set. pages_moved is
 * nullable. (No counterpart in the paper: it answers the fixed-size arena
 * problem of §5.3.)                                                          */
t2i_status t2i_compact(t2i_store* store, uint64_t limit_bytes, void* cuda_stream, uint64_t* pages_moved);

t2i_status t2i_store_stats(const t2i_store* store, t2i_stats* out);

/* The store's host control core (read-only: the t2i_ctl_* queries below
 * accept it; the mutating t2i_ctl_* calls refuse it with INVALID).          */
const t2i_ctl* t2i_store_ctl(const t2i_store* store);

/* Message of the last failed call on this store (or, for NULL, of the last
 * failed call on this thread that has no store: t2i_store_create,
 * t2i_ctl_create, t2i_gather_noalloc, the prefix calls). Never NULL. A
 * store's message lives inside the store: it stays valid until the next
 * call on that store, from any thread, or its destruction; copy it out
 * before then.                                                              */
const char* t2i_last_error(const t2i_store* store);

/* =========================================================================
 * Control core: page allocator, directory, LRU and compaction planner,
 * without device memory. The same code runs inside every store; alone it
 * plans layouts on the host and is what the host-only tests drive.
 * ========================================================================= */

/* total_pages <= 2^32 - 1, page_bytes > 0, alloc_policy 0 or 1 (as in
 * t2i_store_config).                                                         */
t2i_status t2i_ctl_create(uint64_t total_pages, uint64_t page_bytes, uint32_t alloc_policy, t2i_ctl** out);
t2i_status t2i_ctl_destroy(t2i_ctl* ctl);
/* As t2i_put_batch, without copying (src and src_is_host are ignored).      */
t2i_status t2i_ctl_put(t2i_ctl* ctl, const t2i_put_desc* descs, uint32_t n, t2i_id* out_ids);
/* As t2i_get_batch's validation and LRU update (dst/dst_bytes ignored).     */
t2i_status t2i_ctl_get(t2i_ctl* ctl, const t2i_get_desc* descs, uint32_t n, t2i_status* per_item);
t2i_status t2i_ctl_free(t2i_ctl* ctl, const t2i_id* ids, uint32_t n);
/* As t2i_compact's planning and remap. moves (nullable) receives the moves
 * in order if cap is large enough; otherwise INVALID with *n_moves set to
 * the number needed and nothing changed.                                    */
t2i_status t2i_ctl_compact(t2i_ctl* ctl, uint64_t limit_bytes, t2i_move* moves, uint64_t cap, uint64_t* n_moves);

/* Queries (accept a store's control core). pages receives up to cap page
 * numbers of the object in page-list order; info->n_pages is the full count. */
t2i_status t2i_ctl_object(const t2i_ctl* ctl, t2i_id id, t2i_object_info* info, uint32_t* pages, uint64_t cap);
/* The free pages: policy 0, the stack from bottom to top (the top pops
 * first); policy 1, ascending. *n = their number.                            */
t2i_status t2i_ctl_free_pages(const t2i_ctl* ctl, uint32_t* out, uint64_t cap, uint64_t* n);
/* Ids evicted by the last put, in eviction order; *n = their number.         */
t2i_status t2i_ctl_last_evictions(const t2i_ctl* ctl, t2i_id* out, uint64_t cap, uint64_t* n);
t2i_status t2i_ctl_stats(const t2i_ctl* ctl, t2i_stats* out);
const char* t2i_ctl_last_error(const t2i_ctl* ctl);

/* Testing support: the countdown-th kernel launch of this store from now
 * reports T2I_ERR_CUDA without being issued (0 cancels). It exercises the
 * store's recovery on the host -- a put is rolled back (pages, ids and
 * counters as before it; evictions stand), a get counts nothing, a compaction
 * restores its page tables and limit -- without faulting a GPU.            */
t2i_status t2i_inject_launch_failure(t2i_store* store, uint32_t countdown);

/* =========================================================================
 * Gather without allocation. The paper has no counterpart: this is an extra
 * entry point of the library, not a step of the method.
 * ========================================================================= */

/* Copies one object's pages out of a pool into a contiguous device buffer,
 * with the same bytes and the same optional fp32 -> bf16 RNE cast as a
 * one-item t2i_get_batch, but with no store and without allocating any
 * memory. Its launches are those of a store's chunked get: the cast-capable
 * gather kernel for a 16-byte aligned destination or a cast, the copy-only
 * gather kernel for any other destination.
 *
 * Who needs it: a caller that must not allocate device memory while it
 * moves data. In a serving process the free HBM is often reserved up front
 * (by the inference engine, or by PyTorch's caching allocator), so a new
 * cudaMalloc there fails, and a cudaFree waits for the whole device. Code
 * that holds a pool and its page lists but no t2i_store is in the same
 * position: a store allocates its chunk counters when it is created.
 *
 * Scratch: the CTAs of a launch take their chunks from counters kept in a
 * static 2 KiB device array of the library (64 counters of 32 bytes: one
 * per launch of a call). Every GPU that loads the library holds the array
 * until the process exits. A call first zeroes the counters it will use
 * (cudaMemsetAsync on cuda_stream), because every call shares the array and
 * it keeps whatever the last call left. Calls that overlap on the GPU (on
 * other streams or from other threads) race on the counters and can skip or
 * repeat chunks: order such calls on one stream. The first call on a device
 * sets up that device: it looks up the array's device address
 * (cudaGetSymbolAddress) and the gather kernels' occupancy. Make that first
 * call before any stream capture. No call allocates: no cudaMalloc, no
 * cudaFree, no library routine that allocates.
 *
 * pool_dev, pool_bytes: the pool, device memory of `device`; pool_bytes is a
 *   positive multiple of page_bytes, a power of two in [256 B, 1 GiB].
 * pages, n_pages: the object's page list in byte order (a host array of
 *   page indices into the pool, e.g. from t2i_ctl_object), read during the
 *   call. n_pages = ceil(nbytes / page_bytes), at most 64 launches of
 *   min(7,930, 64 GiB / page_bytes) pages, one scratch counter each: 507,520
 *   pages for pages up to 8 MiB. Larger objects are INVALID.
 * nbytes: the object's size. dst_dev, dst_bytes: the destination, device
 *   memory of `device` that does not overlap the pool. cast = 1 writes bf16
 *   (nbytes % 4 == 0, even dst_dev, dst_bytes >= nbytes / 2); cast = 0
 *   copies (dst_bytes >= nbytes).
 * Errors: INVALID (arguments, a page outside the pool, sizes beyond the
 *   maximum; nothing is enqueued), CUDA (set-up or a launch failed).
 *   t2i_last_error(NULL) describes them.                                    */
t2i_status t2i_gather_noalloc(const void* pool_dev, uint64_t pool_bytes, uint64_t page_bytes, const uint32_t* pages,
                              uint32_t n_pages, uint64_t nbytes, void* dst_dev, uint64_t dst_bytes, uint32_t cast,
                              int device, void* cuda_stream);

/* =========================================================================
 * First-layer prefix caching (§5.1). A model of L layers keeps its first L_e
 * layers in the store and streams the rest from host memory while inference
 * runs; T_load / T_comp are one layer's load / inference time. Pure host
 * arithmetic: INVALID for negative or non-finite times, L_e > L or a null out.
 * ========================================================================= */

/* Eq. (1): max(L * t_comp, (L - L_e) * t_load + t_comp) (uniform layers,
 * t_load >= t_comp).                                                         */
t2i_status t2i_e2e_latency(uint32_t L, uint32_t L_e, double t_load, double t_comp, double* out);

/* Eq. (2): ceil((L * (t_load - t_comp) + t_comp) / t_load), clamped to
 * [0, L]: the smallest cached prefix that hides loading (t_load > 0).       */
t2i_status t2i_prefix_layers(uint32_t L, double t_load, double t_comp, uint32_t* out);

/* The schedule Eq. (1) summarises, for per-layer times (the paper notes the
 * equations extend to non-uniform layers): layers >= L_e load back to back
 * from time 0; layer l computes once it is loaded and layer l-1 has
 * computed. *out = the end of the last computation.                          */
t2i_status t2i_pipeline_latency(const double* t_load, const double* t_comp, uint32_t L, uint32_t L_e,
                                double* out);

/* The smallest L_e whose pipeline latency is the plain sum of the
 * computations (loading fully hidden), for per-layer times.                 */
t2i_status t2i_prefix_layers_pipeline(const double* t_load, const double* t_comp, uint32_t L, uint32_t* out);

/* Streams layers [first, n_layers) of one model into the store: for each
 * such layer l, one t2i_put_batch of descs[layer_off[l] .. layer_off[l+1])
 * on cuda_stream, then events[l] (a cudaEvent_t, if events is not NULL)
 * recorded on cuda_stream, so that inference can wait for each layer
 * (cudaStreamWaitEvent or t2i_get_batch_after) while later layers still
 * load (§5.1: inference starts on the cached first layers while the rest
 * load asynchronously). out_ids[layer_off[l] + k] receives the ids of the
 * streamed layers. Stops at the first layer that fails and returns its
 * status: earlier layers stay stored and their events recorded.             */
t2i_status t2i_put_layers(t2i_store* store, const t2i_put_desc* descs, const uint32_t* layer_off, uint32_t n_layers,
                          uint32_t first, t2i_id* out_ids, void* cuda_stream, void* const* events);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* T2ISTORE_H */
