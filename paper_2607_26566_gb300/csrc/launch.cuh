// Launch packing of the store's kernels (part of store.cu; included after
// the Store class). A batch's segments are split into 16-byte-aligned and
// other ones, packed into as few launches as their descriptors allow (each
// launch carries up to ~31 KiB of descriptors and page numbers in its
// parameters), and launched with programmatic dependent launch: chunked
// persistent grids for very large launches, else one CTA per 64 KiB. Together with kernels.cuh this decides what a launch does, so
// profiles are keyed to a hash of both files. Included by store.cu inside
// namespace t2i.
#pragma once

template <Mode M, bool GENERAL, int BLOB>
t2i_status Store::launch_one(const std::vector<SegDesc>& sd, const std::vector<uint32_t>& pages, uint32_t n_granules,
                             cudaStream_t stream) {
    auto* p = reinterpret_cast<LaunchParams<BLOB>*>(param_buf_);
    // a get with no cast segment runs the leaner copy-only kernel: aligned
    // and unchunked (4 resident CTAs per SM instead of 3, +3.8% on the
    // adapter gets; an aligned chunked get keeps the other kernel, 0.5%
    // faster there), or any alignment (the cast's registers left out)
    bool any_cast = false;
    for (const SegDesc& d : sd) any_cast = any_cast || (d.nbytes_flags & kCastFlag) != 0;
    // chunks from the counter when the launch holds at least kDynMinCtaBytes
    // per resident CTA of the kernel that would run chunked
    const bool copy_any = M == Mode::Get && !any_cast && GENERAL && kGetCopyKernel;
    const bool chunked = uint64_t(n_granules) * kGranule >=
                         kDynMinCtaBytes * uint64_t(max_ctas_[copy_any ? int(Mode::GetCopy) : int(M)][GENERAL ? 1 : 0]);
    const int mode =
        (M == Mode::Get && !any_cast && (!chunked || GENERAL) && kGetCopyKernel) ? int(Mode::GetCopy) : int(M);
    p->h.pool = pool_;
    p->h.work = chunked ? cur_work_ : 0;
    p->h.chunk_granules = kChunkGranules;
    p->h.flags = p->h.work == 0 ? launch_flags_ : 0;
    p->h.n_seg = static_cast<uint32_t>(sd.size());
    p->h.n_granules = n_granules;
    p->h.page_shift = page_shift_;
    p->h.piece_bytes = static_cast<uint32_t>(std::min<uint64_t>(kPieceBytes, uint64_t(1) << page_shift_));
    p->h.pages_offset = static_cast<uint32_t>(sd.size() * sizeof(SegDesc));
    std::memcpy(p->blob, sd.data(), sd.size() * sizeof(SegDesc));
    std::memcpy(p->blob + p->h.pages_offset, pages.data(), pages.size() * sizeof(uint32_t));
    // Grid. A chunked launch is persistent: the resident CTAs of the device.
    // Otherwise CTAs take equal static shares of 16-64 KiB: the resident CTAs
    // while that gives each at least kMinCtaBytes, and one CTA per
    // kStaticCtaBytes beyond, so that the hardware hands the CTAs of a larger
    // launch to whichever SMs free up first.
    const uint64_t bytes = uint64_t(n_granules) * kGranule;
    const uint64_t resident = uint64_t(max_ctas_[mode][GENERAL ? 1 : 0]);
    const uint64_t want = (bytes + kMinCtaBytes - 1) / kMinCtaBytes;
    uint64_t g = std::max<uint64_t>(1, std::min<uint64_t>(want, resident));
    if (p->h.work == 0) g = std::max<uint64_t>(g, std::min<uint64_t>((bytes + kStaticCtaBytes - 1) / kStaticCtaBytes,
                                                                     0x7FFFFFFFull));
    const unsigned grid = static_cast<unsigned>(g);
    p->h.prefetch_ctas = kPrefetchFirstWave ? static_cast<uint32_t>(std::min<uint64_t>(g, resident)) : grid;
    void* args[] = {p};
    const void* fn = M == Mode::Put                  ? reinterpret_cast<const void*>(scatter_put_kernel<BLOB, GENERAL>)
                     : mode == int(Mode::GetCopy)     ? reinterpret_cast<const void*>(gather_copy_kernel<BLOB, GENERAL>)
                     : M == Mode::Get                 ? reinterpret_cast<const void*>(gather_get_kernel<BLOB, GENERAL>)
                                                      : reinterpret_cast<const void*>(compact_move_kernel<BLOB>);
    if (fail_countdown_ && --fail_countdown_ == 0) {
        err_ = "kernel launch failed: injected failure (t2i_inject_launch_failure)";
        return T2I_ERR_CUDA;
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(kThreads);
    lc.dynamicSmemBytes = 0;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelExC(&lc, fn, args);
    if (e != cudaSuccess) {
        err_ = std::string("kernel launch failed: ") + cudaGetErrorString(e);
        return T2I_ERR_CUDA;
    }
    ctl_.counters().launches++;
    return T2I_OK;
}

// Segments whose user address is 16-byte aligned go to the aligned kernels,
// the others (rare: views at odd offsets) to the any-alignment kernels.
template <Mode M>
t2i_status Store::launch_segments(const std::vector<Seg>& segs, cudaStream_t stream) {
    aligned_.clear();
    general_.clear();
    for (const Seg& s : segs) ((s.user & 15u) == 0 ? aligned_ : general_).push_back(s);
    t2i_status st = T2I_OK;
    if (!aligned_.empty()) st = launch_group<M, false>(aligned_, stream);
    if (st == T2I_OK && !general_.empty()) {
        if (M == Mode::Move) return T2I_ERR_INVALID;  // pool pages are always aligned
        st = launch_group<(M == Mode::Move ? Mode::Put : M), true>(general_, stream);
    }
    return st;
}

// Packs segments into launches: descriptors and page numbers of as many
// segments as fit one launch's parameter space; an object whose page list
// alone does not fit is split at page boundaries.
template <Mode M, bool GENERAL>
t2i_status Store::launch_group(const std::vector<Seg>& segs, cudaStream_t stream) {
    sd_.clear();
    lp_.clear();
    uint64_t gran = 0;  // next free granule of the launch byte space
    auto flush = [&]() -> t2i_status {
        if (sd_.empty()) return T2I_OK;
        const size_t bytes = sd_.size() * sizeof(SegDesc) + lp_.size() * sizeof(uint32_t);
        t2i_status st;
        if (bytes <= size_t(kBlobTiny))
            st = launch_one<M, GENERAL, kBlobTiny>(sd_, lp_, uint32_t(gran), stream);
        else if (bytes <= size_t(kBlobSmall))
            st = launch_one<M, GENERAL, kBlobSmall>(sd_, lp_, uint32_t(gran), stream);
        else if (bytes <= size_t(kBlobMid))
            st = launch_one<M, GENERAL, kBlobMid>(sd_, lp_, uint32_t(gran), stream);
        else
            st = launch_one<M, GENERAL, kBlobLarge>(sd_, lp_, uint32_t(gran), stream);
        sd_.clear();
        lp_.clear();
        gran = 0;
        return st;
    };
    const uint64_t P = uint64_t(1) << page_shift_;
    // a segment's page list fits one launch, and its bytes fit the 32-bit
    // granule offsets of the launch byte space (64 GiB per segment)
    const uint64_t max_pages_per_seg = std::min<uint64_t>((kBlobLarge - sizeof(SegDesc)) / sizeof(uint32_t),
                                                          std::max<uint64_t>(1, kMaxSegBytes / P));
    for (const Seg& s : segs) {
        const uint64_t nbytes = s.nbytes_flags & kSegBytesMask;
        const uint64_t flags = s.nbytes_flags & kCastFlag;
        // consecutive pages travel as their first page alone
        bool run = s.n_pages > 1;
        for (uint32_t k = 1; run && k < s.n_pages; ++k) run = s.pages[k] == s.pages[0] + k;
        const uint64_t seg_pages = run ? std::max<uint64_t>(1, kMaxSegBytes / P) : max_pages_per_seg;
        for (uint64_t p0 = 0; p0 < s.n_pages; p0 += seg_pages) {
            const uint64_t np = std::min<uint64_t>(seg_pages, s.n_pages - p0);
            const uint64_t entries = run ? 1 : np;
            const uint64_t off = p0 * P;
            const uint64_t seg_bytes = std::min<uint64_t>(nbytes - off, np * P);
            const uint64_t seg_gran = (seg_bytes + kGranule - 1) / kGranule;
            const size_t need = (sd_.size() + 1) * sizeof(SegDesc) + (lp_.size() + entries) * sizeof(uint32_t);
            if (need > size_t(kBlobLarge) || gran + seg_gran > 0xFFFFFFFFull) {
                t2i_status st = flush();
                if (st != T2I_OK) return st;
            }
            SegDesc d;
            // a get with the cast writes half as many bytes as it reads
            d.user = s.user + (flags ? off / 2 : off);
            d.nbytes_flags = seg_bytes | flags | (run && np > 1 ? kRunFlag : 0);
            d.start = static_cast<uint32_t>(gran);
            d.page_begin = static_cast<uint32_t>(lp_.size());
            sd_.push_back(d);
            lp_.insert(lp_.end(), s.pages + p0, s.pages + p0 + entries);
            gran += seg_gran;
        }
    }
    return flush();
}
