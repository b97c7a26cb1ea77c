"""Producer processes for cross-process pulls (imported by spawned children;
not a test module). A producer puts objects into its own store, shares the
store's pool with the parent through CUDA IPC (torch sends CUDA tensors
between processes that way) together with the objects' page lists, and keeps
the pool alive until the parent is done with it."""


def run(to_parent, from_parent, sizes, page_bytes, seed):
    """Objects of ``sizes`` bytes; also sends their expected bytes."""
    import torch

    from paper_2607_26566_gb300 import Store, put_descs

    dev = torch.device("cuda", 0)
    pool = torch.empty(64 * page_bytes, dtype=torch.uint8, device=dev)
    st = Store(pool, page_bytes)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    xs = [torch.randint(0, 256, (n,), dtype=torch.uint8, device=dev, generator=g) for n in sizes]
    s, ids = st.put_batch(put_descs(xs, dtype_tag=7))
    torch.cuda.synchronize()           # the bytes are in the pool before the parent reads them
    objects = [(x.numel(), st.ctl.object(int(i))[2], 7) for x, i in zip(xs, ids)]
    to_parent.put((s, pool, objects, [x.cpu() for x in xs]))
    from_parent.get(timeout=300)       # the parent's copies have run
    st.close()
