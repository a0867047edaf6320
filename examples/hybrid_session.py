"""A hybrid model's multi-turn session moving between two replicas (paper Sec. 2.2).

A hybrid model keeps paged K/V only in its full-attention layers; its
linear-attention layers carry a recurrent state instead, and a prefix can be
resumed only with the state snapshot taken at the prefix's boundary.  Here two
replicas of a 64-layer hybrid (16 attention layers of 8 KV heads x 128 dims,
bf16, 16-token pages; 48 recurrent pages of 1,097,728 bytes) take turns on one
conversation, as a router that alternates placement would send it:

  turn 0   replica A prefills 32k tokens and stores them with the snapshot;
  turn k   the other replica restores the tokens it lacks plus the snapshot at
           the current boundary, appends 2,048 tokens (its "prefill" of the new
           turn), and stores the new chunks with the new boundary's snapshot.

Both replicas run in this process on one GPU and share one pinned host tier
(hybrid.SharedTier).  The new tokens' K/V and the new state are random bytes
standing in for the model's output.  At the end, each replica's pages for the
tokens both hold must be byte-identical, and each replica's state must equal
the snapshot of the boundary it last stored or restored.

Run from the repository root, with the library built:
    python examples/hybrid_session.py
Prints one line per turn and "session bit-exact" and exits 0 on success.
"""
import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

FIRST, APPEND, TURNS, POOL_PAGES = 32768, 2048, 6, 4096


def produce(rep, t0, t1, gen):
    """The model's output for tokens [t0, t1): random K/V bytes into the replica's
    pages of those tokens, and a new recurrent state in slot 0."""
    pb = rep.shape.page_bytes
    pages = torch.tensor(rep.table[t0 // rep.shape.block_tokens:t1 // rep.shape.block_tokens], device="cuda")
    for layer in rep.attn_layers:
        new = torch.randint(0, 256, (len(pages), pb), dtype=torch.uint8, device="cuda", generator=gen)
        layer.view(-1, pb).index_copy_(0, pages, new)
    sb = rep.shape.state_bytes
    for st in rep.state:
        st[:sb].copy_(torch.randint(0, 256, (sb,), dtype=torch.uint8, device="cuda", generator=gen))


def pages_of(rep, t1):
    pb = rep.shape.page_bytes
    idx = torch.tensor(rep.table[:t1 // rep.shape.block_tokens], device="cuda")
    return [layer.view(-1, pb).index_select(0, idx) for layer in rep.attn_layers]


def main():
    from paper_2609_15021_gb300 import kvxfer as k
    from paper_2609_15021_gb300.hybrid import HybridShape, Replica, SharedTier, load_prefix, store_prefix
    shape = HybridShape()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(2026)
    tier = SharedTier(shape, FIRST + (TURNS - 1) * APPEND, max_snapshots=2)
    order = torch.randperm(POOL_PAGES, generator=torch.Generator().manual_seed(7)).tolist()
    reps = [Replica(shape, POOL_PAGES, 1, order), Replica(shape, POOL_PAGES, 1, order[::-1])]
    ctx = k.kv_ctx_create(0)
    stream = torch.cuda.Stream()
    n = 0
    try:
        with torch.cuda.stream(stream):
            for turn in range(TURNS):
                rep = reps[turn % 2]
                name = "AB"[turn % 2]
                a, b, c = (torch.cuda.Event(enable_timing=True) for _ in range(3))
                a.record()
                lo = rep.tokens
                if turn > 0:
                    load_prefix(ctx, rep, tier, lo, n, state_slot=0)
                b.record()
                hi = FIRST if turn == 0 else n + APPEND
                rep.grow(hi)
                produce(rep, n, hi, gen)
                rep.tokens = hi
                d = torch.cuda.Event(enable_timing=True)
                d.record()
                store_prefix(ctx, rep, tier, n, hi, state_slot=0)
                c.record()
                stream.synchronize()
                restored = f"restored {n - lo} tokens + snapshot in {a.elapsed_time(b):.2f} ms" if turn else "prefill"
                print(f"turn {turn} on replica {name}: {restored}; stored {hi - n} tokens + snapshot in "
                      f"{d.elapsed_time(c):.2f} ms")
                n = hi
        if k.kv_get_device_error(ctx) != -1:
            raise SystemExit("a block-table entry was out of range")
        common = min(r.tokens for r in reps)
        for la, lb in zip(pages_of(reps[0], common), pages_of(reps[1], common)):
            if not torch.equal(la, lb):
                raise SystemExit("the replicas' pages differ")
        sb = shape.state_bytes
        for rep in reps:
            snap = tier.snapshot(rep.tokens).to("cuda")
            for l, st in enumerate(rep.state):
                if not torch.equal(st[:sb], snap[l * sb:(l + 1) * sb]):
                    raise SystemExit("a replica's state is not its boundary's snapshot")
        print(f"{common} common tokens in both replicas' pages; session bit-exact")
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()


if __name__ == "__main__":
    main()
