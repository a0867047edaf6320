"""Hybrid six-turn session across two replicas on one GPU (paper Sec. 2.2, Sec. 4.2).

64 layers of which every 4th is full attention (16 paged bf16 layers, 8 KV
heads, head_dim 128, 16-token pages) and 48 hold a recurrent page: an fp32
recurrent state of 16 heads x 128 x 128 plus a bf16 convolution window,
padded to 4 KiB (1,097,728 bytes per layer, moved as opaque bytes as the
paper's patch does, Sec. 2.2).  Replica A prefills a 32k-token
context and stores it with the state snapshot at 32,768; each later turn the
other replica restores the chunks it lacks plus the snapshot at the current
boundary, appends 2,048 tokens (new pages and a new state), and stores the new
chunks with the snapshot at the new boundary.  Every stored chunk and
snapshot, every restored page and state slot, and at the end each replica's
whole context, are checked byte for byte against the CPU oracle.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import POISON, first_mismatch, kvx, np_of
from paper_2609_15021_gb300 import synth
from paper_2609_15021_gb300.hybrid import HybridShape, Replica, SharedTier, load_prefix, store_prefix

pytestmark = pytest.mark.gpu

SHAPE = HybridShape()
FIRST, APPEND, TURNS = 32768, 2048, 6
N_BLK = 4096


def mini_spec(n_pages):
    s = SHAPE
    return oracle.PoolSpec(s.attn_layers, n_pages, s.block_tokens, s.kv_heads, s.head_dim, s.elem_bytes, oracle.HND)


def fill_new_tokens(rep, a, b, seed):
    """'Prefill' tokens [a, b) (whole pages): seeded bytes into the replica's new pages.
    Returns the pages' bytes per layer (host) in token order."""
    pb = SHAPE.page_bytes
    pages = rep.table[a // SHAPE.block_tokens:b // SHAPE.block_tokens]
    idx = torch.tensor(pages, dtype=torch.int64, device="cuda")
    host = []
    for l, layer in enumerate(rep.attn_layers):
        h = synth.splitmix64_bytes(len(pages) * pb, seed * 1000 + l)
        layer.view(-1, pb).index_copy_(0, idx, torch.from_numpy(h).cuda().view(len(pages), pb))
        host.append(h)
    return host


def fill_state(rep, slot, seed):
    sb = SHAPE.state_bytes
    snap = synth.splitmix64_bytes(SHAPE.snapshot_bytes, seed)
    for l, st in enumerate(rep.state):
        st[slot * sb:(slot + 1) * sb].copy_(torch.from_numpy(snap[l * sb:(l + 1) * sb]))
    return snap


def gather(rep, a, b):
    pb = SHAPE.page_bytes
    pages = rep.table[a // SHAPE.block_tokens:-(-b // SHAPE.block_tokens)]
    idx = torch.tensor(pages, dtype=torch.int64, device="cuda")
    return [np_of(layer.view(-1, pb).index_select(0, idx)).reshape(-1) for layer in rep.attn_layers]


def test_hybrid_six_turn_session(orc):
    k = kvx()
    C = SHAPE.chunk_tokens
    total = FIRST + (TURNS - 1) * APPEND
    tier = SharedTier(SHAPE, total, max_snapshots=4)
    A = Replica(SHAPE, N_BLK, 2, list(map(int, synth.permuted_table(N_BLK, N_BLK, 1))))
    B = Replica(SHAPE, N_BLK, 2, list(map(int, synth.permuted_table(N_BLK, N_BLK, 2))))
    for rep in (A, B):
        for t in rep.attn_layers + rep.state:
            t.fill_(POISON)
    ctx = k.kv_ctx_create(0)
    stream = torch.cuda.Stream()
    truth = {}     # chunk index -> oracle bytes
    snaps = {}     # boundary -> snapshot bytes
    times = []
    try:
        n = 0
        for turn in range(TURNS):
            rep = A if turn % 2 == 0 else B
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            ev[0].record(stream)
            if turn > 0:
                lo = rep.tokens
                with torch.cuda.stream(stream):
                    load_prefix(ctx, rep, tier, lo, n, state_slot=0)
                ev[1].record(stream)
                stream.synchronize()
                # restored pages and state against the oracle
                m = mini_spec((n - lo) // SHAPE.block_tokens)
                want = oracle_pages = [np.full(m.layer_bytes, POISON, np.uint8) for _ in range(m.num_layers)]
                ident = np.arange(m.num_blocks, dtype=np.int32)
                rc, _ = orc.load(m, oracle_pages, ident, 0, n - lo, C, [truth[c] for c in range(lo // C, n // C)],
                                 n_threads=8)
                assert rc == 0
                for l, got in enumerate(gather(rep, lo, n)):
                    assert first_mismatch(got, want[l]) is None, (turn, l)
                sb = SHAPE.state_bytes
                for l, st in enumerate(rep.state):
                    assert first_mismatch(np_of(st[:sb]), snaps[n][l * sb:(l + 1) * sb]) is None, (turn, l)
                    assert np.all(np_of(st[sb:]) == POISON)   # the other slot untouched
            else:
                ev[1].record(stream)
            # append (turn 0: prefill) and store the new chunks with the new boundary snapshot
            a, b = n, (FIRST if turn == 0 else n + APPEND)
            rep.grow(b)
            pages_host = fill_new_tokens(rep, a, b, seed=10 + turn)
            snaps[b] = fill_state(rep, 0, seed=50 + turn)
            rep.tokens = b
            torch.cuda.synchronize()
            ev2 = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            ev2[0].record(stream)
            with torch.cuda.stream(stream):
                store_prefix(ctx, rep, tier, a, b, state_slot=0)
            ev2[1].record(stream)
            stream.synchronize()
            m = mini_spec((b - a) // SHAPE.block_tokens)
            want = [np.full(SHAPE.chunk_bytes, POISON, np.uint8) for _ in range((b - a) // C)]
            rc, _ = orc.store(m, pages_host, np.arange(m.num_blocks, dtype=np.int32), 0, b - a, C, want, n_threads=8)
            assert rc == 0
            for i, w in enumerate(want):
                c = a // C + i
                truth[c] = w
                assert first_mismatch(np_of(tier.chunk(c)), w) is None, (turn, c)
            assert first_mismatch(np_of(tier.snapshot(b)), snaps[b]) is None
            times.append((turn, "A" if rep is A else "B", ev[0].elapsed_time(ev[1]), ev2[0].elapsed_time(ev2[1])))
            n = b
        assert k.kv_get_device_error(ctx) == -1
        # each replica's whole context equals the session's truth
        for rep in (A, B):
            m = mini_spec(rep.tokens // SHAPE.block_tokens)
            want = [np.full(m.layer_bytes, POISON, np.uint8) for _ in range(m.num_layers)]
            rc, _ = orc.load(m, want, np.arange(m.num_blocks, dtype=np.int32), 0, rep.tokens, C,
                             [truth[c] for c in range(rep.tokens // C)], n_threads=8)
            assert rc == 0
            for l, got in enumerate(gather(rep, 0, rep.tokens)):
                assert first_mismatch(got, want[l]) is None, l
        # chunks present but no snapshot at that boundary: the prefix is not recoverable
        assert all(c in tier.present for c in range((n - C) // C))
        with pytest.raises(LookupError):
            load_prefix(ctx, A, tier, 0, n - C, state_slot=1)
        for turn, who, load_ms, store_ms in times:
            print(f"turn {turn} on {who}: restore {load_ms:.2f} ms, store {store_ms:.2f} ms")
    finally:
        k.kv_ctx_destroy(ctx)
        tier.close()
