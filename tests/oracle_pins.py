"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each ``pin_*`` takes an oracle object (``oracle.COracle`` or a compiled copy
with a planted mistake) and raises AssertionError on a mismatch.  They are
run by ``test_oracle_pins.py`` against the real oracle and, in a subprocess,
against mutated copies of ``kv_oracle.c`` (``test_oracle_mutations.py``).

What pins the definition (paper Sec. 3.1-3.2: pages of a paged pool gathered
into fixed-token chunks and scattered back):
  * special cases that reduce to a library routine: with an identity table
    and chunk = page, an NHD chunk is the page's bytes (plain slicing) and an
    HND chunk is the page with its head and token axes swapped (np.transpose);
  * the block table acts as np.take over pages;
  * store then load with a table that lists every page reproduces the pool
    byte for byte, and load then store reproduces the chunks;
  * load writes exactly the chunk's bytes and nothing else; store writes no
    byte past a chunk's valid length;
  * chunk boundaries: splitting a chunk in two or starting the range one
    chunk later regroups the same rows;
  * a hand-derived worked example (tests/golden/hand_example.txt);
  * brute force over every block table of a 4-block pool against the
    independent NumPy formulation.
"""
from __future__ import annotations

import itertools
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from oracle import HND, NHD, PoolSpec  # noqa: E402
from paper_2609_15021_gb300 import synth  # noqa: E402

POISON = synth.POISON
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def make_layers(spec: PoolSpec, seed: int, avoid_poison: bool = False):
    out = []
    for l in range(spec.num_layers):
        b = synth.splitmix64_bytes(spec.layer_bytes, seed + 7919 * l)
        if avoid_poison:
            b[b == POISON] = 0
        out.append(b)
    return out


def poisoned_chunks(orc, spec, t0, t1, C, extra=0):
    return [np.full(orc.chunk_bytes(spec, n) + extra, POISON, np.uint8)
            for n in oracle.chunk_tokens_of(t0, t1, C)]


def do_store(orc, spec, layers, table, t0, t1, C, extra=0):
    chunks = poisoned_chunks(orc, spec, t0, t1, C, extra)
    rc, bad = orc.store(spec, layers, table, t0, t1, C, chunks)
    assert rc == oracle.OK, rc
    assert bad == -1, bad
    return chunks


def do_load(orc, spec, layers, table, t0, t1, C, chunks):
    new = [l.copy() for l in layers]
    rc, bad = orc.load(spec, new, table, t0, t1, C, chunks)
    assert rc == oracle.OK, rc
    assert bad == -1, bad
    return new


# ---------------------------------------------------------------- pins


def pin_nhd_identity_is_page_bytes(orc):
    """NHD page = [2][B][H][row] = chunk layout of one layer: chunk c is page c verbatim."""
    for L in (1, 2):
        spec = PoolSpec(L, 4, 4, 3, 8, 2, NHD)
        layers = make_layers(spec, 11)
        C = spec.block_tokens
        for t0 in (0, 2 * C):
            chunks = do_store(orc, spec, layers, np.arange(4, dtype=np.int32), t0, 4 * C, C)
            for i, ch in enumerate(chunks):
                c = t0 // C + i
                pages = [lay[c * spec.page_bytes:(c + 1) * spec.page_bytes] for lay in layers]
                assert np.array_equal(ch, np.concatenate(pages)), (L, t0, c)


def pin_hnd_identity_is_transpose(orc):
    """HND page [2][H][B][row] with chunk = page: the chunk is the page with H and B swapped."""
    for (H, B, D, e) in ((3, 4, 8, 2), (2, 8, 16, 1), (1, 4, 4, 4)):
        spec = PoolSpec(1, 3, B, H, D, e, HND)
        layers = make_layers(spec, 13 + H)
        chunks = do_store(orc, spec, layers, np.arange(3, dtype=np.int32), 0, 3 * B, B)
        for c, ch in enumerate(chunks):
            page = layers[0][c * spec.page_bytes:(c + 1) * spec.page_bytes]
            want = np.transpose(page.reshape(2, H, B, spec.row_bytes), (0, 2, 1, 3)).reshape(-1)
            assert np.array_equal(ch, want), (H, B, c)


def pin_table_is_take(orc):
    """Storing through table T equals storing pool[T] (np.take over pages) through the identity."""
    for layout in (HND, NHD):
        spec = PoolSpec(2, 8, 4, 2, 8, 2, layout)
        layers = make_layers(spec, 17)
        table = synth.permuted_table(8, 6, seed=5)
        t1 = 6 * spec.block_tokens - 3
        C = 2 * spec.block_tokens
        got = do_store(orc, spec, layers, table, 0, t1, C)
        taken = [np.take(l.reshape(8, spec.page_bytes), table, axis=0).reshape(-1) for l in layers]
        spec6 = PoolSpec(2, 6, 4, 2, 8, 2, layout)
        want = do_store(orc, spec6, taken, np.arange(6, dtype=np.int32), 0, t1, C)
        for a, b in zip(got, want):
            assert np.array_equal(a, b), layout


def pin_round_trip_bijective(orc):
    """Table listing every page, full range: load(store(pool)) == pool and store(load(chunks)) == chunks."""
    for layout in (HND, NHD):
        spec = PoolSpec(3, 6, 4, 2, 8, 2, layout)
        layers = make_layers(spec, 19)
        ta = synth.permuted_table(6, 6, seed=1)
        tb = synth.permuted_table(6, 6, seed=2)
        t1, C = 6 * 4, 8
        chunks = do_store(orc, spec, layers, ta, 0, t1, C)
        poisoned = [np.full_like(l, POISON) for l in layers]
        back = do_load(orc, spec, poisoned, ta, 0, t1, C, chunks)
        for a, b in zip(back, layers):
            assert np.array_equal(a, b), layout
        other = do_load(orc, spec, poisoned, tb, 0, t1, C, chunks)
        again = do_store(orc, spec, other, tb, 0, t1, C)
        for a, b in zip(again, chunks):
            assert np.array_equal(a, b), layout


def pin_untouched_bytes(orc):
    """Store writes nothing past a chunk's valid bytes; load writes exactly the chunks' bytes."""
    for layout in (HND, NHD):
        spec = PoolSpec(2, 8, 4, 2, 8, 2, layout)
        layers = make_layers(spec, 23, avoid_poison=True)
        table = synth.permuted_table(8, 5, seed=9)
        t1, C = 5 * 4 - 1, 8  # ragged last page and short last chunk
        extra = 64
        chunks = do_store(orc, spec, layers, table, 0, t1, C, extra=extra)
        total = 0
        for ch in chunks:
            assert np.all(ch[-extra:] == POISON), layout
            valid = ch[:-extra]
            assert not np.any(valid == POISON), layout
            total += valid.size
        assert total == spec.num_layers * 2 * t1 * spec.num_heads * spec.row_bytes
        dest = do_load(orc, spec, [np.full_like(l, POISON) for l in layers], table, 0, t1, C,
                       [ch[:-extra] for ch in chunks])
        changed = sum(int(np.count_nonzero(d != POISON)) for d in dest)
        assert changed == total, (layout, changed, total)
        again = do_store(orc, spec, dest, table, 0, t1, C)
        for a, b in zip(again, chunks):
            assert np.array_equal(a, b[:-extra]), layout


def pin_chunk_boundaries(orc):
    """A chunk of 2C tokens is its two C-token halves regrouped along the token axis, and
    starting the range one chunk later yields the same later chunks."""
    for layout in (HND, NHD):
        spec = PoolSpec(2, 10, 4, 3, 8, 2, layout)
        layers = make_layers(spec, 29)
        table = synth.permuted_table(10, 9, seed=3)
        t1 = 9 * 4 - 2
        big = do_store(orc, spec, layers, table, 0, t1, 8)
        small = do_store(orc, spec, layers, table, 0, t1, 4)
        HR = spec.num_heads * spec.row_bytes
        for c, ch in enumerate(big):
            parts = small[2 * c:2 * c + 2]
            halves = [p.reshape(spec.num_layers, 2, -1, HR) for p in parts]
            want = np.concatenate(halves, axis=2).reshape(-1)
            assert np.array_equal(ch, want), (layout, c)
        later = do_store(orc, spec, layers, table, 8, t1, 8)
        for a, b in zip(later, big[1:]):
            assert np.array_equal(a, b), layout


def _parse_hand_example():
    sections, cur = {}, None
    with open(os.path.join(GOLDEN, "hand_example.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            if line.startswith("[") and line.endswith("]"):
                cur = line[1:-1]
                sections[cur] = []
            else:
                sections[cur].extend(int(x) for x in line.split())
    return sections


def pin_hand_example(orc):
    """The worked example derived by hand in tests/golden/hand_example.txt."""
    s = _parse_hand_example()
    row = 16
    for layout, key in ((HND, "pool_hnd"), (NHD, "pool_nhd")):
        spec = PoolSpec(1, 3, 2, 2, 16, 1, layout)
        layer = np.repeat(np.array(s[key], dtype=np.uint8), row)
        table = np.array(s["table"], dtype=np.int32)
        full = do_store(orc, spec, [layer], table, 0, 4, 4)
        assert np.array_equal(full[0], np.repeat(np.array(s["chunk_t4"], np.uint8), row)), layout
        short = do_store(orc, spec, [layer], table, 0, 3, 4)
        assert np.array_equal(short[0], np.repeat(np.array(s["chunk_t3"], np.uint8), row)), layout
    spec = PoolSpec(1, 3, 2, 2, 16, 1, HND)
    dest = do_load(orc, spec, [np.full(3 * spec.page_bytes, POISON, np.uint8)],
                   np.array(s["load_table"], np.int32), 0, 4, 4,
                   [np.repeat(np.array(s["chunk_t4"], np.uint8), row)])
    assert np.array_equal(dest[0], np.repeat(np.array(s["load_result_hnd"], np.uint8), row))


def pin_bruteforce_vs_numpy(orc):
    """Every table over a 4-block pool, every end token, three chunk sizes, both layouts:
    the C loops agree with the NumPy advanced-indexing formulation."""
    for layout in (HND, NHD):
        spec = PoolSpec(2, 4, 2, 2, 8, 2, layout)
        layers = make_layers(spec, 31)
        B = spec.block_tokens
        tables = [np.array(p, dtype=np.int32) for p in itertools.permutations(range(4))]
        tables += [np.array(p, dtype=np.int32) for p in itertools.permutations(range(4), 2)]
        for table in tables:
            for C in (B, 2 * B, 4 * B):
                for t1 in range(0, len(table) * B + 1):
                    got = do_store(orc, spec, layers, table, 0, t1, C)
                    want = oracle.np_store(spec, layers, table, 0, t1, C)
                    assert len(got) == len(want)
                    for a, b in zip(got, want):
                        assert np.array_equal(a, b), (layout, table, C, t1)
                    if t1 % (3 * B) == 1 or t1 == len(table) * B:
                        dest0 = [np.full_like(l, POISON) for l in layers]
                        gl = do_load(orc, spec, dest0, table, 0, t1, C, got)
                        wl = oracle.np_load(spec, dest0, table, 0, t1, C, got)
                        for a, b in zip(gl, wl):
                            assert np.array_equal(a, b), (layout, table, C, t1)


def pin_error_codes(orc):
    """Argument rules: aligned start, chunk a multiple of the page, range inside the table."""
    spec = PoolSpec(1, 4, 4, 1, 8, 2, HND)
    layers = make_layers(spec, 37)
    table = np.arange(4, dtype=np.int32)
    ch = [np.zeros(orc.chunk_bytes(spec, 8), np.uint8) for _ in range(4)]
    assert orc.store(spec, layers, table, 4, 8, 8, ch)[0] == oracle.EALIGN      # start not on a chunk
    assert orc.store(spec, layers, table, 0, 8, 6, ch)[0] == oracle.EALIGN      # C % B != 0
    assert orc.store(spec, layers, table, 0, 17, 8, ch)[0] == oracle.ERANGE     # past the table
    assert orc.store(spec, layers, table, 0, 16, 8, ch)[0] == oracle.OK         # exactly the table
    assert orc.store(spec, layers, table, 0, 16, 8, ch[:1])[0] == oracle.ERANGE  # too few chunks
    assert orc.store(spec, layers, table, 8, 4, 8, ch)[0] == oracle.ERANGE      # end before start
    assert orc.store(spec, layers, table, 8, 8, 8, [])[0] == oracle.OK          # empty range
    assert orc.load(spec, layers, table, 0, 16, 0, ch)[0] == oracle.EINVAL      # zero chunk size


def pin_bad_block(orc):
    """An out-of-range page id names no page: a store zero-fills its tokens, a load leaves the
    pool alone, and the lowest such logical block is reported."""
    spec = PoolSpec(1, 4, 4, 2, 8, 2, HND)
    layers = make_layers(spec, 41, avoid_poison=True)
    table = np.array([1, 4, 2, -1], dtype=np.int32)  # 4 == num_blocks: first id past the end
    chunks = poisoned_chunks(orc, spec, 0, 16, 16)
    rc, bad = orc.store(spec, layers, table, 0, 16, 16, chunks)
    assert rc == oracle.OK and bad == 1, (rc, bad)
    good = do_store(orc, spec, layers, np.array([1, 0, 2, 3], np.int32), 0, 16, 16)
    HR = spec.num_heads * spec.row_bytes
    got = chunks[0].reshape(2, 16, HR)
    ref = good[0].reshape(2, 16, HR)
    for t in range(16):
        if t // 4 in (1, 3):
            assert np.all(got[:, t] == 0), t
        else:
            assert np.array_equal(got[:, t], ref[:, t]), t
    dest = [np.full_like(layers[0], POISON)]
    rc, bad = orc.load(spec, dest, table, 0, 16, 16, good)
    assert rc == oracle.OK and bad == 1, (rc, bad)
    pages = dest[0].reshape(4, spec.page_bytes)
    assert np.all(pages[0] == POISON) and np.all(pages[3] == POISON)   # pages named by no valid entry
    assert not np.all(pages[1] == POISON) and not np.all(pages[2] == POISON)


def pin_threads_match_single(orc):
    spec = PoolSpec(2, 16, 4, 2, 8, 2, HND)
    layers = make_layers(spec, 43)
    table = synth.permuted_table(16, 13, seed=4)
    one = poisoned_chunks(orc, spec, 8, 13 * 4 - 1, 8)
    many = poisoned_chunks(orc, spec, 8, 13 * 4 - 1, 8)
    assert orc.store(spec, layers, table, 8, 13 * 4 - 1, 8, one, n_threads=1)[0] == oracle.OK
    assert orc.store(spec, layers, table, 8, 13 * 4 - 1, 8, many, n_threads=5)[0] == oracle.OK
    for a, b in zip(one, many):
        assert np.array_equal(a, b)


def pin_state_copy(orc):
    """Recurrent-state snapshot: plain slicing of one slot per layer."""
    L, slots, sb = 3, 5, 64
    layers = [synth.splitmix64_bytes(slots * sb, 50 + l) for l in range(L)]
    obj = np.full(L * sb, POISON, np.uint8)
    assert orc.state_copy(layers, sb, 2, obj, True) == oracle.OK
    assert np.array_equal(obj, np.concatenate([l[2 * sb:3 * sb] for l in layers]))
    dest = [np.full(slots * sb, POISON, np.uint8) for _ in range(L)]
    assert orc.state_copy(dest, sb, 4, obj, False) == oracle.OK
    for d, l in zip(dest, layers):
        assert np.array_equal(d[4 * sb:], l[2 * sb:3 * sb])
        assert np.all(d[:4 * sb] == POISON)
    assert orc.state_copy(dest, sb, 5, obj, False) == oracle.ERANGE


def pin_logical_block_nhd_identity(orc):
    """Logical blocks of P packed pages (Sec. 3.1: 49 pages of 32 tokens per 1,568-token
    block), NHD, identity table, chunk = one logical block: the chunk is the block's P
    pages with the page axis moved inside the K/V axis (np.transpose of [P][2][rest])."""
    for P in (2, 3):
        spec = PoolSpec(1, 4 * P, 4, 3, 8, 2, NHD, P)
        layers = make_layers(spec, 61 + P)
        C = P * spec.block_tokens
        chunks = do_store(orc, spec, layers, np.arange(4, dtype=np.int32), 0, 4 * C, C)
        lb_bytes = P * spec.page_bytes
        for c, ch in enumerate(chunks):
            block = layers[0][c * lb_bytes:(c + 1) * lb_bytes].reshape(P, 2, -1)
            assert np.array_equal(ch, np.transpose(block, (1, 0, 2)).reshape(-1)), (P, c)


def pin_logical_block_table_is_take(orc):
    """Through logical blocks, the table acts as np.take over [blocks][P pages]."""
    for layout in (HND, NHD):
        P = 3
        spec = PoolSpec(2, 6 * P, 4, 2, 8, 2, layout, P)
        layers = make_layers(spec, 67)
        table = synth.permuted_table(6, 5, seed=8)
        C = 2 * spec.block_tokens  # chunks that end inside a logical block
        t1 = 5 * P * spec.block_tokens - 5
        got = do_store(orc, spec, layers, table, 0, t1, C)
        taken = [np.take(l.reshape(6, P * spec.page_bytes), table, axis=0).reshape(-1) for l in layers]
        spec5 = PoolSpec(2, 5 * P, 4, 2, 8, 2, layout, P)
        want = do_store(orc, spec5, taken, np.arange(5, dtype=np.int32), 0, t1, C)
        for a, b in zip(got, want):
            assert np.array_equal(a, b), layout
        # a table of logical blocks covers P pages per entry, no more
        ch = poisoned_chunks(orc, spec, 0, 6 * P * 4, C)  # full-size chunks, more than enough
        assert orc.store(spec, layers, table, 0, 5 * P * 4, C, ch)[0] == oracle.OK
        assert orc.store(spec, layers, table, 0, 5 * P * 4 + 1, C, ch)[0] == oracle.ERANGE
        bad = PoolSpec(2, 6 * P + 1, 4, 2, 8, 2, layout, P)  # pool not a whole number of blocks
        assert orc.store(bad, [np.zeros(bad.layer_bytes, np.uint8)] * 2, table, 0, 8, C, ch)[0] == oracle.EALIGN


PINS = [
    pin_logical_block_nhd_identity,
    pin_logical_block_table_is_take,
    pin_nhd_identity_is_page_bytes,
    pin_hnd_identity_is_transpose,
    pin_table_is_take,
    pin_round_trip_bijective,
    pin_untouched_bytes,
    pin_chunk_boundaries,
    pin_hand_example,
    pin_bruteforce_vs_numpy,
    pin_error_codes,
    pin_bad_block,
    pin_threads_match_single,
    pin_state_copy,
]


def run_all(orc) -> dict:
    res = {}
    for pin in PINS:
        try:
            pin(orc)
            res[pin.__name__] = True
        except AssertionError:
            res[pin.__name__] = False
    return res


if __name__ == "__main__":
    # python tests/oracle_pins.py <path to a compiled kv_oracle.so>: JSON of pin results
    print(json.dumps(run_all(oracle.COracle(sys.argv[1]))))
