"""The CPU oracle against its pins (no GPU).  See tests/oracle_pins.py."""
import numpy as np
import pytest

import oracle
from paper_2609_15021_gb300 import synth
from oracle_pins import PINS


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(orc, pin):
    pin(orc)


def test_splitmix64_published_values():
    # SplitMix64 with seed 0: first outputs 0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4
    w = synth.splitmix64_bytes(16, 0).view("<u8")
    assert int(w[0]) == 0xE220A8397B1DCDAF
    assert int(w[1]) == 0x6E789E6AA1B965F4


def test_paper_chunk_geometry(orc):
    """Table 1 / Sec. 3.1: 1,568-token chunks of 32-token pages are 49 pages; with the
    paper's 16 full-attention layers, 4 KV heads, head_dim 256 and FP8 (1 byte) KV, a
    token costs 16*2*4*256 = 32,768 bytes and a chunk 1,568 * 32,768 = 51,380,224 bytes."""
    spec = oracle.PoolSpec(16, 1262 * 49, 32, 4, 256, 1, oracle.HND)
    assert 1568 % spec.block_tokens == 0 and 1568 // spec.block_tokens == 49
    assert orc.chunk_bytes(spec, 1) == 32768
    assert orc.chunk_bytes(spec, 1568) == 51_380_224


def test_numpy_oracle_random_configs(orc):
    """The two formulations agree on random shapes, ragged ranges and both layouts."""
    r = synth.rng(2024)
    for trial in range(40):
        layout = int(r.integers(0, 2))
        B = int(r.choice([1, 2, 4, 16]))
        H = int(r.integers(1, 5))
        D = int(r.choice([1, 8, 16, 64]))
        e = int(r.choice([1, 2, 4]))
        N = int(r.integers(2, 20))
        L = int(r.integers(1, 4))
        spec = oracle.PoolSpec(L, N, B, H, D, e, layout)
        n_used = int(r.integers(1, N + 1))
        table = synth.permuted_table(N, n_used, seed=trial)
        C = B * int(r.integers(1, 4))
        n_chunks_total = (n_used * B + C - 1) // C
        c0 = int(r.integers(0, n_chunks_total))
        t0 = c0 * C
        t1 = int(r.integers(t0, n_used * B + 1))
        layers = [synth.splitmix64_bytes(spec.layer_bytes, 1000 * trial + l) for l in range(L)]
        chunks = [np.full(orc.chunk_bytes(spec, n), synth.POISON, np.uint8)
                  for n in oracle.chunk_tokens_of(t0, t1, C)]
        rc, bad = orc.store(spec, layers, table, t0, t1, C, chunks)
        assert rc == 0 and bad == -1
        want = oracle.np_store(spec, layers, table, t0, t1, C)
        assert len(want) == len(chunks)
        for a, b in zip(chunks, want):
            assert np.array_equal(a, b), trial
        dest = [np.full_like(l, synth.POISON) for l in layers]
        want_l = oracle.np_load(spec, dest, table, t0, t1, C, chunks)
        rc, bad = orc.load(spec, dest, table, t0, t1, C, chunks)
        assert rc == 0 and bad == -1
        for a, b in zip(dest, want_l):
            assert np.array_equal(a, b), trial
