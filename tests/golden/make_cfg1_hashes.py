"""Write tests/golden/cfg1_tiny_hashes.txt: per-chunk SHA-256 of the tiny
paged-KV workload (2 layers, 2 KV heads, head_dim 64, bf16, 16-token pages,
a 64-page pool, a 512-token context on 32 pages in seeded random order,
256-token chunks), and of both layers after loading the chunks into a
poisoned pool through a second random table.

Calls only the oracle (the C oracle, checked here against the NumPy one) and
the seeded input generators.  Run from the repository root:

    python tests/golden/make_cfg1_hashes.py
"""
import hashlib
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2609_15021_gb300 import synth  # noqa: E402

OUT = os.path.join(ROOT, "tests", "golden", "cfg1_tiny_hashes.txt")
SPEC = oracle.PoolSpec(2, 64, 16, 2, 64, 2, oracle.HND)
TOKENS, C = 512, 256
SEED_A, SEED_B = synth.SEED, 271828


def inputs():
    """Pool layers, table A (store) and table B (load) of the workload."""
    layers = [synth.normal_bf16_bytes(SPEC.layer_bytes // 2, synth.SEED + 1000 * l) for l in range(SPEC.num_layers)]
    ta = synth.portable_table(SPEC.num_blocks, TOKENS // SPEC.block_tokens, SEED_A)
    tb = synth.portable_table(SPEC.num_blocks, TOKENS // SPEC.block_tokens, SEED_B)
    return layers, ta, tb


def sha(a: np.ndarray) -> str:
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).hexdigest()


def expected():
    """{name: sha256} from the C oracle, after checking it against the NumPy oracle."""
    orc = oracle.c_oracle()
    layers, ta, tb = inputs()
    chunks = [np.full(orc.chunk_bytes(SPEC, n), synth.POISON, np.uint8) for n in oracle.chunk_tokens_of(0, TOKENS, C)]
    rc, _ = orc.store(SPEC, layers, ta, 0, TOKENS, C, chunks)
    assert rc == oracle.OK
    restored = [np.full(SPEC.layer_bytes, synth.POISON, np.uint8) for _ in range(SPEC.num_layers)]
    rc, _ = orc.load(SPEC, restored, tb, 0, TOKENS, C, chunks)
    assert rc == oracle.OK
    np_chunks = oracle.np_store(SPEC, layers, ta, 0, TOKENS, C)
    np_restored = oracle.np_load(SPEC, [np.full(SPEC.layer_bytes, synth.POISON, np.uint8)] * SPEC.num_layers,
                                 tb, 0, TOKENS, C, np_chunks)
    assert all(np.array_equal(a, b) for a, b in zip(chunks, np_chunks))
    assert all(np.array_equal(a, b) for a, b in zip(restored, np_restored))
    out = {f"chunk{i}": sha(c) for i, c in enumerate(chunks)}
    out.update({f"restored_layer{l}": sha(r) for l, r in enumerate(restored)})
    return out


def read(path: str = OUT) -> dict:
    with open(path) as f:
        return dict(line.split() for line in f if line.strip() and not line.startswith("#"))


if __name__ == "__main__":
    oracle.build()
    with open(OUT, "w") as f:
        f.write("# Tiny paged KV: 2 layers x 2 KV heads x head_dim 64, bf16 (synth.normal_bf16_bytes,\n"
                f"# seed {synth.SEED} + 1000 * layer), 16-token HND pages, 64-page pool, 512 tokens on the\n"
                f"# pages synth.portable_table(64, 32, {SEED_A}), 256-token chunks; restored through\n"
                f"# synth.portable_table(64, 32, {SEED_B}) into a pool poisoned with 0x{synth.POISON:02X}.\n"
                "# SHA-256 of each chunk and each restored layer, written by make_cfg1_hashes.py from the oracle.\n")
        for name, h in expected().items():
            f.write(f"{name} {h}\n")
    print(open(OUT).read())
