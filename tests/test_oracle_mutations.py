"""Plant plausible mistakes in copies of the C oracle and check the pins catch each.

Each mutation edits one expression of kv_oracle.c (on the CPU, in a temporary
copy), compiles it, and runs every pin of tests/oracle_pins.py against it in a
subprocess (a planted out-of-bounds access may crash it, which also counts as
caught).  At least one pin other than the comparison with the NumPy
formulation must fail, so each mistake is caught by a fact independent of the
second oracle.
"""
import json
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(os.path.dirname(HERE), "oracle", "kv_oracle.c")

MUTATIONS = {
    "hnd_head_slot_swapped": ("* H + h) * B + s) * row_bytes(P)", "* H + s) * B + h) * row_bytes(P)"),
    "hnd_slot_dropped": ("* H + h) * B + s) * row_bytes(P)", "* H + h) * B + 0) * row_bytes(P)"),
    "nhd_slot_head_swapped": ("* B + s) * H + h) * row_bytes(P)", "* B + h) * H + s) * row_bytes(P)"),
    "hnd_kv_reversed": ("(((p * 2 + kv) * H + h)", "(((p * 2 + (1 - kv)) * H + h)"),
    "chunk_kv_dropped": ("(((l * 2 + kv) * T_c + u) * H + h)", "(((l * 2 + 0) * T_c + u) * H + h)"),
    "chunk_token_head_transposed": ("(((l * 2 + kv) * T_c + u) * H + h)", "(((l * 2 + kv) * H + h) * T_c + u)"),
    "chunk_padded_tail": ("chunk_row(P, T_c, l, kv, u, h)", "chunk_row(P, C, l, kv, u, h)"),
    "block_from_local_token": ("int64_t kpage = t / B;", "int64_t kpage = u / B;"),
    "tail_length_ignored": ("int64_t T_c = (J->t_end - first < C) ? (J->t_end - first) : C;", "int64_t T_c = C;"),
    "load_copies_backwards": ("memcpy(p_ptr, c_ptr, (size_t)row);", "memcpy(c_ptr, p_ptr, (size_t)row);"),
    "chunk_index_ignores_start": ("int64_t c = c0 + i;", "int64_t c = i;"),
    "capacity_off_by_one": ("if (t_end > table_len * ppb_of(P) * (int64_t)P->block_tokens) return OR_ERANGE;",
                            "if (t_end >= table_len * ppb_of(P) * (int64_t)P->block_tokens) return OR_ERANGE;"),
    "capacity_ignores_logical_blocks": ("if (t_end > table_len * ppb_of(P) * (int64_t)P->block_tokens)",
                                        "if (t_end > table_len * (int64_t)P->block_tokens)"),
    "start_alignment_unchecked": ("if (t_begin % C != 0) return OR_EALIGN;", ""),
    "page_bound_off_by_one": ("if (entry < 0 || entry >= P->num_blocks / ppb) {",
                              "if (entry < 0 || entry > P->num_blocks / ppb) {"),
    "logical_block_not_scaled": ("int64_t p = entry * ppb + kpage % ppb;", "int64_t p = entry + kpage % ppb;"),
    "subpage_dropped": ("int64_t p = entry * ppb + kpage % ppb;", "int64_t p = entry * ppb;"),
    "subpage_from_slot": ("int64_t p = entry * ppb + kpage % ppb;", "int64_t p = entry * ppb + s % ppb;"),
    "row_ignores_elem_bytes": ("return (int64_t)P->head_dim * P->elem_bytes;", "return (int64_t)P->head_dim;"),
    "state_slot_offset_dropped": ("uint8_t* s = layers[l] + slot * slot_bytes;", "uint8_t* s = layers[l] + slot_bytes;"),
}


def _run(name, tmpdir):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(old) >= 1, f"mutation {name}: expression not found in kv_oracle.c"
    mutated = src.replace(old, new, 1)
    c_path = os.path.join(tmpdir, f"{name}.c")
    so_path = os.path.join(tmpdir, f"{name}.so")
    with open(c_path, "w") as f:
        f.write(mutated)
    oracle.build(c_path, so_path, force=True)
    r = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py"), so_path],
                       capture_output=True, text=True, timeout=300)
    if r.returncode != 0:
        return {"crashed": True}
    return json.loads(r.stdout.strip().splitlines()[-1])


@pytest.fixture(scope="module")
def mutation_results(tmp_path_factory):
    d = str(tmp_path_factory.mktemp("mut"))
    with ThreadPoolExecutor(max_workers=8) as ex:
        res = dict(zip(MUTATIONS, ex.map(lambda n: _run(n, d), MUTATIONS)))
    return res


def test_unmutated_copy_passes_every_pin(tmp_path):
    so = os.path.join(str(tmp_path), "clean.so")
    oracle.build(SRC, so, force=True)
    r = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py"), so],
                       capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    assert all(json.loads(r.stdout.strip().splitlines()[-1]).values())


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_mutation_is_caught(mutation_results, name):
    res = mutation_results[name]
    if res.get("crashed"):
        return
    independent = {k: v for k, v in res.items() if k != "pin_bruteforce_vs_numpy"}
    assert not all(independent.values()), f"{name} survived every independent pin: {res}"
