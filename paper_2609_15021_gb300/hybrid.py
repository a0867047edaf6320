"""Hybrid-model prefixes: paged attention KV plus recurrent-state snapshots.

Paper Sec. 2.2: in a hybrid model the reusable state of a prefix is the K/V
pages of its full-attention layers *and* the recurrent (linear-attention)
state snapshotted at the prefix boundary; the state is opaque bytes, and a
prefix is recovered only with both parts, the snapshot taken exactly at the
boundary being restored.  Table 1 / Sec. 2.1: the shared tier is one pinned
host pool holding fixed-token chunks.

``SharedTier`` is that host pool: chunk ``c`` of a sequence lives at a fixed
slot of one exact-size pinned allocation (``kv_host_alloc``), snapshots live
in a second one keyed by their token boundary.  ``Replica`` is one engine's
paged attention pool, block table and state slots on one GPU.
``store_prefix`` / ``load_prefix`` move a token range and the boundary
snapshot through ``kv_store`` / ``kv_load`` / ``kv_state_store`` /
``kv_state_load``, all ordered on the caller's stream; ``load_prefix``
refuses a range whose chunks or whose boundary snapshot are missing.

All data movement is in libkvxfer; this module only keeps the bookkeeping.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Sequence

from . import kvxfer as k


@dataclass
class HybridShape:
    attn_layers: int = 16          # every 4th of 64 layers is full attention
    state_layers: int = 48         # the rest hold a recurrent state
    block_tokens: int = 16
    kv_heads: int = 8
    head_dim: int = 128
    elem_bytes: int = 2            # bf16 K/V
    recurrent_bytes: int = 16 * 128 * 128 * 4   # fp32 recurrent state: 16 heads x 128 x 128
    conv_bytes: int = 3 * 8192 * 2              # convolution window: 3 past steps x 8192 channels, bf16
    slot_align: int = 4096                      # the page is padded to a multiple of this
    chunk_tokens: int = 256

    @property
    def state_bytes(self) -> int:
        """One recurrent page (Sec. 2.2): recurrent state, convolution state and padding,
        moved as opaque bytes."""
        raw = self.recurrent_bytes + self.conv_bytes
        return -(-raw // self.slot_align) * self.slot_align

    @property
    def page_bytes(self) -> int:
        return 2 * self.kv_heads * self.block_tokens * self.head_dim * self.elem_bytes

    @property
    def chunk_bytes(self) -> int:
        return self.attn_layers * 2 * self.chunk_tokens * self.kv_heads * self.head_dim * self.elem_bytes

    @property
    def snapshot_bytes(self) -> int:
        return self.state_layers * self.state_bytes


class SharedTier:
    """Pinned host pool: fixed chunk slots for one sequence plus boundary snapshots."""

    def __init__(self, shape: HybridShape, max_tokens: int, max_snapshots: int):
        self.shape = shape
        self.max_chunks = -(-max_tokens // shape.chunk_tokens)
        self.chunks = k.HostBuffer(self.max_chunks * shape.chunk_bytes)
        self.snaps = k.HostBuffer(max_snapshots * shape.snapshot_bytes)
        self.max_snapshots = max_snapshots
        self.present: set[int] = set()              # chunk indices stored
        self.snapshot_slot: dict[int, int] = {}      # boundary token -> slot, oldest first
        self._free_snaps = list(range(max_snapshots))
        cb = shape.chunk_bytes
        self._chunk_views = [self.chunks.tensor[c * cb:(c + 1) * cb] for c in range(self.max_chunks)]
        # Raw addresses of the slots, each exactly one chunk long (the library still
        # checks that every chunk it is given is pinned host memory).
        self._chunk_ptrs = [v.data_ptr() for v in self._chunk_views]

    def chunk(self, c: int):
        return self._chunk_views[c]

    def chunk_ptrs(self, c0: int, c1: int) -> list[int]:
        """Host addresses of chunk slots c0 .. c1-1."""
        return self._chunk_ptrs[c0:c1]

    def snapshot(self, boundary: int):
        sb = self.shape.snapshot_bytes
        s = self.snapshot_slot[boundary]
        return self.snaps.tensor[s * sb:(s + 1) * sb]

    def reserve_snapshot(self, boundary: int):
        """Host slot for the snapshot at `boundary`; evicts the oldest boundary when full.
        Slots are reused, so tier operations must be ordered on one stream (or synchronised)."""
        if boundary not in self.snapshot_slot:
            if not self._free_snaps:
                oldest = next(iter(self.snapshot_slot))
                self._free_snaps.append(self.snapshot_slot.pop(oldest))
            self.snapshot_slot[boundary] = self._free_snaps.pop(0)
        return self.snapshot(boundary)

    def has_prefix(self, t0: int, t1: int) -> bool:
        C = self.shape.chunk_tokens
        chunks = all(c in self.present for c in range(t0 // C, -(-t1 // C)))
        return chunks and t1 in self.snapshot_slot

    def close(self):
        self._chunk_views = []
        self._chunk_ptrs = []
        self.chunks.close()
        self.snaps.close()


@dataclass
class Replica:
    """One replica's paged attention KV, block table and recurrent-state slots on a GPU."""

    shape: HybridShape
    num_blocks: int
    state_slots: int
    free_pages: Sequence[int]                  # allocation order (seeded by the caller)
    device: str = "cuda"
    table: list[int] = field(default_factory=list)
    tokens: int = 0                            # context length held locally

    def __post_init__(self):
        import numpy as np
        import torch
        s = self.shape
        self._free = np.asarray(self.free_pages, dtype=np.int32)  # taken from the front by a cursor
        self._next_free = 0
        self.attn_layers = [torch.empty(self.num_blocks * s.page_bytes, dtype=torch.uint8, device=self.device)
                            for _ in range(s.attn_layers)]
        self.pool = k.KvPool(self.attn_layers, self.num_blocks, s.block_tokens, s.kv_heads, s.head_dim,
                             s.elem_bytes)
        self.state = [torch.empty(self.state_slots * s.state_bytes, dtype=torch.uint8, device=self.device)
                      for _ in range(s.state_layers)]
        self.state_layers = k.StateLayers(self.state)
        # The block table only grows (pages are appended), so it lives on the
        # device at its largest size and each new entry is uploaded once, on the
        # caller's stream, from a pinned staging copy written once (when the page
        # is allocated).
        self._table_dev = torch.empty(self.num_blocks, dtype=torch.int32, device=self.device)
        self._table_pinned = torch.empty(self.num_blocks, dtype=torch.int32).pin_memory()
        self._table_np = self._table_pinned.numpy()
        self._uploaded = 0

    def grow(self, n_tokens: int):
        """Allocate fresh pages so the table covers n_tokens."""
        need = -(-n_tokens // self.shape.block_tokens)
        have = len(self.table)
        if need <= have:
            return
        take = need - have
        if self._next_free + take > len(self._free):
            raise MemoryError(f"replica has {len(self._free) - self._next_free} free pages, needs {take}")
        new = self._free[self._next_free:self._next_free + take]
        self._next_free += take
        self._table_np[have:need] = new
        self.table.extend(new.tolist())

    def table_tensor(self, stream=None):
        """Device view of the table; entries added since the last call are copied up
        on `stream` (default: the current stream), ahead of the work that uses them."""
        n = len(self.table)
        if self._uploaded < n:
            a = self._uploaded
            src, dst = self._table_pinned[a:n], self._table_dev[a:n]
            if stream is None:
                dst.copy_(src, non_blocking=True)
            else:
                import torch
                with torch.cuda.stream(stream):
                    dst.copy_(src, non_blocking=True)
            self._uploaded = n
        return self._table_dev[:n]


def store_prefix(ctx, rep: Replica, tier: SharedTier, t0: int, t1: int, state_slot: int, stream=None):
    """Store tokens [t0, t1) of rep and its state (slot state_slot) as the snapshot at t1."""
    s = tier.shape
    C = s.chunk_tokens
    # The snapshot needs no block table, so it is enqueued first: the GPU copies
    # it while the host prepares the KV store (both on the caller's stream).
    snap = tier.reserve_snapshot(t1)
    k.kv_state_store(ctx, rep.state_layers, rep.state_slots, s.state_bytes, state_slot, snap, stream=stream)
    chunks = tier.chunk_ptrs(t0 // C, -(-t1 // C))
    k.kv_store(ctx, rep.pool, rep.table_tensor(stream), t0, t1, C, chunks, stream=stream)
    tier.present.update(range(t0 // C, -(-t1 // C)))


def load_prefix(ctx, rep: Replica, tier: SharedTier, t0: int, t1: int, state_slot: int, stream=None):
    """Restore tokens [t0, t1) into fresh pages of rep and the snapshot at t1 into state_slot.

    Raises LookupError unless the tier holds every chunk of the range and the
    snapshot at exactly t1 (a hybrid prefix is recoverable only with both)."""
    if not tier.has_prefix(t0, t1):
        raise LookupError(f"shared tier lacks chunks of [{t0}, {t1}) or the state snapshot at {t1}")
    s = tier.shape
    C = s.chunk_tokens
    # The snapshot goes first: the GPU copies it while the host allocates the
    # pages and uploads their table entries for the KV restore behind it.
    k.kv_state_load(ctx, rep.state_layers, rep.state_slots, s.state_bytes, state_slot, tier.snapshot(t1),
                    stream=stream)
    rep.grow(t1)
    chunks = tier.chunk_ptrs(t0 // C, -(-t1 // C))
    k.kv_load(ctx, rep.pool, rep.table_tensor(stream), t0, t1, C, chunks, stream=stream)
    rep.tokens = t1
