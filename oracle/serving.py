"""Oracle for the serving-side placement of a repaired cache, in plain numpy.

TEST INFRASTRUCTURE, like the rest of this package: imported only by the
tests; the product path never imports it.

  App. A  "Online execution and timing": the repaired document prefix is
          injected into the serving engine's paged cache, loaded through the
          last complete 16-token cache block; the document tokens after that
          block are left to the query pass.
  Sec. 4.1 / R9  A repaired row is token-major, D_KV = 2 L H_kv d_h wide,
          coordinate j = ((layer * 2 + kv) * H_kv + head) * d_h + d.

Reading (R26): the paged target cache is layer-major, one plane per
(layer, K|V) pair, plane p = layer * 2 + kv holding [num_slots, H_kv * d_h];
slot s of a plane is block s // block_size, offset s % block_size, and a
request's blocks are listed in its block table (the vLLM layout).  A token
whose slot is negative is not written; every slot no token maps to keeps its
previous contents.
"""
from __future__ import annotations

import numpy as np

__all__ = ["paged_slot_mapping", "paged_scatter"]


def paged_slot_mapping(n_tokens: int, block_table, block_size: int = 16) -> np.ndarray:
    """Slot of each of a request's n_tokens tokens, or -1 for the tokens after its
    last complete block (App. A: the prefix is loaded through the last complete
    block).  Token t of a complete block lands in slot
    block_table[t // block_size] * block_size + t % block_size."""
    table = np.asarray(block_table, np.int64)
    n_full = (n_tokens // block_size) * block_size
    if len(table) < n_full // block_size:
        raise ValueError("the block table has fewer blocks than the request's complete blocks")
    slots = np.full(n_tokens, -1, np.int64)
    for t in range(n_full):
        slots[t] = table[t // block_size] * block_size + t % block_size
    return slots


def paged_scatter(rows: np.ndarray, slot_mapping: np.ndarray, paged: np.ndarray, n_layers: int,
                  n_kv_heads: int, head_dim: int) -> np.ndarray:
    """Copy of `paged` ([2 L, num_slots, H_kv d_h]) with each token's row written to
    its slot: row t's columns [p W, (p + 1) W), W = H_kv d_h, go to plane p at slot
    slot_mapping[t] (R9, R26).  Tokens with a negative slot are skipped; a slot
    outside the planes is an error.  rows: [N, D_KV] in any dtype `paged` holds."""
    planes, num_slots, width = paged.shape
    if planes != 2 * n_layers or width != n_kv_heads * head_dim:
        raise ValueError("paged cache shape does not match the target")
    if rows.shape[1] != planes * width or len(slot_mapping) != rows.shape[0]:
        raise ValueError("rows and slot mapping do not match")
    out = paged.copy()
    for t, s in enumerate(np.asarray(slot_mapping, np.int64)):
        if s < 0:
            continue
        if s >= num_slots:
            raise IndexError(f"token {t}: slot {s} outside the {num_slots} slots")
        for p in range(planes):
            out[p, s] = rows[t, p * width:(p + 1) * width]
    return out
