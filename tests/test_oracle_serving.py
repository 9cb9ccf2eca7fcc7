"""Pins of the paged-cache placement oracle (App. A serving setup; R9, R26)
against hand-built cases whose expected slots and planes are written out here."""
import numpy as np
import pytest

import oracle as O


def test_slot_mapping_hand_built_three_blocks():
    # 40 tokens, 16-token blocks: two complete blocks (32 tokens), an 8-token tail
    # that is not loaded; the request's blocks are physical blocks 2, 0, 5
    s = O.paged_slot_mapping(40, [2, 0, 5])
    assert s[0] == 32 and s[15] == 47          # block 2 holds tokens 0..15
    assert s[16] == 0 and s[31] == 15          # block 0 holds tokens 16..31
    assert np.all(s[32:] == -1)                # third block incomplete: not written
    assert len(set(s[:32].tolist())) == 32
    # an exact multiple of the block size loads every token
    assert np.all(O.paged_slot_mapping(32, [1, 3]) >= 0)
    # shorter than one block: nothing is loaded
    assert np.all(O.paged_slot_mapping(15, [4]) == -1)
    with pytest.raises(ValueError):
        O.paged_slot_mapping(48, [0, 1])


def test_scatter_hand_built_layer_major_planes():
    # L = 1, H_kv = 2, d_h = 2: D_KV = 8, planes K (p = 0) and V (p = 1), 4 columns each
    L, H, dh = 1, 2, 2
    n = 3
    rows = np.array([[10 * t + j for j in range(8)] for t in range(n)], np.float64)
    slots = np.array([5, -1, 0])
    paged = np.full((2, 6, 4), -7.0)
    out = O.paged_scatter(rows, slots, paged, L, H, dh)
    # token 0 -> slot 5: K columns 0..3 in plane 0, V columns 4..7 in plane 1
    assert out[0, 5].tolist() == [0, 1, 2, 3] and out[1, 5].tolist() == [4, 5, 6, 7]
    # token 2 -> slot 0
    assert out[0, 0].tolist() == [20, 21, 22, 23] and out[1, 0].tolist() == [24, 25, 26, 27]
    # token 1 is skipped; every slot nobody maps to keeps its contents
    for s in (1, 2, 3, 4):
        assert np.all(out[:, s] == -7.0)
    assert np.all(paged == -7.0)               # the input is not modified
    with pytest.raises(IndexError):
        O.paged_scatter(rows, np.array([0, 1, 6]), paged, L, H, dh)


def test_scatter_then_gather_is_the_identity_on_loaded_tokens():
    # two layers, 16-token blocks in a shuffled table: reading each loaded token's
    # slot back out of every plane rebuilds its row (coordinate order of R9)
    L, H, dh = 2, 2, 4
    g = np.random.default_rng(0)
    n = 45
    rows = g.standard_normal((n, 2 * L * H * dh))
    table = g.permutation(6)[:3]
    slots = O.paged_slot_mapping(n, table)
    out = O.paged_scatter(rows, slots, np.zeros((2 * L, 6 * 16, H * dh)), L, H, dh)
    for t in range(n):
        if slots[t] < 0:
            continue
        back = np.concatenate([out[p, slots[t]] for p in range(2 * L)])
        assert np.array_equal(back, rows[t])
    assert int((slots >= 0).sum()) == 32
