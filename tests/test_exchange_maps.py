"""Exhaustive host checks of the lane mappings that let the kernels replace CTA
barriers by warp barriers.  Each check restates the index formulas of the kernel it
covers and proves the property the kernel relies on:

* n = 4096 (16 x 16 x 16, 256 threads): the last-pass frequency groups form a
  permutation of 0..255 with every M partner group (256 - K) at lane ^ 16, except
  the self-paired groups 0 and 128 (lanes 0 and 16 of warp 0); each warp's pass-1
  groups lie in exactly the two pass-0 blocks its last-pass groups use; and every
  half-warp access of pass 1 and of the last pass hits distinct bank pairs.
* n = 11008 (43 x 16 x 16, 256 threads, groups dealt round-robin): pass 1 and the
  last pass touch each slot from the same half-warp.
* the randomized-Hadamard rotation: the exchange between passes 0 and 1 moves data
  only inside a half-warp, and pass 1's writes into the next exchange land only on
  slots the same half-warp read before, for every block size with three or more
  passes, forward and inverse."""

import pytest


def pad(i):
    return i + (i >> 4) + (i >> 8)


def warp_local_4096():
    """(frequency group K, pass-1 group g1) of each of the 256 threads."""
    out = []
    for lt in range(256):
        w, l = divmod(lt, 32)
        h, i = divmod(l, 16)
        bb = (16 * i if i < 8 else 16 * i - 120) if w == 0 else w + 16 * i
        k = (256 - bb if bb else 128) if h else bb
        g1 = ((8 * h) if w == 0 else (16 - w if h else w)) * 16 + i
        out.append((k, g1))
    return out


def test_n4096_groups_pair_across_lanes():
    m = warp_local_4096()
    assert sorted(k for k, _ in m) == list(range(256))
    assert sorted(g for _, g in m) == list(range(256))
    for lt, (k, _) in enumerate(m):
        partner = m[lt ^ 16][0]
        if lt in (0, 16):
            assert k == (0 if lt == 0 else 128)
        else:
            assert (k + partner) % 256 == 0 and k != partner


def test_n4096_warp_owns_its_blocks():
    m = warp_local_4096()
    for w in range(8):
        last = {m[lt][0] % 16 for lt in range(32 * w, 32 * w + 32)}    # pass-0 digit = block
        first = {m[lt][1] // 16 for lt in range(32 * w, 32 * w + 32)}
        assert last == first and len(last) == 2


def test_n4096_accesses_conflict_free():
    m = warp_local_4096()
    for w in range(8):
        for h in range(2):
            lanes = range(32 * w + 16 * h, 32 * w + 16 * h + 16)
            for j in range(16):
                last = [pad((m[lt][0] % 16) * 256 + (m[lt][0] // 16) * 16 + j) for lt in lanes]
                p1 = [pad((m[lt][1] // 16) * 256 + m[lt][1] % 16 + 16 * j) for lt in lanes]
                assert len({a % 16 for a in last}) == 16 and len({a % 16 for a in p1}) == 16


def test_n11008_pass1_and_last_pass_share_half_warps():
    n, t_count = 11008, 256
    owner1, owner2 = {}, {}
    for g in range(n // 16):
        t = g % t_count
        blk, np_ = divmod(g, 16)
        for j in range(16):
            owner1[blk * 256 + np_ + 16 * j] = t     # pass 1: radix 16 at stride 16 in 256-slot blocks
            owner2[g * 16 + j] = t                   # last pass: 16 contiguous slots
    assert len(owner1) == len(owner2) == n
    assert all(owner1[i] // 16 == owner2[i] // 16 for i in range(n))


def _radix(lb, k):
    return 16 if lb - 4 * k >= 4 else 1 << (lb - 4 * k)


def _base(lb, k, t):
    s = 1 << (4 * k)
    if k == 0:
        return 16 * t
    return (t & (s - 1)) + 16 * s * (t // s) if _radix(lb, k) == 16 else t


def _off(lb, k, e):
    tb, s, r = (1 << lb) // 16, 1 << (4 * k), _radix(lb, k)
    return e if k == 0 else (s * e if r == 16 else tb * (e // r) + s * (e % r))


def _rpad(x, i):
    return i + (i >> 4) if x == 0 else i + ((i >> (4 * x + 4)) << 4)


@pytest.mark.parametrize("log_b", range(9, 17))
@pytest.mark.parametrize("inverse", [False, True])
def test_rht_exchange_locality(log_b, inverse):
    npass, tb = (log_b + 3) // 4, (1 << log_b) // 16
    order = list(range(npass))[::-1] if inverse else list(range(npass))
    prev_reader = None   # slot -> thread that read it in the previous exchange
    for ki in range(1, npass):
        k, kp = order[ki], order[ki - 1]
        x = min(k, kp)
        writer, reader = {}, {}
        for t in range(tb):
            for e in range(16):
                writer[_rpad(x, _base(log_b, kp, t) + _off(log_b, kp, e))] = t
                reader[_rpad(x, _base(log_b, k, t) + _off(log_b, k, e))] = t
        assert len(writer) == len(reader) == 16 * tb and set(writer) == set(reader)
        if x == 0:       # read-after-write inside the half-warp
            assert all(writer[slot] // 16 == t // 16 for slot, t in reader.items())
        if kp == 1 and ki >= 2:   # write-after-read inside the half-warp
            assert all(prev_reader[slot] // 16 == t // 16 for slot, t in writer.items() if slot in prev_reader)
        prev_reader = reader


# n = 11008 = 43 x 16 x 16 with warp-local units: after the 43-point pass the vector
# falls into 43 blocks of 256 slots (one per pass-0 output digit b); the M partner of
# every frequency of block b lies in block 43 - b (block 0 pairs with itself).  Unit 0
# is block 0, unit u >= 1 the blocks u and 43 - u; warp w takes units w, w + 8, w + 16.
# In a unit, lane l < 16 takes group i = l of the first block and lane l >= 16 group
# i = 31 - l of the second (unit 0: lanes 0..15 only).  Pass 1 works on the group
# (block b, np = i) at slots 256 b + i + 16 j, the last pass on the group (b, k1 = i)
# at slots 256 b + 16 i + k2, holding frequencies b + 43 i + 688 k2.

def units_11008():
    """(warp, q, lane, block, i, active) for every unit a warp processes."""
    out = []
    for w in range(8):
        for q in range(3):
            u = w + 8 * q
            if u >= 22:
                continue
            for l in range(32):
                if u == 0:
                    out.append((w, q, l, 0, l % 16, l < 16))
                else:
                    out.append((w, q, l, u if l < 16 else 43 - u, l if l < 16 else 31 - l, True))
    return out


def test_n11008_units_cover_every_group_once():
    seen = [(b, i) for (_, _, _, b, i, act) in units_11008() if act]
    assert sorted(seen) == [(b, i) for b in range(43) for i in range(16)]


def test_n11008_partners_in_registers():
    n = 11008
    by = {(w, q, l): (b, i, act) for (w, q, l, b, i, act) in units_11008()}
    for (w, q, l), (b, i, act) in by.items():
        if not act:
            continue
        u = w + 8 * q
        for k2 in range(16):
            k = b + 43 * i + 688 * k2
            if u == 0:
                if i == 0:       # own register (16 - k2) % 16
                    assert (n - k) % n == 688 * ((16 - k2) % 16)
                else:            # lane 16 - l, register 15 - k2
                    b2, i2, _ = by[(w, q, 16 - l)]
                    assert b2 + 43 * i2 + 688 * (15 - k2) == n - k
            else:                # lane l ^ 16, register 15 - k2
                b2, i2, _ = by[(w, q, l ^ 16)]
                assert b2 + 43 * i2 + 688 * (15 - k2) == n - k


def test_n11008_unit_accesses_conflict_free():
    """Every half-warp access of pass 1 (per j) and of the last pass (per k2) hits 16
    distinct bank pairs (8-byte slots: 32 four-byte banks)."""
    groups = {}
    for (w, q, l, b, i, act) in units_11008():
        if act:
            groups.setdefault((w, q, l // 16), []).append((b, i))
    for g in groups.values():
        for j in range(16):
            banks = {(2 * pad(256 * b + i + 16 * j)) % 32 for b, i in g}
            assert len(banks) == len(g)
            banks = {(2 * pad(256 * b + 16 * i + j)) % 32 for b, i in g}
            assert len(banks) == len(g)
