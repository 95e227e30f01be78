"""The rule that reassembles a user's sketch from the pieces left by workers
whose tile ranges cut it (host model of the finalize step; no GPU)."""
import numpy as np


def range_begin(total, W, w):
    return (total * w) // W


def owner(total, W, t):
    return max(w for w in range(W) if range_begin(total, W, w) <= t)


def test_pieces_tile_each_segment_exactly():
    rng = np.random.default_rng(1)
    for trial in range(40):
        B = int(rng.integers(1, 12))
        H = int(rng.integers(1, 4))
        tiles = rng.integers(0, 9, size=B)
        prefix = np.concatenate([[0], np.cumsum(tiles)])
        tph = int(prefix[-1])
        total = tph * H
        W = int(rng.integers(1, 40))
        if total == 0:
            continue
        # what each worker writes: (segment, slot) -> set of tiles
        written = {}
        for w in range(W):
            tb, te = range_begin(total, W, w), range_begin(total, W, w + 1)
            t = tb
            while t < te:
                h, rem = divmod(t, tph)
                b = int(np.searchsorted(prefix, rem, side="right") - 1)
                s0, s1 = h * tph + prefix[b], h * tph + prefix[b + 1]
                end = min(s1, te)
                whole = s0 >= tb and s1 <= te
                slot = None if whole else (0 if tb >= s0 else 1)
                key = (w, slot)
                assert whole or key not in written, "two pieces in one slot"
                written[key] = (s0, s1, set(range(t, end)))
                t = end
        for h in range(H):
            for b in range(B):
                s0, s1 = h * tph + prefix[b], h * tph + prefix[b + 1]
                if s0 == s1:
                    continue
                g0, g1 = owner(total, W, s0), owner(total, W, s1 - 1)
                if g0 == g1:
                    assert (g0, None) in written
                    continue
                covered = set()
                for g in range(g0, g1 + 1):
                    if range_begin(total, W, g) == range_begin(total, W, g + 1):
                        continue
                    slot = 0 if range_begin(total, W, g) >= s0 else 1
                    seg = written[(g, slot)]
                    assert seg[0] == s0 and seg[1] == s1
                    assert not (covered & seg[2])
                    covered |= seg[2]
                assert covered == set(range(s0, s1))
