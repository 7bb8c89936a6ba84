"""The compaction's balanced split, checked on the CPU.

A plain restatement of the plan the compaction kernels follow (the moved rows
of all evicting (entry, layer, K|V) streams laid end to end, cut into one
equal chunk per CTA; before the copy, the sources in [a, n_new) that a
chunk's last rows read, where the next chunk begins at row a, are saved in
that chunk's stash), checked by brute force over random kept lists:

* every moved row is copied exactly once;
* no chunk reads, from the cache, a slot another chunk writes (the in-place
  copy needs no wait between CTAs);
* every stash holds at most stash_rows rows and every redirected read lands
  inside it, whenever the admission rule holds -- every entry's largest
  shift kept[n-1] - (n-1) is at most stash_rows, or no chunk is longer than
  stash_rows;
* the rows to stash lie in the window the kernel searches, [max(segment
  start, a - stash_rows), a).
A pair is an evicting entry (its 2L streams; token budgets) or an (entry,
layer) pair (its K and V streams; per-layer budgets), where a layer may move
nothing.
"""
import numpy as np
import pytest


def _plan(kept_lists, fes, ns, L, G, stash_rows):
    lens = [n - fe for n, fe in zip(ns, fes)]
    upe = 2 * L
    pre = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    n_ev = len(lens)
    total = int(pre[n_ev] * upe)
    shifts_ok = all(kept_lists[e][ns[e] - 1] - (ns[e] - 1) <= stash_rows for e in range(n_ev) if lens[e])
    chunk_ok = -(-total // G) <= stash_rows
    if not (shifts_ok or chunk_ok):
        return None

    def locate(o):
        e = int(np.searchsorted(pre[1:] * upe, o, side="right"))
        rel = o - int(pre[e]) * upe
        q, r = divmod(rel, lens[e])
        return e, q, r

    stash = {}
    for g in range(1, G):
        o = g * total // G
        if o >= total:
            continue
        e, q, r = locate(o)
        if r == 0:
            continue
        fe, n_new, kl = fes[e], ns[e], kept_lists[e]
        a = fe + r
        s0 = int(pre[e]) * upe + q * lens[e]
        seg_start = fe + max(0, (g - 1) * total // G - s0)
        lo = max(seg_start, a - stash_rows)
        need = [i for i in range(seg_start, a) if kl[i] >= a]
        assert need == [i for i in range(lo, a) if kl[i] >= a], "a row to stash outside the searched window"
        i0 = lo + sum(1 for i in range(lo, a) if kl[i] < a)
        i1 = lo + sum(1 for i in range(lo, a) if kl[i] < n_new)
        assert i1 - i0 <= stash_rows
        stash[g] = (e, q, a, i0, i1 - i0)

    writes, reads, done = {}, [], {}
    for g in range(G):
        o, o_stop = g * total // G, (g + 1) * total // G
        while o < o_stop:
            e, q, r = locate(o)
            fe, n_new, kl = fes[e], ns[e], kept_lists[e]
            i, rest = fe + r, lens[e] - r
            if o_stop - o < rest:
                end, stash_at = i + (o_stop - o), i + (o_stop - o)
            else:
                end, stash_at = i + rest, None
            for row in range(i, end):
                src = kl[row]
                assert src >= row
                writes[(e, q, row)] = g
                if stash_at is not None and stash_at <= src < n_new:
                    se, sq, sa, i0, cnt = stash[g + 1]
                    assert (se, sq, sa) == (e, q, stash_at) and 0 <= row - i0 < cnt
                else:
                    reads.append((g, e, q, src))
                done[(e, q, row)] = done.get((e, q, row), 0) + 1
            o += end - i
    for g, e, q, src in reads:
        assert writes.get((e, q, src), g) == g, "a chunk reads a slot another chunk writes"
    assert sorted(done.values()) == [1] * total
    return "shift" if shifts_ok else "chunk"


def _random_eviction(rng, small_shift):
    n_old = int(rng.integers(2, 1500))
    ev = int(rng.integers(1, min(n_old, 40))) if small_shift else int(rng.integers(1, n_old))
    drop = rng.choice(n_old, ev, replace=False)
    keep = np.setdiff1d(np.arange(n_old), drop)
    n_new = n_old - ev
    fe = next((i for i in range(n_new) if keep[i] != i), n_new)
    return keep, fe, n_new


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_balanced_split_plan_has_no_cross_cta_hazard(seed):
    rng = np.random.default_rng(seed)
    seen = {"shift": 0, "chunk": 0, None: 0}
    for _ in range(250):
        kl, fes, ns = [], [], []
        for _ in range(int(rng.integers(1, 4))):
            if rng.random() < 0.2:   # a pair that moves nothing (a layer that did not evict)
                n = int(rng.integers(1, 50))
                kl.append(np.arange(n)), fes.append(n), ns.append(n)
                continue
            keep, fe, n_new = _random_eviction(rng, rng.random() < 0.5)
            kl.append(keep), fes.append(fe), ns.append(n_new)
        if sum(n - fe for n, fe in zip(ns, fes)) == 0:
            continue
        L = int(rng.integers(1, 4))
        G = int(rng.choice([1, 3, 19, 64, 304]))
        seen[_plan(kl, fes, ns, L, G, int(rng.choice([8, 32, 128])))] += 1
    assert seen["shift"] > 20 and seen["chunk"] > 5 and seen[None] > 5


def test_one_large_eviction_is_admitted_by_its_short_chunks():
    """The 2,048 -> 512 single-sequence eviction: 64 streams of ~500 moved
    rows over 304 CTAs give chunks of ~105 rows, within the stash, although
    the shift is 1,536."""
    rng = np.random.default_rng(9)
    keep = np.sort(np.concatenate([rng.choice(1920, 384, replace=False), np.arange(1920, 2048)]))
    fe = next(i for i in range(512) if keep[i] != i)
    assert keep[-1] - 511 == 1536
    assert _plan([keep], [fe], [512], 32, 304, 128) == "chunk"
