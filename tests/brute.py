"""Literal Algorithms 1 and 3 for tiny inputs, independent of the oracle.

Pure Python, written differently from the oracle on purpose: it scans every
j' from the sequence start (no use of the length bound K) and tests
membership by a linear scan over the f-gram list (no map), so it pins the
oracle's window bound and its dictionary. For Algorithm 3 it enumerates every
n-gram over the vocabulary and counts it against every window, where the
oracle counts the windows it sees in a map.
"""

from typing import List, Sequence, Tuple


def find_fgram(fgrams: Sequence[Tuple[int, ...]], window: Tuple[int, ...]):
    for r, g in enumerate(fgrams):
        if tuple(g) == window:
            return r
    return None


def alg1_sequence(seq: Sequence[int], fgrams: Sequence[Tuple[int, ...]], vocab: int):
    """Returns (rows, lens) for one sequence; invalid token -> (-1, 0)."""
    rows: List[int] = []
    lens: List[int] = []
    for i in range(len(seq)):
        if not 0 <= seq[i] < vocab:
            rows.append(-1)
            lens.append(0)
            continue
        j, r = i, -1
        for jp in range(0, i):                 # smallest j' < i first
            hit = find_fgram(fgrams, tuple(seq[jp:i + 1]))
            if hit is not None:
                j, r = jp, hit
                break
        rows.append(r)
        lens.append(i - j + 1)
    return rows, lens


def alg3_counts(seqs: Sequence[Sequence[int]], vocab: int, K: int):
    """Algorithm 3's counting loops, literally: every n-gram over the vocabulary,
    n = 2..K, counted by comparing it with every window of every sequence.
    Returns {gram: (count, start of first occurrence in the flattened corpus)}
    for the grams that appear. Only for tiny vocabularies."""
    from itertools import product

    L = len(seqs[0]) if seqs else 0
    out = {}
    for n in range(2, K + 1):
        for w in product(range(vocab), repeat=n):
            count, first = 0, None
            for b, seq in enumerate(seqs):
                for p in range(len(seq) - n + 1):
                    if tuple(seq[p:p + n]) == w:
                        count += 1
                        if first is None:
                            first = b * L + p
            if count:
                out[w] = (count, first)
    return out


def alg3_select(counts, S: int, min_count: int):
    """The S most frequent grams with count >= min_count; ties by length, then
    first occurrence; listed by length, then first occurrence."""
    cand = [(w, c, f) for w, (c, f) in counts.items() if c >= min_count]
    cand.sort(key=lambda x: (-x[1], len(x[0]), x[2]))
    sel = cand[:S]
    sel.sort(key=lambda x: (len(x[0]), x[2]))
    return sel
