"""Literal Algorithm 1 for tiny inputs, independent of the oracle.

Pure Python, written differently from the oracle on purpose: it scans every
j' from the sequence start (no use of the length bound K) and tests
membership by a linear scan over the f-gram list (no map), so it pins the
oracle's window bound and its dictionary.
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
