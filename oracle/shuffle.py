"""Coded shuffling (Sec. IV) in plain Python: TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this module.  It shares no code with the CUDA library: the sets of
Sec. IV are Python sets, Alg. 1 enumerates every worker set I literally, and
sums are exact (fp64 for the real sum of fp32 rows, integers for xor).

What each function follows:
  * ``partition``          Sec. IV-A: a uniformly random partition of [q] into
                           n sets of q/n rows before every iteration;
  * ``initial_caches``     Sec. IV-B: C_i \\ S_i uniform without replacement in
                           [q] \\ S_i (the marginal law of the update rule);
  * ``update_caches``      Sec. IV-B, cache update rule: S_i^{t+1} plus s - q/n
                           rows drawn from C_i^t \\ S_i^{t+1};
  * ``exclusive_cache``    Sec. IV-B: C~_I, rows cached at every worker of I
                           and at no other;
  * ``encode``             Alg. 1: for every I with |I| >= 2, the sum over
                           i in I of the zero-padded blocks A(S_i & C~_{I\\{i}});
  * ``decode``             Sec. IV-B decoding: worker i subtracts from every
                           message of an I containing i the rows of the other
                           blocks, which it caches;
  * ``uncoded_rate``       eq. for R_u;
  * ``coded_rate``         coded shuffling rate theorem (closed form);
  * ``coded_rate_series``  the sum over |I| in the theorem's proof.

Random draws (passed to both sides by their published definition, SplitMix64:
Steele, Lea, Flood, OOPSLA 2014): iteration t's partition orders the rows by
(key(partition_seed, t q + r), r) and gives positions [i q/n, (i+1) q/n) to
worker i; a refill of cache i at iteration t keeps the s - q/n candidates with
the smallest (key(cache_seed, (t n + i) q + r), r).

Parity pins (``tests/test_shuffle_oracle.py``): the n = 3 example of Sec.
IV-C worked by hand (golden file), a brute-force regrouping of the needed rows
by the set of their holders, the theorem's closed form against its series,
the printed 81 % reduction, both corollaries, the exact expectation of the
uncoded count, the marginal cache law, and the simulated coded count against
the theorem in its large-q regime.
"""
from __future__ import annotations

import itertools
import math

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def splitmix64(seed: int, index: int) -> int:
    """Output `index` of the SplitMix64 stream at `seed` (index 1 = first)."""
    z = (seed + index * GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def _keys(seed: int, first: int, count: int) -> list[int]:
    return [splitmix64(seed, first + r) for r in range(count)]


def partition(partition_seed: int, t: int, n: int, q: int) -> list[set[int]]:
    """S_1^t .. S_n^t (0-based workers): rows ordered by their keys."""
    keys = _keys(partition_seed, t * q, q)
    order = sorted(range(q), key=lambda r: (keys[r], r))
    per = q // n
    return [set(order[i * per:(i + 1) * per]) for i in range(n)]


def _draw(cache_seed: int, t: int, n: int, q: int, i: int, candidates, count: int) -> set[int]:
    ranked = sorted(candidates, key=lambda r: (splitmix64(cache_seed, (t * n + i) * q + r), r))
    return set(ranked[:count])


def initial_caches(cache_seed: int, S: list[set[int]], q: int, s: int) -> list[set[int]]:
    n = len(S)
    extra = s - q // n
    return [S[i] | _draw(cache_seed, 0, n, q, i, set(range(q)) - S[i], extra) for i in range(n)]


def update_caches(cache_seed: int, t1: int, C: list[set[int]], S1: list[set[int]], q: int,
                  s: int) -> list[set[int]]:
    """C^{t+1} from C^t and the new partition S^{t+1}."""
    n = len(C)
    extra = s - q // n
    return [S1[i] | _draw(cache_seed, t1, n, q, i, C[i] - S1[i], extra) for i in range(n)]


def exclusive_cache(C: list[set[int]], I) -> set[int]:
    """C~_I = (intersection of C_i, i in I) minus (union of C_j, j not in I)."""
    I = set(I)
    inside = set.intersection(*[C[i] for i in I])
    outside = set().union(*[C[j] for j in range(len(C)) if j not in I])
    return inside - outside


def worker_sets(n: int):
    """Every I of [n] with |I| >= 2, in ascending order of its bit mask."""
    sets = [I for size in range(2, n + 1) for I in itertools.combinations(range(n), size)]
    return sorted(sets, key=lambda I: sum(1 << i for i in I))


def encode(C, S, A, op: str = "add"):
    """Alg. 1.  A maps a row index to its data (fp32 array, or uint32 for xor).

    Returns a list of (I, blocks, message): blocks[i] lists the rows of
    S_i & C~_{I\\{i}} in ascending order (the rows of B_i before padding);
    message is the ell x r sum of the zero-padded blocks (fp64 for "add",
    uint32 for "xor").  Sets I whose blocks are all empty send nothing."""
    out = []
    r = len(next(iter(A.values()))) if isinstance(A, dict) else A.shape[1]
    for I in worker_sets(len(C)):
        blocks = {i: sorted(S[i] & exclusive_cache(C, set(I) - {i})) for i in I}
        ell = max(len(b) for b in blocks.values())
        if ell == 0:
            continue
        if op == "add":
            msg = np.zeros((ell, r), np.float64)
            for i in I:
                for j, row in enumerate(blocks[i]):
                    msg[j] += np.asarray(A[row], np.float64)
        else:
            msg = np.zeros((ell, r), np.uint32)
            for i in I:
                for j, row in enumerate(blocks[i]):
                    msg[j] ^= np.asarray(A[row], np.uint32)
        out.append((tuple(I), blocks, msg))
    return out


def decode(i: int, messages, cache_rows: dict, op: str = "add") -> dict:
    """Rows of S_i missing from cache i, recovered by worker i alone.

    cache_rows maps each row cached at worker i to the data it holds."""
    got = {}
    for I, blocks, msg in messages:
        if i not in I:
            continue
        for j, row in enumerate(blocks[i]):
            val = msg[j].copy()
            for other in I:
                if other == i or j >= len(blocks[other]):
                    continue
                known = cache_rows[blocks[other][j]]   # KeyError = not decodable
                if op == "add":
                    val = val - np.asarray(known, np.float64)
                else:
                    val = val ^ np.asarray(known, np.uint32)
            got[row] = val
    return got


def uncoded_rate(q: float, s: float) -> float:
    return q * (1.0 - s / q)


def coded_rate(n: int, q: float, s: float) -> float:
    """Closed form of the coded shuffling rate theorem; the limit of the
    corollary for s = q/n (p = 0)."""
    p = (s - q / n) / (q - q / n)
    if p == 0.0:
        return q * (1.0 - s / q) / (1.0 + n * s / q)
    return q / (n * p) ** 2 * ((1 - p) ** (n + 1) + (n - 1) * p * (1 - p) - (1 - p) ** 2)


def coded_rate_series(n: int, q: float, s: float) -> float:
    """The sum of the theorem's proof: sum_{i=2}^n C(n,i) (q/n) ((i-1)/n)
    p^{i-2} (1-p)^{n-(i-1)}."""
    p = (s - q / n) / (q - q / n)
    return sum(math.comb(n, i) * (q / n) * ((i - 1) / n) * p ** (i - 2) * (1 - p) ** (n - i + 1)
               for i in range(2, n + 1))


class Simulation:
    """The partitions and caches of successive iterations, as sets."""

    def __init__(self, n: int, q: int, s: int, partition_seed: int, cache_seed: int):
        if q % n or not q // n <= s <= q:
            raise ValueError("need q % n == 0 and q/n <= s <= q")
        self.n, self.q, self.s = n, q, s
        self.pseed, self.cseed = partition_seed, cache_seed
        self.t = 0
        self.S = partition(partition_seed, 0, n, q)
        self.C = initial_caches(cache_seed, self.S, q, s)

    def step(self):
        """Advances to t+1; returns (C^t, S^{t+1}) of the transition."""
        S1 = partition(self.pseed, self.t + 1, self.n, self.q)
        C0 = self.C
        self.C = update_caches(self.cseed, self.t + 1, C0, S1, self.q, self.s)
        self.S = S1
        self.t += 1
        return C0, S1


def transition_counts(C, S):
    """(coded rows, uncoded rows) of one transition under Alg. 1."""
    coded = 0
    for I in worker_sets(len(C)):
        coded += max(len(S[i] & exclusive_cache(C, set(I) - {i})) for i in I)
    uncoded = sum(len(S[i] - C[i]) for i in range(len(C)))
    return coded, uncoded
