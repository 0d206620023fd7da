"""CPU oracle of EVO's schedule search (Sec. 3.2 and Sec. 3.3): the genetic
algorithm over fixed-budget schedules and target-conditioned early stopping.

TEST INFRASTRUCTURE ONLY.  Only the tests (and bench.py's reference leg) may
import this module; the library's search (evo_search in the C ABI) shares no
code with it.

What it follows, in the paper's terms:

* Individual (Eq. 3): K unique lattice positions (b, t); here cell c = b*T + t,
  kept as a sorted tuple (its canonical signature).
* Fitness F(S) (Eq. 4) is supplied by the caller (rollouts are out of scope; the
  tests use synthetic fitness functions and the population deviation).
* Per generation: evaluate the individuals not seen before (signature memo),
  rank by fitness, keep the elites, and fill the population with children:
  tournament-selected parents, set-level crossover, mutation, repair to
  exactly K positions (Sec. 3.2).
* Initial population (Sec. 3.3): guided individuals drawn by Eq. 7 from the
  redundancy weights, plus random individuals.
* Block-wise variant (ablation, Sec. 4.3): every unit keeps exactly m refresh
  steps; operators act row by row.
* Early stopping (Eq. 8, Eq. 9): a candidate whose quick fitness reaches q_base
  is evaluated formally; it is accepted, and the search stops, when its formal
  fitness is at least q_base - delta_acc.

Readings (the paper gives the operators but not their parameters or order):
* Randomness: SplitMix64 (Steele, Lea and Flood 2014), one stream seeded by the
  caller; below(n) = next() mod n; unit() = (next() >> 11) * 2^-53.
* Ranking: by fitness, ties by signature (lexicographic), best first.
* Tournament: k uniform picks (with replacement) from the ranked population,
  the best one wins.
* Set-level crossover: positions present in both parents are kept, a position
  present in one parent is taken with probability 1/2 (one draw each, in
  increasing cell order), applied with probability crossover_rate; otherwise
  the child copies the first parent.
* Mutation: each position, in increasing order, is replaced with probability
  mutation_rate by a uniform cell of the lattice (block-wise: of its row).
* Repair: drop repeated positions (keeping the first), add uniform cells not yet
  present until K, remove uniform positions while above K; sort.
* Guided / random initial individuals: sequential draws without replacement,
  target = next() mod (sum of the remaining weights), the first remaining cell
  whose running weight sum exceeds it; guided weights are those of Eq. 7 in
  fixed point (oracle.evo_oracle.guided_weights), random ones all equal.
* Early stopping: checked after every generation on the triggered candidates in
  rank order; formal evaluations are batched per generation and memoised.
"""
from __future__ import annotations

import numpy as np

from oracle import evo_oracle as O

MASK64 = (1 << 64) - 1


class SplitMix64:
    """SplitMix64 generator, from its published definition."""

    def __init__(self, seed: int):
        self.state = seed & MASK64

    def next(self) -> int:
        self.state = (self.state + 0x9E3779B97F4A7C15) & MASK64
        z = self.state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
        return z ^ (z >> 31)

    def below(self, n: int) -> int:
        return self.next() % n

    def unit(self) -> float:
        return (self.next() >> 11) * (1.0 / 9007199254740992.0)


def _draw(weights, K, rng, offset=0):
    """K distinct indices of `weights` by sequential weighted draws (exact integers)."""
    w = [int(v) for v in weights]
    taken = [False] * len(w)
    out = []
    for _ in range(K):
        total = sum(v for v, t in zip(w, taken) if not t)
        r = rng.next()
        if total == 0:
            i = taken.index(False)
        else:
            target = r % total
            run = 0
            for i, v in enumerate(w):
                if taken[i]:
                    continue
                run += v
                if run > target:
                    break
        taken[i] = True
        out.append(offset + i)
    return out


def _repair_cells(cells, K, lo, hi, rng):
    """Repair to exactly K distinct cells in [lo, hi)."""
    seen, out = set(), []
    for c in cells:
        if c not in seen:
            seen.add(c)
            out.append(c)
    while len(out) < K:
        c = lo + rng.below(hi - lo)
        if c not in seen:
            seen.add(c)
            out.append(c)
    while len(out) > K:
        c = out.pop(rng.below(len(out)))
        seen.discard(c)
    return sorted(out)


class Search:
    def __init__(self, U: int, T: int, budget: int, block_wise: bool = False, population: int = 30,
                 elites: int = 10, generations: int = 30, tournament: int = 3, guided: int = 0,
                 crossover_rate: float = 0.9, mutation_rate: float = 0.02, eps: float = 0.05, gamma: int = 2,
                 early_stop: bool = False, q_base: float = 0.0, delta_acc: float = 0.0, seed: int = 0):
        self.U, self.T, self.block_wise = U, T, block_wise
        self.m = budget if block_wise else None
        self.K = budget * U if block_wise else budget
        self.P, self.E, self.G, self.k = population, elites, generations, tournament
        self.guided, self.cx, self.mut = guided, crossover_rate, mutation_rate
        self.eps, self.gamma = eps, gamma
        self.early_stop, self.q_base, self.delta_acc = early_stop, q_base, delta_acc
        self.rng = SplitMix64(seed)

    # ---------------------------------------------------------------- operators
    def _init_one(self, q):
        T = self.T
        if not self.block_wise:
            w = q if q is not None else [1] * (self.U * T)
            return tuple(sorted(_draw(w, self.K, self.rng)))
        cells = []
        for b in range(self.U):
            w = q[b * T:(b + 1) * T] if q is not None else [1] * T
            cells += _draw(w, self.m, self.rng, offset=b * T)
        return tuple(sorted(cells))

    def _crossover(self, a, b):
        sa, sb = set(a), set(b)
        child = []
        for c in sorted(sa | sb):
            if c in sa and c in sb:
                child.append(c)
            elif self.rng.next() & 1:
                child.append(c)
        return child

    def _mutate(self, cells):
        out = []
        C, T = self.U * self.T, self.T
        for c in cells:
            if self.rng.unit() < self.mut:
                c = (c // T) * T + self.rng.below(T) if self.block_wise else self.rng.below(C)
            out.append(c)
        return out

    def _repair(self, cells):
        if not self.block_wise:
            return tuple(_repair_cells(cells, self.K, 0, self.U * self.T, self.rng))
        T, out = self.T, []
        for b in range(self.U):
            row = [c for c in cells if c // T == b]
            out += _repair_cells(row, self.m, b * T, (b + 1) * T, self.rng)
        return tuple(out)

    def _tournament(self, ranked):
        best = None
        for _ in range(self.k):
            cand = ranked[self.rng.below(len(ranked))]
            if best is None or ranked.index(cand) < ranked.index(best):
                best = cand
        return best

    def lattice(self, ind):
        S = np.zeros(self.U * self.T, dtype=np.uint8)
        S[list(ind)] = 1
        return S.reshape(self.U, self.T)

    # ---------------------------------------------------------------- the search
    def run(self, quick, formal=None, d_map=None):
        """quick / formal: callables [P][U][T] uint8 -> [P] fitness (higher is better)."""
        q = None
        if d_map is not None and self.guided > 0:
            q = [int(v) for v in O.guided_weights(np.asarray(d_map, dtype=np.float32), self.eps, self.gamma)]
        pop = [self._init_one(q) for _ in range(self.guided)]
        pop += [self._init_one(None) for _ in range(self.P - self.guided)]
        memo, fmemo = {}, {}
        stats = dict(generations=0, evaluations=0, formal_evaluations=0, memo_hits=0, stopped_early=0)
        best = None
        accepted = None
        for g in range(self.G):
            new = []
            for ind in pop:
                if ind in memo or ind in new:
                    stats["memo_hits"] += 1
                else:
                    new.append(ind)
            if new:
                fit = quick(np.stack([self.lattice(i) for i in new]))
                for ind, f in zip(new, fit):
                    memo[ind] = float(f)
                stats["evaluations"] += len(new)
            key = lambda ind: (-memo[ind], ind)
            ranked = sorted(pop, key=key)
            if best is None or key(ranked[0]) < key(best):
                best = ranked[0]
            stats["generations"] = g + 1
            if self.early_stop:
                trig = []
                for ind in ranked:
                    if memo[ind] >= self.q_base and ind not in fmemo and ind not in trig:
                        trig.append(ind)
                if trig:
                    fit = formal(np.stack([self.lattice(i) for i in trig]))
                    for ind, f in zip(trig, fit):
                        fmemo[ind] = float(f)
                    stats["formal_evaluations"] += len(trig)
                for ind in ranked:
                    if ind in fmemo and memo[ind] >= self.q_base and fmemo[ind] >= self.q_base - self.delta_acc:
                        accepted = ind
                        break
                if accepted is not None:
                    stats["stopped_early"] = 1
                    break
            if g == self.G - 1:
                break
            nxt = ranked[:self.E]
            while len(nxt) < self.P:
                a = self._tournament(ranked)
                b = self._tournament(ranked)
                child = self._crossover(a, b) if self.rng.unit() < self.cx else list(a)
                nxt.append(self._repair(self._mutate(child)))
            pop = nxt
        result = accepted if accepted is not None else best
        fitness = fmemo[result] if accepted is not None else memo[result]
        return self.lattice(result), fitness, stats
