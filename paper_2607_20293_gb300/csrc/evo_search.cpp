// Schedule search (Sec. 3.2, Sec. 3.3): the genetic algorithm over
// fixed-budget schedules (individual of Eq. 3: K unique lattice positions),
// redundancy-guided initial individuals (Eq. 7) and target-conditioned early
// stopping (Eq. 8, Eq. 9).  Host code: fitness evaluation is the caller's
// callback (typically evo_denoise_population on the GPU); the search itself
// is bookkeeping over at most a few thousand lattice cells per individual.
//
// Procedure (every random decision draws from one SplitMix64 stream):
//   init      `guided` individuals by sequential weighted draws without
//             replacement (Eq. 7 weights in fixed point), the rest with equal
//             weights; block-wise variant: m draws per unit row
//   per generation
//     evaluate  individuals not seen before (signature = sorted cell list)
//     rank      by fitness, ties by signature, best first
//     stop      (optional) candidates whose quick fitness reaches q_base are
//               evaluated formally; the first in rank order whose formal
//               fitness is at least q_base - delta_acc is accepted
//     breed     elites carried over; children: two tournament winners,
//               set-level crossover (common positions kept, each other one
//               with probability 1/2) with probability crossover_rate,
//               mutation (each position, with probability mutation_rate, a
//               uniform cell of the lattice / of its unit row), repair to
//               exactly K unique positions (drop repeats, add uniform cells,
//               remove uniform positions)
// below(n) = next() mod n, unit() = (next() >> 11) * 2^-53.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <map>
#include <vector>

#include "evo.h"

namespace {

struct Rng {
  uint64_t s;
  uint64_t next() {
    s += 0x9E3779B97F4A7C15ull;
    uint64_t z = s;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
  }
  uint64_t below(uint64_t n) { return next() % n; }
  double unit() { return (double)(next() >> 11) * (1.0 / 9007199254740992.0); }
};

using Ind = std::vector<int32_t>;   // sorted cells c = b * T + t

// K distinct indices of w (offset added) by sequential weighted draws
void draw(const int64_t* w, int n, int K, Rng& rng, int offset, Ind& out) {
  std::vector<char> taken(n, 0);
  for (int k = 0; k < K; ++k) {
    int64_t total = 0;
    for (int i = 0; i < n; ++i)
      if (!taken[i]) total += w[i];
    const uint64_t r = rng.next();
    int pick = -1;
    if (total == 0) {
      for (int i = 0; i < n && pick < 0; ++i)
        if (!taken[i]) pick = i;
    } else {
      const uint64_t target = r % (uint64_t)total;
      uint64_t run = 0;
      for (int i = 0; i < n; ++i) {
        if (taken[i]) continue;
        run += (uint64_t)w[i];
        if (run > target) {
          pick = i;
          break;
        }
      }
    }
    taken[pick] = 1;
    out.push_back(offset + pick);
  }
}

// exactly K distinct cells of [lo, hi), sorted, appended to out
void repair_cells(const Ind& cells, int K, int lo, int hi, Rng& rng, Ind& out) {
  std::vector<char> seen(hi - lo, 0);
  Ind v;
  for (int c : cells)
    if (!seen[c - lo]) {
      seen[c - lo] = 1;
      v.push_back(c);
    }
  while ((int)v.size() < K) {
    const int c = lo + (int)rng.below((uint64_t)(hi - lo));
    if (!seen[c - lo]) {
      seen[c - lo] = 1;
      v.push_back(c);
    }
  }
  while ((int)v.size() > K) {
    const size_t i = (size_t)rng.below(v.size());
    seen[v[i] - lo] = 0;
    v.erase(v.begin() + (long)i);
  }
  std::sort(v.begin(), v.end());
  out.insert(out.end(), v.begin(), v.end());
}

struct Searcher {
  const evo_search_config& c;
  int U, T, C, K, m;
  Rng rng;
  std::map<Ind, double> memo, fmemo;
  Searcher(const evo_search_config& cfg)
      : c(cfg), U(cfg.n_units), T(cfg.n_steps), C(cfg.n_units * cfg.n_steps),
        K(cfg.block_wise ? cfg.budget * cfg.n_units : cfg.budget), m(cfg.budget), rng{cfg.seed} {}

  // fitness order: higher first, then the smaller signature
  bool better(const Ind& a, const Ind& b, const std::map<Ind, double>& f) const {
    const double fa = f.at(a), fb = f.at(b);
    if (fa != fb) return fa > fb;
    return a < b;
  }

  Ind init_one(const std::vector<int64_t>* q) {
    Ind out;
    if (!c.block_wise) {
      std::vector<int64_t> ones;
      if (!q) ones.assign(C, 1);
      draw(q ? q->data() : ones.data(), C, K, rng, 0, out);
    } else {
      std::vector<int64_t> ones(T, 1);
      for (int b = 0; b < U; ++b) draw(q ? q->data() + (size_t)b * T : ones.data(), T, m, rng, b * T, out);
    }
    std::sort(out.begin(), out.end());
    return out;
  }

  Ind crossover(const Ind& a, const Ind& b) {
    Ind child;
    size_t i = 0, j = 0;
    while (i < a.size() || j < b.size()) {    // union in increasing order
      if (j == b.size() || (i < a.size() && a[i] < b[j])) {
        if (rng.next() & 1) child.push_back(a[i]);
        ++i;
      } else if (i == a.size() || b[j] < a[i]) {
        if (rng.next() & 1) child.push_back(b[j]);
        ++j;
      } else {                                 // in both parents
        child.push_back(a[i]);
        ++i;
        ++j;
      }
    }
    return child;
  }

  Ind mutate(const Ind& cells) {
    Ind out;
    out.reserve(cells.size());
    for (int cell : cells) {
      if (rng.unit() < c.mutation_rate)
        cell = c.block_wise ? (cell / T) * T + (int)rng.below((uint64_t)T) : (int)rng.below((uint64_t)C);
      out.push_back(cell);
    }
    return out;
  }

  Ind repair(const Ind& cells) {
    Ind out;
    if (!c.block_wise) {
      repair_cells(cells, K, 0, C, rng, out);
      return out;
    }
    for (int b = 0; b < U; ++b) {
      Ind row;
      for (int cell : cells)
        if (cell / T == b) row.push_back(cell);
      repair_cells(row, m, b * T, (b + 1) * T, rng, out);
    }
    return out;
  }

  const Ind& tournament(const std::vector<Ind>& ranked) {
    int best = -1;
    for (int i = 0; i < c.tournament; ++i) {
      const int j = (int)rng.below(ranked.size());
      if (best < 0 || better(ranked[j], ranked[best], memo)) best = j;
    }
    return ranked[best];
  }

  void lattices(const std::vector<Ind>& v, std::vector<uint8_t>& S) const {
    S.assign(v.size() * (size_t)C, 0);
    for (size_t i = 0; i < v.size(); ++i)
      for (int cell : v[i]) S[i * C + cell] = 1;
  }
};

}  // namespace

extern "C" {

evo_status evo_search(const evo_search_config* cfg, const float* d_map, evo_fitness_fn quick, evo_fitness_fn formal,
                      void* user, uint8_t* best_S, evo_search_result* result) {
  if (!cfg || !quick || !best_S) return EVO_ERR_ARG;
  const evo_search_config& c = *cfg;
  if (c.n_units <= 0 || c.n_steps <= 0 || c.budget <= 0 || c.population <= 0 || c.elites < 0 ||
      c.elites > c.population || c.generations <= 0 || c.tournament <= 0 || c.guided < 0 ||
      c.guided > c.population || (c.guided > 0 && !d_map) || (c.early_stop && !formal) || c.gamma < 1 ||
      !(c.eps >= 0.f))
    return EVO_ERR_ARG;
  if (c.block_wise ? c.budget > c.n_steps : c.budget > c.n_units * c.n_steps) return EVO_ERR_SHAPE;
  Searcher s(c);
  // Eq. 7 weights in fixed point: floor((eps + d / max d)^gamma * 2^40)
  std::vector<int64_t> q;
  if (c.guided > 0) {
    float mx = 0.f;
    for (int i = 0; i < s.C; ++i) mx = std::max(mx, d_map[i]);
    if (!(mx > 0.f)) return EVO_ERR_ARG;
    q.resize(s.C);
    for (int i = 0; i < s.C; ++i) {
      const double base = (double)c.eps + (double)d_map[i] / (double)mx;
      double v = base;
      for (int g = 1; g < c.gamma; ++g) v = v * base;
      q[i] = (int64_t)std::floor(v * 1099511627776.0);
    }
  }
  std::vector<Ind> pop;
  for (int i = 0; i < c.guided; ++i) pop.push_back(s.init_one(&q));
  for (int i = c.guided; i < c.population; ++i) pop.push_back(s.init_one(nullptr));

  evo_search_result st{};
  Ind best;
  bool have_best = false, accepted = false;
  Ind acc;
  std::vector<uint8_t> S;
  std::vector<double> fit;
  for (int g = 0; g < c.generations; ++g) {
    std::vector<Ind> fresh;
    for (const Ind& ind : pop) {
      if (s.memo.count(ind) || std::find(fresh.begin(), fresh.end(), ind) != fresh.end()) {
        ++st.memo_hits;
      } else {
        fresh.push_back(ind);
      }
    }
    if (!fresh.empty()) {
      s.lattices(fresh, S);
      fit.assign(fresh.size(), 0.0);
      if (quick(user, S.data(), (int32_t)fresh.size(), c.n_units, c.n_steps, fit.data()) != 0) return EVO_ERR_ARG;
      for (size_t i = 0; i < fresh.size(); ++i) s.memo[fresh[i]] = fit[i];
      st.evaluations += (int32_t)fresh.size();
    }
    std::vector<Ind> ranked = pop;
    std::sort(ranked.begin(), ranked.end(), [&](const Ind& a, const Ind& b) { return s.better(a, b, s.memo); });
    if (!have_best || s.better(ranked[0], best, s.memo)) {
      best = ranked[0];
      have_best = true;
    }
    st.generations = g + 1;
    if (c.early_stop) {
      std::vector<Ind> trig;
      for (const Ind& ind : ranked)
        if (s.memo.at(ind) >= c.q_base && !s.fmemo.count(ind) &&
            std::find(trig.begin(), trig.end(), ind) == trig.end())
          trig.push_back(ind);
      if (!trig.empty()) {
        s.lattices(trig, S);
        fit.assign(trig.size(), 0.0);
        if (formal(user, S.data(), (int32_t)trig.size(), c.n_units, c.n_steps, fit.data()) != 0) return EVO_ERR_ARG;
        for (size_t i = 0; i < trig.size(); ++i) s.fmemo[trig[i]] = fit[i];
        st.formal_evaluations += (int32_t)trig.size();
      }
      for (const Ind& ind : ranked) {
        auto it = s.fmemo.find(ind);
        if (it != s.fmemo.end() && s.memo.at(ind) >= c.q_base && it->second >= c.q_base - c.delta_acc) {
          acc = ind;
          accepted = true;
          break;
        }
      }
      if (accepted) {
        st.stopped_early = 1;
        break;
      }
    }
    if (g == c.generations - 1) break;
    std::vector<Ind> next(ranked.begin(), ranked.begin() + c.elites);
    while ((int)next.size() < c.population) {
      const Ind a = s.tournament(ranked);
      const Ind b = s.tournament(ranked);
      Ind child = s.rng.unit() < c.crossover_rate ? s.crossover(a, b) : a;
      next.push_back(s.repair(s.mutate(child)));
    }
    pop.swap(next);
  }
  const Ind& res = accepted ? acc : best;
  std::memset(best_S, 0, (size_t)s.C);
  for (int cell : res) best_S[cell] = 1;
  st.best_fitness = accepted ? s.fmemo.at(res) : s.memo.at(res);
  if (result) *result = st;
  return EVO_OK;
}

}  // extern "C"
