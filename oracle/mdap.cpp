// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// Maximising-differential advantage pruning (MDAP), Sec. 3.2 Eqs. 6-9, with the order of
// traversal, the |S'_k| >= 1 guarantee and the DP-alignment fill of Algorithm 1 (Phase 2).
//
// Readings taken where the paper leaves a choice (each one is also listed in the design notes):
//  - Eq. 6 groups trajectories by equal advantage.  Inside one group A_i is r_i minus the mean,
//    divided by a positive std, so A_i = A_j exactly when r_i = r_j; when the std is zero all
//    advantages are 0 and so are all reward differences.  Classes are therefore formed by exact
//    reward equality, which does not depend on how A was rounded.
//  - Algorithm 1 visits each class "ordered by |A_i| descending".  |A_i| is |r_i - mean| over
//    a common positive std, so the order key is |r_i - mean| (fp64, Eq. 5's mean); ties, which
//    include every pair inside one class, go to the lower index.
//  - Eq. 7's n is not given; it is a parameter.  N_n(o) holds the distinct length-n windows of
//    the completion's token ids.  Two completions that both have no window are identical, so
//    their distance is 0.
//  - Continuous rewards (the grounding extension): two trajectories share an advantage group
//    when |A_i - A_j| < eps.  That relation is not transitive; its transitive closure is taken:
//    sorted by A, a new class starts wherever the gap to the previous value is >= eps.  With
//    class_eps = 0 the classes are the exact-equality classes above.
//  - The per-prompt cap (keep_cap) is not in the paper; keep_cap >= G leaves Eq. 9's set as is.
//    Above the cap, classes take turns (ordered by the visiting position of their first visited
//    member) and each turn adds the class's next kept member in visiting order (for classes of
//    equal rewards: lowest index first).
//  - DP alignment "adds the unselected trajectory with the highest |A_i| via round-robin":
//    prompts are visited cyclically from prompt 0; each visit adds that prompt's unselected
//    rollout with the largest |r - mean| (lower index on ties); prompts with none are skipped.
#include <algorithm>
#include <cmath>
#include <set>
#include <vector>

#include "oracle.h"

namespace {

using Gram = std::vector<int32_t>;
using GramSet = std::set<Gram>;

// N_n(o): the set of distinct n-grams (as exact tuples of token ids) of one completion.
GramSet ngram_set(const int32_t* ids, int64_t len, int n) {
  GramSet s;
  for (int64_t t = 0; t + n <= len; ++t) s.insert(Gram(ids + t, ids + t + n));
  return s;
}

// Eq. 7: theta_ij = 1 - |N(o_i) & N(o_j)| / |N(o_i) | N(o_j)|.
double jaccard_distance(const GramSet& a, const GramSet& b) {
  std::vector<Gram> common;
  std::set_intersection(a.begin(), a.end(), b.begin(), b.end(), std::back_inserter(common));
  const double inter = (double)common.size();
  const double uni = (double)(a.size() + b.size() - common.size());
  if (uni == 0.0) return 0.0;
  return 1.0 - inter / uni;
}

struct Group {
  std::vector<double> dist;  // |r_i - mean|
  std::vector<int> order;    // visiting order
};

Group order_group(const float* r, int G) {
  Group g;
  double sum = 0.0;
  for (int i = 0; i < G; ++i) sum += (double)r[i];
  const double mean = sum / (double)G;
  g.dist.resize(G);
  for (int i = 0; i < G; ++i) g.dist[i] = std::fabs((double)r[i] - mean);
  g.order.resize(G);
  for (int i = 0; i < G; ++i) g.order[i] = i;
  std::stable_sort(g.order.begin(), g.order.end(),
                   [&](int a, int b) { return g.dist[a] > g.dist[b]; });
  return g;
}

}  // namespace

extern "C" double oracle_jaccard_distance(const int32_t* ids, const int64_t* off, int i, int j,
                                          int ngram_n) {
  const GramSet a = ngram_set(ids + off[i], off[i + 1] - off[i], ngram_n);
  const GramSet b = ngram_set(ids + off[j], off[j + 1] - off[j], ngram_n);
  return jaccard_distance(a, b);
}

// Class of each rollout of a group: exact reward equality, or chains of sorted advantages whose
// consecutive gaps are below class_eps.  Returns the class label (its smallest member index).
static std::vector<int> classes_of(const float* r, const float* a, int G, float class_eps) {
  std::vector<int> cls(G);
  if (class_eps <= 0.0f) {
    for (int i = 0; i < G; ++i) {
      cls[i] = i;
      for (int j = 0; j < i; ++j)
        if (r[j] == r[i]) {
          cls[i] = j;
          break;
        }
    }
    return cls;
  }
  std::vector<int> by_a(G);
  for (int i = 0; i < G; ++i) by_a[i] = i;
  std::stable_sort(by_a.begin(), by_a.end(), [&](int x, int y) { return a[x] < a[y]; });
  std::vector<int> chain(G);
  int c = 0;
  for (int k = 0; k < G; ++k) {
    if (k > 0 && (double)a[by_a[k]] - (double)a[by_a[k - 1]] >= (double)class_eps) ++c;
    chain[by_a[k]] = c;
  }
  for (int i = 0; i < G; ++i) {
    cls[i] = i;
    for (int j = 0; j < i; ++j)
      if (chain[j] == chain[i]) {
        cls[i] = j;
        break;
      }
  }
  return cls;
}

extern "C" int oracle_prune(const float* rewards, const int32_t* ids, const int64_t* off, int P,
                            int G, int ngram_n, float tau, int keep_cap, int dp_divisor,
                            uint8_t* keep, int32_t* kept_per_prompt) {
  return oracle_prune_classes(rewards, nullptr, 0.0f, ids, off, P, G, ngram_n, tau, keep_cap,
                              dp_divisor, keep, kept_per_prompt);
}

extern "C" int oracle_prune_classes(const float* rewards, const float* adv, float class_eps,
                                    const int32_t* ids, const int64_t* off, int P, int G,
                                    int ngram_n, float tau, int keep_cap, int dp_divisor,
                                    uint8_t* keep, int32_t* kept_per_prompt) {
  if (P < 0 || G < 1 || ngram_n < 1 || keep_cap < 1 || dp_divisor < 1) return 1;
  if (class_eps > 0.0f && adv == nullptr) return 1;
  std::vector<Group> groups(P);
  for (int p = 0; p < P; ++p) {
    const float* r = rewards + (long)p * G;
    const std::vector<int> cls = classes_of(r, adv ? adv + (long)p * G : nullptr, G, class_eps);
    Group& grp = groups[p];
    grp = order_group(r, G);
    std::vector<GramSet> sets(G);
    for (int i = 0; i < G; ++i) {
      const long ro = (long)p * G + i;
      sets[i] = ngram_set(ids + off[ro], off[ro + 1] - off[ro], ngram_n);
    }
    // Eq. 8, greedily: visit in order; drop o_i if a kept o_j of its class is within tau.
    std::vector<bool> kept(G, false);
    for (int i : grp.order) {
      bool drop = false;
      for (int j : grp.order) {
        if (!kept[j] || cls[j] != cls[i]) continue;
        if (jaccard_distance(sets[i], sets[j]) < (double)tau) drop = true;
      }
      kept[i] = !drop;
    }
    // Per-prompt cap: classes take turns.
    int count = 0;
    for (int i = 0; i < G; ++i) count += kept[i] ? 1 : 0;
    if (count > keep_cap) {
      struct Cls {
        int label;
        std::vector<int> members;  // kept members, in visiting order
      };
      std::vector<Cls> classes;  // in visiting order of their first visited member
      for (int i : grp.order) {
        if (!kept[i]) continue;
        bool placed = false;
        for (Cls& c : classes) {
          if (c.label == cls[i]) {
            c.members.push_back(i);
            placed = true;
            break;
          }
        }
        if (!placed) classes.push_back(Cls{cls[i], {i}});
      }
      std::vector<bool> capped(G, false);
      int taken = 0;
      for (size_t round = 0; taken < keep_cap; ++round) {
        for (const Cls& c : classes) {
          if (taken == keep_cap) break;
          if (round < c.members.size()) {
            capped[c.members[round]] = true;
            ++taken;
          }
        }
      }
      kept = capped;
    }
    for (int i = 0; i < G; ++i) keep[(long)p * G + i] = kept[i] ? 1 : 0;
  }
  // DP alignment fill across prompts.
  long total = 0;
  for (long i = 0; i < (long)P * G; ++i) total += keep[i];
  int cursor = 0;
  while (dp_divisor > 1 && total % dp_divisor != 0) {
    bool added = false;
    for (int tries = 0; tries < P && !added; ++tries) {
      const int p = cursor;
      cursor = (cursor + 1) % P;
      int best = -1;
      for (int i = 0; i < G; ++i) {
        if (keep[(long)p * G + i]) continue;
        if (best < 0 || groups[p].dist[i] > groups[p].dist[best]) best = i;
      }
      if (best >= 0) {
        keep[(long)p * G + best] = 1;
        ++total;
        added = true;
      }
    }
    if (!added) break;
  }
  for (int p = 0; p < P; ++p) {
    int c = 0;
    for (int i = 0; i < G; ++i) c += keep[(long)p * G + i];
    kept_per_prompt[p] = c;
  }
  return 0;
}
