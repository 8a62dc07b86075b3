// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// Compaction of the kept rollouts' tokens.  Sec. 3.2 (after Eq. 9) feeds only the retained
// trajectories to the old, current and reference models, and Algorithm 1 updates the policy on
// the selected set only.  The compacted layout lists the kept rollouts in ascending index
// order, each with its tokens in order.
#include "oracle.h"

extern "C" int oracle_compact(const uint8_t* keep, const int64_t* off, int n_rollouts,
                              int32_t* kept_idx, int64_t* kept_off, int64_t* src_token,
                              int32_t* token_rollout, int64_t* counts) {
  if (n_rollouts < 0) return 1;
  int64_t k = 0, t_kept = 0;
  for (int r = 0; r < n_rollouts; ++r) {
    if (!keep[r]) continue;
    kept_idx[k] = r;
    kept_off[k] = t_kept;
    for (int64_t s = off[r]; s < off[r + 1]; ++s) {
      src_token[t_kept] = s;
      token_rollout[t_kept] = r;
      ++t_kept;
    }
    ++k;
  }
  kept_off[k] = t_kept;
  counts[0] = k;
  counts[1] = t_kept;
  return 0;
}
