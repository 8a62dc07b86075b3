// Oracle — TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// Group-relative advantage, Eq. 5 (Sec. 3.2):
//   A_i = (r_i - mean{r_1..r_G}) / std{r_1..r_G}
// The paper does not say which standard deviation it means; std_mode 0 takes the sample
// standard deviation (divisor G-1), std_mode 1 the population one (divisor G).  When the
// deviation is zero (all rewards of the group equal) the advantage is defined as 0, which is
// the limit the paper relies on when it calls such trajectories uninformative (Sec. 3.1).
#include <cmath>

#include "oracle.h"

extern "C" int oracle_advantage(const float* rewards, int P, int G, int std_mode, float* adv,
                                double* key) {
  if (P < 0 || G < 1 || (std_mode != 0 && std_mode != 1)) return 1;
  for (int p = 0; p < P; ++p) {
    const float* r = rewards + (long)p * G;
    // mean{r}: sum in index order, then divide.
    double sum = 0.0;
    for (int i = 0; i < G; ++i) sum += (double)r[i];
    const double mean = sum / (double)G;
    // std{r}: square root of the summed squared deviations over G-1 (or G).
    double ss = 0.0;
    for (int i = 0; i < G; ++i) {
      const double dev = (double)r[i] - mean;
      ss += dev * dev;
    }
    const int divisor = std_mode == 0 ? G - 1 : G;
    const double sd = divisor > 0 ? std::sqrt(ss / (double)divisor) : 0.0;
    for (int i = 0; i < G; ++i) {
      const double dev = (double)r[i] - mean;
      const double a = sd > 0.0 ? dev / sd : 0.0;
      adv[(long)p * G + i] = (float)a;
      if (key) key[(long)p * G + i] = std::fabs(dev);
    }
  }
  return 0;
}
