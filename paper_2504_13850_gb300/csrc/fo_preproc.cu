// Pre-processor split selection (Sec. 3.2, "Splitting the DNN", Eqs. 4-6):
// host-only, evaluated once when the server is set up.  For each candidate
// split point l the slowest device's bottleneck time is
//   max_k max( sum_{i<=l} O_i / o_k ,  S_l / b_k )
// and the split minimises it (first minimum on ties).
#include "../../include/fedoptima.h"

#include <cmath>
#include <string>

namespace fo {
int report_error(int code, const std::string& msg);
}

extern "C" FO_API int fo_select_split(const double* O, const double* S, int L, const double* b, const double* o,
                                      int K, const unsigned char* allowed, int* split, double* cost) {
  if (!O || !S || !b || !o || !split || !cost || L < 1 || K < 1) {
    return fo::report_error(FO_ERR_ARG, "fo_select_split: null pointer, L < 1 or K < 1");
  }
  for (int l = 0; l < L; ++l)
    if (!(O[l] >= 0.0) || !(S[l] >= 0.0)) {
      return fo::report_error(FO_ERR_ARG, "fo_select_split: O and S must be non-negative");
    }
  for (int k = 0; k < K; ++k)
    if (!(b[k] > 0.0) || !(o[k] > 0.0)) {
      return fo::report_error(FO_ERR_ARG, "fo_select_split: b and o must be positive");
    }
  int best = 0;
  double best_cost = INFINITY;
  double cum = 0.0;   // sum_{i<=l} O_i
  for (int l = 1; l <= L; ++l) {
    cum += O[l - 1];
    if (allowed && !allowed[l - 1]) continue;
    double worst = 0.0;
    for (int k = 0; k < K; ++k) {
      const double t = std::fmax(cum / o[k], S[l - 1] / b[k]);
      if (t > worst) worst = t;
    }
    if (best == 0 || worst < best_cost) {
      best = l;
      best_cost = worst;
    }
  }
  if (best == 0) {
    return fo::report_error(FO_ERR_ARG, "fo_select_split: no allowed split point");
  }
  *split = best;
  *cost = best_cost;
  return FO_OK;
}
