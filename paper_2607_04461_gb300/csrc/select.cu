// Stage 2 of Flash-BoN (§4.2): multi-stage selection with Elo ratings. Host code only:
// it runs between fb_draft and fb_refine and calls a caller-supplied pairwise verifier.
//  1. Elo seeding from pointwise scores, r = 1500 + (s - 5) * 100; keep the top
//     ceil(rho1 M) (ties to the lower index).
//  2. ceil(kappa M1) comparisons between adjacent entries of the survivors sorted by
//     rating: passes over the list from the top, re-sorted before each pass. Each result
//     updates both ratings with K = k_base x {1.2, 1.0, 0.7} for the verifier's
//     high / medium / low confidence. Keep the top ceil(rho2 M1).
//  3. Every pair (i, j), i < j, of the survivors in rating order; the winner is the
//     survivor with the highest rating.
// Elo update: E_a = 1 / (1 + 10^((r_b - r_a) / 400)), r_a += K (S_a - E_a), r_b likewise.
#include <algorithm>
#include <cmath>
#include <vector>

#include "../../include/flashbon.h"

namespace {
const double kConf[3] = {1.2, 1.0, 0.7};

// ceil of a product of a decimal ratio and a count: 0.3 * 20 is 6, not 7
size_t ceil_count(double x) { return (size_t)std::ceil(x - 1e-9); }

std::vector<int> top(const std::vector<int>& ids, const std::vector<double>& r, size_t count) {
  std::vector<int> o(ids);
  std::stable_sort(o.begin(), o.end(), [&](int a, int b) {
    return r[a] > r[b] || (r[a] == r[b] && a < b);
  });
  if (o.size() > count) o.resize(count);
  return o;
}
}  // namespace

extern "C" fb_status fb_select_elo(const int32_t* scores, int M, double rho1, double rho2,
                                   double kappa, double k_base, fb_pair_verifier compare,
                                   void* user, int* winner, double* out_ratings,
                                   int* out_calls) {
  if (!scores || !compare || !winner || M < 1) return FB_EINVAL;
  if (!(rho1 > 0.0 && rho1 <= 1.0) || !(rho2 > 0.0 && rho2 <= 1.0) || !(kappa >= 0.0) ||
      !(k_base > 0.0))
    return FB_EINVAL;
  std::vector<double> r(M);
  for (int j = 0; j < M; ++j) r[j] = 1500.0 + (scores[j] - 5.0) * 100.0;
  int calls = 0;
  bool bad = false;
  auto play = [&](int a, int b) {
    int conf = 1;
    const int a_wins = compare(user, a, b, &conf);
    ++calls;
    if (conf < 0 || conf > 2) {
      bad = true;
      conf = 1;
    }
    const double k = k_base * kConf[conf];
    const double ea = 1.0 / (1.0 + std::pow(10.0, (r[b] - r[a]) / 400.0));
    const double sa = a_wins ? 1.0 : 0.0;
    const double ra = r[a] + k * (sa - ea), rb = r[b] + k * ((1.0 - sa) - (1.0 - ea));
    r[a] = ra;
    r[b] = rb;
  };
  std::vector<int> all(M);
  for (int j = 0; j < M; ++j) all[j] = j;
  const std::vector<int> s1 = top(all, r, ceil_count(rho1 * M));
  const long c2 = (long)ceil_count(kappa * (double)s1.size());
  long done = 0;
  while (done < c2 && s1.size() > 1) {
    const std::vector<int> order = top(s1, r, s1.size());
    for (size_t i = 0; i + 1 < order.size() && done < c2; ++i, ++done) play(order[i], order[i + 1]);
  }
  const std::vector<int> s2 = top(s1, r, ceil_count(rho2 * (double)s1.size()));
  const std::vector<int> order = top(s2, r, s2.size());
  for (size_t i = 0; i < order.size(); ++i)
    for (size_t j = i + 1; j < order.size(); ++j) play(order[i], order[j]);
  *winner = top(s2, r, 1)[0];
  if (out_ratings)
    for (int j = 0; j < M; ++j) out_ratings[j] = r[j];
  if (out_calls) *out_calls = calls;
  return bad ? FB_EINVAL : FB_OK;
}
