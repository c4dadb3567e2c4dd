// Host planner: layer budgets in exact integer arithmetic.
//
// Paper: Eq. (parabolic) b_l = 1 - (l-1)^2 / (2 (h-1)^2) for l <= h, layers
// l > h evicted; the proportions are normalised to sum to h*m; the overall
// retention is RR = p*q*(h/L)*m (Sec. 4, Implementation Details), p = 1 here.
// The ablation schedules (Table "ablation": uniform, arithmetic, geometric
// over four layer blocks) replace b_l and keep the rest.
//
// Integer form: b_l is proportional to an integer weight w_l (l = 0..h-1):
//   parabola    2(h-1)^2 - l^2
//   fixed       1
//   arithmetic  2(h-1) - l                 (b from 1 down to 1/2)
//   geometric   2^(nb-1-k), k the block of layer l among nb = min(4, h)
//               contiguous blocks, sizes differing by at most one, larger first
// (w = 1 when h = 1).  T = round(RR*n*L) (token, layer) pairs per KV head are
// split over layers 1..h by largest remainder (ties to the lower layer); the
// survivors of the top-q step are Nq = round(T / (h*m)), clamped to [B_1, n]
// (Nq = n when every non-kept token is dropped).  round() is round-half-up on
// exact rationals.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "viscache.h"

namespace {

// floor((2a + b) / (2b)) for a >= 0, b > 0: round-half-up of a/b.
int64_t round_ratio(unsigned __int128 a, unsigned __int128 b) {
  return (int64_t)((2 * a + b) / (2 * b));
}

}  // namespace

extern "C" int viscache_plan_budgets_ex(int32_t L, int32_t n_vis, uint32_t rr_num, uint32_t rr_den,
                                        int32_t h, uint32_t m_num, uint32_t m_den, int32_t schedule,
                                        int32_t drop_mode, int32_t* B_out, int32_t* n_survive_out,
                                        int32_t* h_out) {
  if (!B_out || !n_survive_out) return VC_ERR_INVALID_ARG;
  if (schedule < VC_SCHED_PARABOLA || schedule > VC_SCHED_GEOMETRIC) return VC_ERR_INVALID_ARG;
  if (drop_mode != VC_DROP_SURVIVORS && drop_mode != VC_DROP_ALL) return VC_ERR_INVALID_ARG;
  if (L < 1 || L > 256 || n_vis < 1) return VC_ERR_INVALID_ARG;
  if (rr_den == 0 || rr_num == 0 || rr_num > rr_den) return VC_ERR_INVALID_ARG;
  if (m_den == 0) { m_num = 3; m_den = 4; }
  if (m_num == 0 || m_num > m_den) return VC_ERR_INVALID_ARG;
  if (h == 0) {
    h = (int32_t)round_ratio((unsigned __int128)3 * (uint32_t)L, 4);
    h = std::max(std::min(2, L), std::min(h, L));
  }
  if (h < 1 || h > L) return VC_ERR_INVALID_ARG;

  // T = round(rr * n * L)
  const int64_t T = round_ratio((unsigned __int128)rr_num * (uint32_t)n_vis * (uint32_t)L, rr_den);

  // integer weights w_l proportional to b_l
  std::vector<int64_t> w(h, 1);
  if (h > 1) {
    if (schedule == VC_SCHED_PARABOLA) {
      const int64_t hh = (int64_t)(h - 1) * (h - 1);
      for (int l = 0; l < h; ++l) w[l] = 2 * hh - (int64_t)l * l;
    } else if (schedule == VC_SCHED_ARITHMETIC) {
      for (int l = 0; l < h; ++l) w[l] = 2 * (int64_t)(h - 1) - l;
    } else if (schedule == VC_SCHED_GEOMETRIC) {
      const int nb = std::min(4, h), per = h / nb, extra = h % nb;
      int l = 0;
      for (int k = 0; k < nb; ++k)
        for (int i = 0; i < per + (k < extra ? 1 : 0); ++i) w[l++] = (int64_t)1 << (nb - 1 - k);
    }
  }
  int64_t wsum = 0;
  for (int64_t x : w) wsum += x;

  // largest remainder: floor(T w_l / wsum), then +1 to the largest remainders
  std::vector<int64_t> base(h), rem(h);
  int64_t assigned = 0;
  for (int l = 0; l < h; ++l) {
    const unsigned __int128 q = (unsigned __int128)T * (uint64_t)w[l];
    base[l] = (int64_t)(q / (uint64_t)wsum);
    rem[l] = (int64_t)(q % (uint64_t)wsum);
    assigned += base[l];
  }
  std::vector<int> order(h);
  for (int l = 0; l < h; ++l) order[l] = l;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rem[a] > rem[b]; });
  for (int64_t k = 0; k < T - assigned; ++k) base[order[k]] += 1;

  if (base[0] > n_vis) return VC_ERR_INFEASIBLE;
  for (int l = 0; l < L; ++l) B_out[l] = l < h ? (int32_t)base[l] : 0;

  // Nq = round(T / (h*m)) = round(T * m_den / (h * m_num)), clamped to [B_1, n]
  int64_t nq = round_ratio((unsigned __int128)T * m_den, (unsigned __int128)(uint32_t)h * m_num);
  nq = std::min<int64_t>(n_vis, std::max<int64_t>(nq, base[0]));
  if (drop_mode == VC_DROP_ALL) nq = n_vis;
  *n_survive_out = (int32_t)nq;
  if (h_out) *h_out = h;
  return VC_OK;
}

extern "C" int viscache_plan_budgets(int32_t L, int32_t n_vis, uint32_t rr_num, uint32_t rr_den,
                                     int32_t h, uint32_t m_num, uint32_t m_den, int32_t* B_out,
                                     int32_t* n_survive_out, int32_t* h_out) {
  return viscache_plan_budgets_ex(L, n_vis, rr_num, rr_den, h, m_num, m_den, VC_SCHED_PARABOLA,
                                  VC_DROP_SURVIVORS, B_out, n_survive_out, h_out);
}
