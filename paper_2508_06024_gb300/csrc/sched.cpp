// Route-aware heuristic pipeline scheduler of the end-cloud pipeline
// (Eq. 9-11): host code, no CUDA.
//
//   Eq. 10  P(t_i) = C(t_i) / (Comm(t_i) + eps)
//   Eq. 11  Location(t_i) = End if Load_end + C(t_i) <= T_end and P(t_i) >= beta,
//           Cloud otherwise
//   Eq. 9   objective sum_i alpha * ExecTime(t_i) + (1 - alpha) * Comm(t_i)
//
// The greedy visits tasks in decreasing priority with ties to the lower task
// index (a stable sort), keeps going after Cloud decisions, and grows the End
// load by the cost of every task it keeps local.  Route-aware tasks come from
// the routing histogram: one task per expert that received rows.
#include <algorithm>
#include <cmath>
#include <numeric>
#include <vector>

#include "ec2moe.h"

namespace {

bool bad_nonneg(double v) { return !(v >= 0.0); }  // negative or NaN

}  // namespace

extern "C" {

ec2moe_status ec2moe_schedule(int32_t n, const double* cost, const double* comm, double load_end,
                              double load_cloud, double T_end, double beta, double eps, int32_t* location,
                              int32_t* order, double* load_end_out, double* load_cloud_out) {
  if (n < 0 || std::isnan(eps) || eps < 0.0 || std::isnan(load_end) || std::isnan(load_cloud) ||
      std::isnan(T_end) || std::isnan(beta))
    return EC2MOE_ERR_INVALID_ARG;
  if (n > 0 && (!cost || !comm || !location)) return EC2MOE_ERR_INVALID_ARG;
  std::vector<double> P(static_cast<size_t>(n));
  for (int32_t i = 0; i < n; ++i) {
    if (bad_nonneg(cost[i]) || bad_nonneg(comm[i]) || !(comm[i] + eps > 0.0)) return EC2MOE_ERR_INVALID_ARG;
    P[i] = cost[i] / (comm[i] + eps);  // Eq. 10
  }
  std::vector<int32_t> idx(static_cast<size_t>(n));
  std::iota(idx.begin(), idx.end(), 0);
  std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) { return P[a] > P[b]; });
  double le = load_end, lc = load_cloud;
  for (int32_t j = 0; j < n; ++j) {
    const int32_t i = idx[j];
    if (le + cost[i] <= T_end && P[i] >= beta) {  // Eq. 11
      location[i] = EC2MOE_END;
      le = le + cost[i];
    } else {
      location[i] = EC2MOE_CLOUD;
      lc = lc + cost[i];
    }
    if (order) order[j] = i;
  }
  if (load_end_out) *load_end_out = le;
  if (load_cloud_out) *load_cloud_out = lc;
  return EC2MOE_OK;
}

ec2moe_status ec2moe_schedule_objective(int32_t n, const double* cost, const double* comm,
                                        const int32_t* location, double rate_end, double rate_cloud,
                                        double alpha, double* objective) {
  if (n < 0 || !objective || !(rate_end > 0.0) || !(rate_cloud > 0.0) || std::isnan(alpha))
    return EC2MOE_ERR_INVALID_ARG;
  if (n > 0 && (!cost || !comm || !location)) return EC2MOE_ERR_INVALID_ARG;
  double total = 0.0;
  for (int32_t i = 0; i < n; ++i) {
    if (location[i] != EC2MOE_END && location[i] != EC2MOE_CLOUD) return EC2MOE_ERR_INVALID_ARG;
    const bool end = location[i] == EC2MOE_END;
    const double exec_time = cost[i] / (end ? rate_end : rate_cloud);
    const double paid = end ? 0.0 : comm[i];
    const double a = alpha * exec_time;
    const double b = (1.0 - alpha) * paid;
    total = total + (a + b);  // Eq. 9
  }
  *objective = total;
  return EC2MOE_OK;
}

ec2moe_status ec2moe_expert_tasks(const ec2moe_layer_desc* desc, const int32_t* counts, int32_t* expert_of_task,
                                  double* cost, double* comm, int32_t* n_tasks) {
  if (!desc || !counts || !expert_of_task || !cost || !comm || !n_tasks) return EC2MOE_ERR_INVALID_ARG;
  if (desc->E < 1 || desc->d < 1 || desc->d_ff < 1 || desc->r < 0 ||
      (desc->dtype != EC2MOE_BF16 && desc->dtype != EC2MOE_F32) ||
      (desc->act != EC2MOE_GELU && desc->act != EC2MOE_SWIGLU))
    return EC2MOE_ERR_INVALID_ARG;
  const double proj = desc->act == EC2MOE_SWIGLU ? 3.0 : 2.0;
  const double bytes = desc->dtype == EC2MOE_BF16 ? 2.0 : 4.0;
  const double w_in = desc->r > 0 ? desc->r : desc->d;
  int32_t j = 0;
  for (int32_t e = 0; e < desc->E; ++e) {
    if (counts[e] < 0) return EC2MOE_ERR_INVALID_ARG;
    if (counts[e] == 0) continue;
    const double rows = counts[e];
    expert_of_task[j] = e;
    cost[j] = 2.0 * rows * desc->d * desc->d_ff * proj;
    comm[j] = rows * (w_in + desc->d) * bytes;
    ++j;
  }
  *n_tasks = j;
  return EC2MOE_OK;
}

}  // extern "C"
