// Discrete-event model of length-aware serving (Sec. 5.3 and the appendix "System-Level Evaluation Details"): RR / LB routing to
// decode instances and FCFS / SJF admission, driven by the static prediction.
// The model and its tie rules are stated in include/outlets_sched.h.  Built
// without contracted multiply-adds (-ffp-contract=off) so that times are the
// same IEEE double results on every host.
#include "outlets_sched.h"

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <limits>
#include <set>
#include <tuple>
#include <vector>

namespace {

struct Instance {
  std::vector<int> running;       // admission order
  std::set<std::tuple<long long, double, int>> waiting;  // admission key (SJF or FCFS), unique by index
  long long load = 0;             // LB: predicted remaining tokens of running + waiting requests
  double step_end = 0.0;
  bool busy = false;
};

bool valid(const outlets_sched_config* c, int n, const double* a, const int32_t* p, const int32_t* o,
           const float* r) {
  if (c->n_decode < 1 || c->max_running < 1) return false;
  if (c->route != OUTLETS_ROUTE_RR && c->route != OUTLETS_ROUTE_LB) return false;
  if (c->order != OUTLETS_ORDER_FCFS && c->order != OUTLETS_ORDER_SJF) return false;
  const double k[] = {c->pf_base_s, c->pf_per_token_s, c->step_base_s, c->step_per_seq_s, c->step_per_kv_token_s};
  for (double v : k)
    if (!std::isfinite(v) || v < 0) return false;
  for (int i = 0; i < n; ++i) {
    if (!std::isfinite(a[i]) || p[i] < 0 || o[i] < 1) return false;
    if (!std::isfinite(r[i]) || r[i] < 0 || r[i] > 2e9f) return false;
  }
  return true;
}

}  // namespace

extern "C" outlets_status outlets_sched_simulate(const outlets_sched_config* cfg, int32_t n, const double* arrival,
                                                 const int32_t* prompt, const int32_t* output, const float* predicted,
                                                 double* finish, int32_t* instance) {
  if (!cfg || n < 0) return OUTLETS_EINVAL;
  if (n == 0) return OUTLETS_OK;
  if (!arrival || !prompt || !output || !predicted || !finish || !instance) return OUTLETS_EINVAL;
  if (!valid(cfg, n, arrival, prompt, output, predicted)) return OUTLETS_EINVAL;

  std::vector<long long> cost(n);
  for (int i = 0; i < n; ++i) cost[i] = (long long)std::ceil((double)predicted[i]);

  // prefill: one instance, arrival order
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::sort(order.begin(), order.end(), [&](int x, int y) {
    return arrival[x] < arrival[y] || (arrival[x] == arrival[y] && x < y);
  });
  std::vector<double> ready(n);
  double t = -std::numeric_limits<double>::infinity();
  for (int i : order) {
    const double start = arrival[i] > t ? arrival[i] : t;
    const double svc = cfg->pf_base_s + cfg->pf_per_token_s * (double)prompt[i];
    t = start + svc;
    ready[i] = t;
  }
  std::vector<int> arr(n);
  for (int i = 0; i < n; ++i) arr[i] = i;
  std::sort(arr.begin(), arr.end(), [&](int x, int y) {
    return ready[x] < ready[y] || (ready[x] == ready[y] && x < y);
  });

  const int nd = cfg->n_decode;
  const bool sjf = cfg->order == OUTLETS_ORDER_SJF;
  std::vector<Instance> I(nd);
  std::vector<long long> gen(n, 0);
  auto key = [&](int i) { return std::make_tuple(sjf ? cost[i] : 0LL, ready[i], i); };

  auto start_step = [&](int j, double tt) {
    Instance& x = I[j];
    while (!x.waiting.empty() && (int)x.running.size() < cfg->max_running) {
      const int best = std::get<2>(*x.waiting.begin());
      x.waiting.erase(x.waiting.begin());
      x.running.push_back(best);  // its cost stays in load (not yet generated anything)
    }
    if (x.running.empty()) {
      x.busy = false;
      return;
    }
    long long kv = 0;
    for (int r : x.running) kv += (long long)prompt[r] + gen[r];
    const double dt = cfg->step_base_s + cfg->step_per_seq_s * (double)x.running.size() +
                      cfg->step_per_kv_token_s * (double)kv;
    x.step_end = tt + dt;
    x.busy = true;
  };

  int a = 0;
  long long rr = 0;
  while (true) {
    int jn = -1;
    double tn = std::numeric_limits<double>::infinity();
    for (int j = 0; j < nd; ++j)
      if (I[j].busy && I[j].step_end < tn) {
        jn = j;
        tn = I[j].step_end;
      }
    if (a < n && ready[arr[a]] < tn) {
      const int i = arr[a++];
      int j = 0;
      if (cfg->route == OUTLETS_ROUTE_RR) {
        j = (int)(rr % nd);
        ++rr;
      } else {
        for (int j2 = 1; j2 < nd; ++j2)
          if (I[j2].load < I[j].load) j = j2;
      }
      instance[i] = j;
      I[j].waiting.insert(key(i));
      I[j].load += cost[i];
      if (!I[j].busy) start_step(j, ready[i]);
      continue;
    }
    if (jn < 0) break;
    Instance& x = I[jn];
    std::vector<int> still;
    still.reserve(x.running.size());
    for (int r : x.running) {
      if (gen[r] < cost[r]) x.load -= 1;  // one predicted token spent
      gen[r] += 1;
      if (gen[r] >= output[r]) {
        finish[r] = tn;
        x.load -= std::max(cost[r] - gen[r], 0LL);  // what was left of its prediction
      } else {
        still.push_back(r);
      }
    }
    x.running.swap(still);
    start_step(jn, tn);
  }
  return OUTLETS_OK;
}
