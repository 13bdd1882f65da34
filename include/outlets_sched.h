/*
 * Serving-side use of the static length prediction (Sec. 5.3 and the appendix
 * "System-Level Evaluation Details"): a discrete-event model of a disaggregated
 * deployment (one prefill instance, n decode instances) in which the static
 * prediction r_hat_0 of every request steers
 *   instance routing   RR (fixed cyclic order) or LB (the decode instance with
 *                      the lowest predicted remaining workload of its queued
 *                      and running requests), and
 *   queue order        FCFS (arrival order) or SJF (shortest predicted first).
 * Host code only (no GPU); part of the same library as outlets.h.
 *
 * Model (the paper runs the policies inside vLLM and gives no simulator):
 *  - prefill: one instance, one request at a time in arrival order (ties: lower
 *    index), service pf_base_s + pf_per_token_s * prompt_len;
 *  - decode: continuous batching; a step gives every running request one token
 *    and lasts step_base_s + step_per_seq_s * |R| + step_per_kv_token_s *
 *    sum_{r in R} (prompt_len_r + generated_r); at a step boundary finished
 *    requests leave, then waiting requests are admitted (FCFS / SJF) while
 *    fewer than max_running run, then the next step starts; an idle instance
 *    starts when a request arrives; no preemption;
 *  - a request needs output_len (>= 1) decode tokens;
 *  - the LB cost of a request is ceil(predicted_len) tokens; a running request
 *    counts max(cost - generated, 0) as of its instance's last step boundary;
 *    ties go to the lower instance; RR counts requests in the order they reach
 *    the decode tier (prefill finish time, then index);
 *  - SJF admits by (cost, decode arrival time, index), FCFS by (decode arrival
 *    time, index); simultaneous events: step ends first, lower instance first.
 * Results are deterministic and do not depend on the host (IEEE double, no
 * contracted multiply-adds).
 */
#ifndef OUTLETS_SCHED_H_
#define OUTLETS_SCHED_H_

#include <stdint.h>

#include "outlets.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum outlets_route { OUTLETS_ROUTE_RR = 0, OUTLETS_ROUTE_LB = 1 } outlets_route;
typedef enum outlets_order { OUTLETS_ORDER_FCFS = 0, OUTLETS_ORDER_SJF = 1 } outlets_order;

typedef struct outlets_sched_config {
  int32_t n_decode;      /* decode instances, >= 1 (3 in the paper's 1P3D setting) */
  int32_t max_running;   /* requests in a decode instance's continuous batch, >= 1 */
  int32_t route;         /* outlets_route */
  int32_t order;         /* outlets_order */
  double pf_base_s;      /* prefill service time: pf_base_s + pf_per_token_s * prompt_len */
  double pf_per_token_s;
  double step_base_s;    /* decode step time (see above), all >= 0 */
  double step_per_seq_s;
  double step_per_kv_token_s;
} outlets_sched_config;

/* Simulates n requests (host arrays, caller-owned):
 *   arrival_s [n] (finite), prompt_len [n] (>= 0), output_len [n] (>= 1),
 *   predicted_len [n] (finite, >= 0: e.g. the len_out of
 *   outlets_predict_prefill for each request)
 * and writes finish_s [n] (time the last token is generated) and instance [n]
 * (decode instance).  Errors: OUTLETS_EINVAL for NULL pointers, n < 0 or a
 * value outside its range (nothing is written). */
outlets_status outlets_sched_simulate(const outlets_sched_config* cfg, int32_t n, const double* arrival_s,
                                      const int32_t* prompt_len, const int32_t* output_len,
                                      const float* predicted_len, double* finish_s, int32_t* instance);

#ifdef __cplusplus
}
#endif

#endif /* OUTLETS_SCHED_H_ */
