/*
 * sky_alloc.h -- C ABI of the layer allocator of Sky Computing (Sec. IV).
 *
 * A model of L layers is split over D devices by a partition index pi of
 * length D+1 (Sec. IV-D): device i runs layers pi[i] .. pi[i+1]-1, with
 * pi[0] = 0 and pi[D] = L.  On one device that range is what one
 * sky_slice_create(layer_begin = pi[i], layer_end = pi[i+1]) computes, and
 * sky_slice_layer_cost measures the per-layer time, FLOPs and memory that
 * feed lf and lm below.
 *
 * Inputs (Sec. IV-B, IV-D):
 *   dt[i]  benchmark time ratio of device i (larger = slower),
 *   dm[i]  memory available on device i,
 *   ct[i]  communication time of device i,
 *   lf[j]  FLOPs of layer j,  lm[j]  memory needed by layer j
 * (any consistent units).  All arrays are host memory owned by the caller;
 * nothing here allocates device memory or touches a GPU, and every call is
 * thread-safe (no shared state).
 *
 * Errors: SKY_ERR_INVALID_ARG for null pointers, D < 1, L < D, negative or
 * non-finite inputs, or a pi that is not a partition (strictly increasing,
 * pi[0] = 0, pi[D] = L); SKY_ERR_INFEASIBLE when no partition the algorithm
 * can reach fits the memory limits; SKY_ERR_UNSUPPORTED beyond a stated size
 * limit.  On error the output arrays are left unspecified.
 */
#ifndef SKY_ALLOC_H
#define SKY_ALLOC_H

#include <stdint.h>

#include "sky_slice.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t devices;   /* D >= 1                                   */
  int32_t layers;    /* L >= D                                   */
  const double* dt;  /* [D] device benchmark time ratio, > 0     */
  const double* dm;  /* [D] device memory, >= 0                  */
  const double* ct;  /* [D] device communication time, >= 0     */
  const double* lf;  /* [L] layer FLOPs, >= 0                    */
  const double* lm;  /* [L] layer memory, >= 0                   */
} sky_alloc_problem;

/* How a device's communication time enters its workload.  The model of
 * Sec. IV-C charges it once per device: w_i = dt_i * sum_j lf_j + ct_i.  The
 * text before Alg. 2 defines a layer's workload on device i as
 * dt_i * lf_j + ct_i and a device's as the sum over its layers, so ct is
 * charged once per layer; Alg. 2 (sky_alloc_finetune) uses that form. */
typedef enum { SKY_COST_CT_PER_DEVICE = 0, SKY_COST_CT_PER_LAYER = 1 } sky_cost_model;

/* Sec. IV-A: equal layer counts; the first L % D devices get one more layer.
 * pi: [D+1] out. */
sky_status sky_alloc_even(int32_t layers, int32_t devices, int32_t* pi);

/* Alg. 1 (coarse allocation by memory).  Starts from the even partition; each
 * sweep visits boundaries i = 0 .. D-2: while device i exceeds dm[i] and
 * holds more than one layer it gives its last layer to device i+1, then while
 * the next device's first layer still fits (dm[i] > am[i] + lm[pi[i+1]],
 * strict) and device i+1 keeps a layer, device i takes it.  Returns as soon
 * as every device fits; SKY_ERR_INFEASIBLE when a sweep changes nothing.
 * pi: [D+1] out. */
sky_status sky_alloc_coarse(const sky_alloc_problem* p, int32_t* pi);

/* Alg. 2 (optimise workload).  Per sweep the target is the mean device
 * workload (ct per layer).  At boundary i = 0 .. D-2, with workloads
 * recomputed from the current pi: if device i is below target, device i+1
 * keeps a layer and every device still fits after the move, device i takes
 * device i+1's first layer; otherwise, if device i+1 is below target, device
 * i without its last layer is still above target, device i keeps a layer
 * and every device fits, device i gives its last layer away.  Stops after a
 * sweep with no move or after max_iter sweeps (max_iter >= 0).
 * pi: [D+1] in (a partition) and out; sweeps (may be null): sweeps run. */
sky_status sky_alloc_finetune(const sky_alloc_problem* p, int32_t max_iter, int32_t* pi,
                              int32_t* sweeps);

/* Sec. IV-D: Alg. 1, then Alg. 2 with max_iter sweeps.  pi: [D+1] out. */
sky_status sky_alloc_heuristic(const sky_alloc_problem* p, int32_t max_iter, int32_t* pi);

/* Per-device workloads of partition pi under `model`.  w: [D] out. */
sky_status sky_alloc_workloads(const sky_alloc_problem* p, const int32_t* pi, sky_cost_model model,
                               double* w);

/* The best partition in device order: minimises q = max_i (dt_i * sum lf +
 * ct_i) (the Sec. IV-C cost) over every pi with at least one layer per device
 * and every device within memory, by dynamic programming over (device, first
 * layer) in O(D L^2).  This is the optimum of the heuristic's own search
 * space.  pi: [D+1] out; q: out.  SKY_ERR_INFEASIBLE if no such pi fits. */
sky_status sky_alloc_best_ordered(const sky_alloc_problem* p, int32_t* pi, double* q);

/* The mixed-integer model of Sec. IV-C solved exactly: each layer on one
 * device, each device's layers contiguous, memory respected, device order
 * free and empty devices allowed (an empty device still counts ct_i in q, as
 * the constraint q >= dt_i sum_j x_ij lf_j + ct_i reads).  Every device order
 * is tried with the dynamic program above, so D <= 8 (else UNSUPPORTED).
 * owner: [L] out, the device of each layer; q: out. */
sky_status sky_alloc_milp_exact(const sky_alloc_problem* p, int32_t* owner, double* q);

#ifdef __cplusplus
}
#endif

#endif /* SKY_ALLOC_H */
