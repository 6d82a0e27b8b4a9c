/* A C99 caller of the library that needs no GPU: it includes every public
 * header, rejects a bad slice configuration, runs the layer allocator (host
 * code) on a small problem and prints what it got, one fact per line, then
 * the size and field offsets of every public struct. */
#include <stddef.h>
#include <stdio.h>
#include <string.h>

#include "sky_alloc.h"
#include "sky_ops.h"
#include "sky_slice.h"

int main(void) {
  sky_slice_config cfg;
  sky_slice* s = NULL;
  int32_t pi[4];
  double dt[3] = {1.0, 3.0, 1.0}, dm[3] = {100.0, 100.0, 100.0}, ct[3] = {0.0, 0.0, 0.0};
  double lf[9] = {1, 1, 1, 1, 1, 1, 1, 1, 1}, lm[9] = {1, 1, 1, 1, 1, 1, 1, 1, 1};
  sky_alloc_problem p;
  sky_status st;

  memset(&cfg, 0, sizeof cfg);
  cfg.width = 768;
  cfg.heads = 5; /* 768 % 5 != 0 */
  cfg.ffn = 3072;
  cfg.layer_begin = 0;
  cfg.layer_end = 4;
  cfg.max_batch = 8;
  cfg.max_seq = 128;
  cfg.dtype = SKY_DTYPE_BF16;
  cfg.ln_eps = 1e-12f;
  st = sky_slice_create(&cfg, &s);
  printf("create %s %d\n", sky_status_string(st), s == NULL);

  st = sky_alloc_even(9, 3, pi);
  printf("even %s %d %d %d %d\n", sky_status_string(st), pi[0], pi[1], pi[2], pi[3]);

  p.devices = 3;
  p.layers = 9;
  p.dt = dt;
  p.dm = dm;
  p.ct = ct;
  p.lf = lf;
  p.lm = lm;
  st = sky_alloc_heuristic(&p, 100, pi);
  printf("heuristic %s %d %d %d %d\n", sky_status_string(st), pi[0], pi[1], pi[2], pi[3]);
  printf("launches %lld\n", (long long)sky_launch_count());

#define OFF(T, f) (unsigned long)offsetof(T, f)
  printf("layout sky_slice_config %lu %lu %lu %lu %lu %lu %lu %lu %lu %lu %lu %lu\n",
         (unsigned long)sizeof(sky_slice_config), OFF(sky_slice_config, width),
         OFF(sky_slice_config, heads), OFF(sky_slice_config, ffn),
         OFF(sky_slice_config, layer_begin), OFF(sky_slice_config, layer_end),
         OFF(sky_slice_config, max_batch), OFF(sky_slice_config, max_seq),
         OFF(sky_slice_config, dtype), OFF(sky_slice_config, ln_eps),
         OFF(sky_slice_config, io_fp32), OFF(sky_slice_config, stash_slots));
  printf("layout sky_layer_cost %lu %lu %lu %lu %lu %lu %lu %lu %lu %lu %lu\n",
         (unsigned long)sizeof(sky_layer_cost), OFF(sky_layer_cost, layer),
         OFF(sky_layer_cost, _pad), OFF(sky_layer_cost, fwd_ms), OFF(sky_layer_cost, bwd_ms),
         OFF(sky_layer_cost, fwd_flops), OFF(sky_layer_cost, bwd_flops),
         OFF(sky_layer_cost, param_bytes), OFF(sky_layer_cost, grad_bytes),
         OFF(sky_layer_cost, stash_bytes), OFF(sky_layer_cost, workspace_bytes));
  printf("layout sky_kernel_stat %lu %lu %lu %lu %lu %lu\n",
         (unsigned long)sizeof(sky_kernel_stat), OFF(sky_kernel_stat, name),
         OFF(sky_kernel_stat, launches), OFF(sky_kernel_stat, total_ms),
         OFF(sky_kernel_stat, flops), OFF(sky_kernel_stat, bytes));
  printf("layout sky_optimizer_config %lu %lu %lu %lu %lu %lu %lu %lu\n",
         (unsigned long)sizeof(sky_optimizer_config), OFF(sky_optimizer_config, kind),
         OFF(sky_optimizer_config, lr), OFF(sky_optimizer_config, beta1),
         OFF(sky_optimizer_config, beta2), OFF(sky_optimizer_config, eps),
         OFF(sky_optimizer_config, weight_decay), OFF(sky_optimizer_config, momentum));
  printf("layout sky_alloc_problem %lu %lu %lu %lu %lu %lu %lu %lu\n",
         (unsigned long)sizeof(sky_alloc_problem), OFF(sky_alloc_problem, devices),
         OFF(sky_alloc_problem, layers), OFF(sky_alloc_problem, dt), OFF(sky_alloc_problem, dm),
         OFF(sky_alloc_problem, ct), OFF(sky_alloc_problem, lf), OFF(sky_alloc_problem, lm));
  return 0;
}
