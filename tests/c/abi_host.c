/* A C99 caller of the library that needs no GPU: it includes every public
 * header, rejects a bad slice configuration, runs the layer allocator (host
 * code) on a small problem and prints what it got, one fact per line. */
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
  return 0;
}
