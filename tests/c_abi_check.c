/* Uses include/smetric.h from plain C (no CUDA headers, no C++) and links
 * libsmetric.so: prints the layout of every public struct and the enum
 * values, then makes the calls whose refusals need no GPU. The pytest in
 * test_abi.py compiles it with -std=c99 -pedantic -Werror, runs it on the
 * CPU and compares what it prints with the Python binding. */
#include <stddef.h>
#include <stdio.h>
#include <string.h>

#include "smetric.h"

#define FIELD(T, f) printf("offset %s.%s %zu %zu\n", #T, #f, offsetof(T, f), sizeof(((T*)0)->f))

int main(void) {
  smetric_index* out = (smetric_index*)&out; /* must come back NULL */
  smetric_index_config cfg;
  smetric_weights w = {1, 4, 2};
  int rc;

  printf("sizeof smetric_index_config %zu\n", sizeof(smetric_index_config));
  FIELD(smetric_index_config, num_instances);
  FIELD(smetric_index_config, block_size);
  FIELD(smetric_index_config, session_blocks);
  FIELD(smetric_index_config, flags);
  FIELD(smetric_index_config, capacity_slots);
  FIELD(smetric_index_config, hash_seed);
  FIELD(smetric_index_config, max_batch_requests);
  FIELD(smetric_index_config, max_batch_tokens);
  printf("sizeof smetric_weights %zu\n", sizeof(smetric_weights));
  FIELD(smetric_weights, w_load);
  FIELD(smetric_weights, w_miss);
  FIELD(smetric_weights, w_glob);
  printf("sizeof smetric_policy %zu\n", sizeof(smetric_policy));
  FIELD(smetric_policy, c_lin);
  FIELD(smetric_policy, c_att);
  FIELD(smetric_policy, ttft_d0);
  FIELD(smetric_policy, ttft_d1);
  FIELD(smetric_policy, hit_num);
  FIELD(smetric_policy, hit_den);
  FIELD(smetric_policy, rr_base);
  FIELD(smetric_policy, reserved);
  printf("enum SMETRIC_OK %d\nenum SMETRIC_ERR_INVALID_ARG %d\nenum SMETRIC_ERR_OOM %d\n", SMETRIC_OK,
         SMETRIC_ERR_INVALID_ARG, SMETRIC_ERR_OOM);
  printf("enum SMETRIC_ERR_TABLE_FULL %d\nenum SMETRIC_ERR_CUDA %d\nenum SMETRIC_ERR_OVERFLOW %d\n",
         SMETRIC_ERR_TABLE_FULL, SMETRIC_ERR_CUDA, SMETRIC_ERR_OVERFLOW);
  printf("enum SMETRIC_ERR_TOO_LARGE %d\n", SMETRIC_ERR_TOO_LARGE);

  /* refusals that return before any CUDA call */
  memset(&cfg, 0, sizeof cfg);
  cfg.num_instances = 4;
  cfg.block_size = 7; /* odd: invalid */
  cfg.session_blocks = 1;
  cfg.capacity_slots = 64;
  rc = smetric_index_create(&cfg, &out);
  printf("call create_odd_block %d %d\n", rc, out == NULL);
  rc = smetric_route_batch(NULL, NULL, 0, NULL, 0, NULL, w, NULL, NULL, NULL, NULL, NULL, 0, NULL);
  printf("call route_null_index %d\n", rc);
  rc = smetric_index_destroy(NULL);
  printf("call destroy_null %d\n", rc);
  printf("strerror %s\n", smetric_strerror(SMETRIC_ERR_TABLE_FULL));
  return 0;
}
