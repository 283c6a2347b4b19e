/* A plain C consumer of include/budgetdraft.h: compiled by tests/test_abi.py with gcc
 * against the built library, it calls the entry points that need no GPU (sizes of a
 * rejected shape, argument validation, status strings) and prints one line per check. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "budgetdraft.h"

int main(void) {
  bd_shape s;
  memset(&s, 0, sizeof(s));
  s.batch = 2;
  s.h_q = 8;
  s.h_kv = 2;
  s.head_dim = 96; /* unsupported: every call must refuse it before touching a device */
  s.t_ctx = 100;
  s.t_cap = 110;
  s.seq_lens = NULL;
  void* fake = (void*)(uintptr_t)0x10000;
  printf("workspace_size %zu\n", bd_workspace_size(&s, BD_OP_VERIFY, 1, 6));
  printf("verify %d\n", bd_verify_attn(&s, fake, 6, fake, fake, fake, (float*)fake, fake, 1 << 20, NULL));
  printf("argmax %d\n", bd_argmax(fake, 3, 4, 100, (int32_t*)fake, NULL));
  printf("accept_empty %d\n", bd_accept(0, 5, NULL, NULL, NULL, NULL, NULL));
  printf("strerror %s\n", bd_strerror(BD_ERR_MISALIGNED));
  return 0;
}
