/* A plain C11 user of the SelKV C ABI: include/selkv.h compiles as C, and the host-side calls
 * (status names, workspace sizes, argument checks that fail before any CUDA call) link and run
 * without a GPU.  Prints one line per check; exits non-zero on the first failure. */
#include <stdio.h>
#include <string.h>

#include "selkv.h"

#define CHECK(cond, what)                              \
  do {                                                 \
    if (!(cond)) {                                     \
      printf("FAIL %s\n", what);                       \
      return 1;                                        \
    }                                                  \
    printf("ok %s\n", what);                           \
  } while (0)

int main(void) {
  selkv_shape s;
  memset(&s, 0, sizeof(s));
  s.dtype = SELKV_BF16;
  s.batch = 1;
  s.num_q_heads = 32;
  s.num_kv_heads = 8;
  s.head_dim = 128;
  s.obs_window = 64;
  s.n_cap = 16384;
  s.m_cap = 4160;

  CHECK(strcmp(selkv_status_string(SELKV_OK), "ok") == 0, "status string");
  const char* name = NULL;
  CHECK(selkv_last_cuda_error(&name) == 0 && name != NULL, "no CUDA error recorded");
  CHECK(selkv_compress_workspace_size(&s) > 0, "compress workspace size");
  CHECK(selkv_decode_workspace_size(&s) > 0, "decode workspace size");
  CHECK(selkv_score_workspace_size(&s) > 0, "score workspace size");

  /* a NULL query: rejected on the host, nothing enqueued */
  CHECK(selkv_decode_attn(&s, NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, NULL, 0, NULL) ==
            SELKV_ERR_INVALID_ARG,
        "decode rejects NULL tensors");
  s.num_q_heads = 30; /* Hkv must divide Hq */
  CHECK(selkv_decode_workspace_size(&s) == 0, "size query rejects Hq % Hkv != 0");
  printf("done\n");
  return 0;
}
