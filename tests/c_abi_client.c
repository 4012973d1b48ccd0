/* A plain C99 client of the C ABI (include/deepshift.h), built and run by
 * tests/test_abi.py without a GPU: the size queries, and argument validation
 * that answers before any CUDA call.  Exit status 0 when every answer is the
 * documented one; otherwise the number of the first failed check. */
#include <stdio.h>
#include <string.h>

#include "deepshift.h"

int main(void) {
  ds_weights w;
  memset(&w, 0, sizeof(w));
  if (ds_version() <= 0) return 1;
  if (ds_abi_struct_size(0) != sizeof(ds_weights) || ds_abi_struct_size(1) != sizeof(ds_layer)) return 2;
  /* a 4 x 40 code matrix: 2 chunks of 32 reduction indices, packed into whole 256-byte blocks */
  if (ds_packed_weight_bytes(4, 40) == 0 || ds_packed_weight_bytes(4, 40) % 256 != 0) return 3;
  if (ds_packed_weight_bytes(0, 40) != 0) return 4;
  if (ds_expanded_weight_bytes(64, 1024) != (size_t)2 * 1024 * 64 * 4) return 5;
  /* validation errors come back as statuses with a message, before anything reaches the GPU */
  if (ds_linear_shift(NULL, &w, NULL, NULL, 1, 1, 1, 0, NULL, NULL) != DS_ERR_INVALID_ARG) return 6;
  if (ds_last_error()[0] == '\0') return 7;
  if (ds_conv2d_shift((const int32_t*)16, &w, NULL, NULL, (int32_t*)4096, 1, 1, 8, 8, 1, 3, 3, 1, 1, 0x40000005, 0,
                      0, NULL, NULL) != DS_ERR_UNSUPPORTED)
    return 8; /* padded extent beyond 2^31 - 1 */
  if (ds_quantize_shift_weights((const float*)16, 4, -16, (int8_t*)16, (int8_t*)32, NULL) != DS_ERR_INVALID_ARG)
    return 9; /* p_min outside [-15, 0] */
  if (ds_shift_forward_workspace_bytes(NULL, 0, 1) != 0) return 10;
  printf("c abi client ok (version %d)\n", ds_version());
  return 0;
}
