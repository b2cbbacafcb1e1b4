// Tensor-core certified decode (bf16): placeholder until the TMA/mma path lands.
#include "decode.cuh"
#include "internal.h"

namespace ebd {

bool fast_decode_supported(ebd_dtype, int, int, int) { return false; }
void fast_decode_plan(DecodePlan&, long long, int, int, int) {}
ebd_status launch_fast_decode(ebd_dtype, int, const DecodePlan&, const DecodeArgs&, int,
                              cudaStream_t) {
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
