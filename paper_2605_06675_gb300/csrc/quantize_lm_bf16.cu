// quantize_pack_kernel<__nv_bfloat16, unrotated> for layers whose keys and values are both
// Lloyd-Max: its own translation unit, compiled in parallel with the others.
#include "quantize_kernel.cuh"

namespace rq {
rq_status launch_quantize_lm_bf16(const QuantArgs& a, cudaStream_t s) {
  return launch_persistent(quantize_pack_kernel<__nv_bfloat16, false, true>, a, quant_smem_bytes(false), s);
}
}  // namespace rq
