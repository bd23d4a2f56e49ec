// quantize_pack_kernel<__nv_bfloat16, rotated> for layers whose keys and values are both
// Lloyd-Max: its own translation unit, compiled in parallel with the others.
#include "quantize_kernel.cuh"

namespace rq {
rq_status launch_quantize_lm_bf16_rot(const QuantArgs& a, cudaStream_t s) {
  return launch_persistent(quantize_pack_kernel<__nv_bfloat16, true, true>, a, quant_smem_bytes(true), s);
}
}  // namespace rq
