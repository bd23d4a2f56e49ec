// quantize_pack_kernel<__half, unrotated> for layers whose keys and values are both
// Lloyd-Max: its own translation unit, compiled in parallel with the others.
#include "quantize_kernel.cuh"

namespace rq {
rq_status launch_quantize_lm_f16(const QuantArgs& a, cudaStream_t s) {
  return launch_persistent(quantize_pack_kernel<__half, false, true>, a, quant_smem_bytes(false), s);
}
}  // namespace rq
