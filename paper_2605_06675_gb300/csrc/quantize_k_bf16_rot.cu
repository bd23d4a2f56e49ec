// quantize_pack_kernel<__nv_bfloat16, rotated>: one instance per translation
// unit so the instances compile in parallel.
#include "quantize_kernel.cuh"

namespace rq {
rq_status launch_quantize_bf16_rot(const QuantArgs& a, cudaStream_t s) {
  return launch_persistent(quantize_pack_kernel<__nv_bfloat16, true>, a, quant_smem_bytes(true), s);
}
}  // namespace rq
