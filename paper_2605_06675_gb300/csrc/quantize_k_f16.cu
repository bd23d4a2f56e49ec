// quantize_pack_kernel<__half, unrotated>: one instance per translation
// unit so the instances compile in parallel.
#include "quantize_kernel.cuh"

namespace rq {
rq_status launch_quantize_f16(const QuantArgs& a, cudaStream_t s) {
  return launch_persistent(quantize_pack_kernel<__half, false>, a, quant_smem_bytes(false), s);
}
}  // namespace rq
