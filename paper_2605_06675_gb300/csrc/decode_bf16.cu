// Decode attention kernels, bf16 queries and caches (one translation unit per dtype).
#include "decode_kernel.cuh"

namespace rq {

rq_status launch_decode_bf16(const dk::DecodeArgs& a, float* out, const void* res_layer, int R,
                         cudaStream_t s) {
  return dk::launch_decode_t<__nv_bfloat16>(a, out, res_layer, R, s);
}

rq_status decode_split_ctas_per_sm(int* per_sm) { return dk::split_ctas_per_sm_t<__nv_bfloat16>(per_sm); }

}  // namespace rq
