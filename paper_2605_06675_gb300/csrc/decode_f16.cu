// Decode attention kernels, fp16 queries and caches (one translation unit per dtype).
#include "decode_kernel.cuh"

namespace rq {

rq_status launch_decode_f16(const dk::DecodeArgs& a, float* out, const void* res_layer, int R,
                         cudaStream_t s) {
  return dk::launch_decode_t<__half>(a, out, res_layer, R, s);
}

}  // namespace rq
