// Host side of decode attention: the split plan of a call, workspace
// layout, argument checks and the C entry points. The kernels are in
// decode_kernel.cuh (one instance per input dtype: decode_f16.cu,
// decode_bf16.cu).
#include <algorithm>
#include <atomic>

#include "decode_kernel.cuh"

namespace rq {

rq_status current_sm_count(int* sms) {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) {
      *sms = c;
      return RQ_OK;
    }
  }
  int v = 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
    return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) cache[dev].store(v, std::memory_order_relaxed);
  *sms = v;
  return RQ_OK;
}
namespace {

using dk::DecodeArgs;
using dk::kMaxHeads;
using dk::kPart;

// Resident splits per SM on the current device (cached per device): resident
// split-kernel CTAs x the split groups of a CTA.
rq_status split_ctas_per_sm(int* per_sm) {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) {
      *per_sm = c;
      return RQ_OK;
    }
  }
  int v = 0;
  if (decode_split_ctas_per_sm(&v) != RQ_OK) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) cache[dev].store(v, std::memory_order_relaxed);
  *per_sm = v;
  return RQ_OK;
}

struct SplitPlan {
  int splits, bps;      // units [u_lo, B * H_kv): splits and blocks per split
  int s_lo, bps_lo;     // units [0, u_lo)
  int u_lo;
};

// Splits of the sequence per (batch, kv head) unit: as many as fit in one
// wave of resident splits (slots = SMs x splits per SM), so every split
// streams a long run of blocks and none waits for a second wave; at least one
// per unit. When the units do not divide the slots, the wave is filled with
// two split counts: units [0, u_lo) take s_lo = slots / units splits and the
// rest s_lo + 1, so that every SM holds the same number of splits (units x
// s_lo splits would leave some SMs one split short and the others, with
// their full complement, setting the time). The s_lo-split units' splits
// (the larger ones) come first in the plan; the kernel gives consecutive
// splits to the groups of a CTA, so a CTA holds splits of one size.
// nblk: the packed blocks attended (<= the capacity's); splits <= the
// capacity's split bound (max_splits), which sizes the workspace.
int max_splits(const rq_cache_desc* desc, int slots) {
  const long long units = static_cast<long long>(desc->B) * desc->H_kv;
  long long sp = units > 0 ? slots / units : 1;
  if (units > 0 && units <= slots && slots % units != 0) ++sp;
  return static_cast<int>(std::max<long long>(1, std::min<long long>(sp, desc->S / kTile)));
}

namespace {
// blocks per CTA and the resulting split count for sp requested splits
void split_even(int nblk, long long sp, int* splits, int* bps) {
  sp = std::max<long long>(1, std::min<long long>(sp, nblk));
  *bps = std::max(1, static_cast<int>((nblk + sp - 1) / sp));
  *splits = std::max(1, (nblk + *bps - 1) / *bps);
}
}  // namespace

SplitPlan decode_plan(const rq_cache_desc* desc, int nblk, int slots) {
  SplitPlan p;
  const long long units = static_cast<long long>(desc->B) * desc->H_kv;
  const long long sp = units > 0 ? slots / units : 1;
  split_even(nblk, sp, &p.splits, &p.bps);
  p.s_lo = p.splits;
  p.bps_lo = p.bps;
  p.u_lo = static_cast<int>(units);
  if (units > 0 && units <= slots && slots % units != 0 && sp < nblk) {
    int s_hi = 1, bps_hi = 1;
    split_even(nblk, sp + 1, &s_hi, &bps_hi);
    if (s_hi > p.s_lo) {
      p.splits = s_hi;
      p.bps = bps_hi;
      p.u_lo = static_cast<int>(units - (slots - units * sp));
    }
  }
  return p;
}

rq_status decode_slots(int* slots) {
  int sms = 0, per_sm = 0;
  if (current_sm_count(&sms) != RQ_OK || split_ctas_per_sm(&per_sm) != RQ_OK) return RQ_ERR_CUDA;
  *slots = sms * per_sm;
  return RQ_OK;
}

rq_status check_desc(const rq_cache_desc* desc) {
  if (!desc) return RQ_ERR_INVALID_ARG;
  if (desc->L <= 0 || desc->B < 0 || desc->H_kv <= 0 || desc->H_q <= 0 || desc->S < 0)
    return RQ_ERR_INVALID_ARG;
  if (desc->dtype != RQ_F16 && desc->dtype != RQ_BF16) return RQ_ERR_INVALID_ARG;
  for (int g : {desc->k_grouping, desc->v_grouping})
    if (!grouping_ok(g)) return RQ_ERR_INVALID_ARG;
  if (!quantizers_ok(desc->k_quantizer, desc->k_grouping, desc->v_quantizer, desc->v_grouping))
    return RQ_ERR_INVALID_ARG;
  if (desc->d != kD || desc->group != kG || desc->S % kTile != 0 || desc->S == 0)
    return RQ_ERR_SHAPE;
  if (desc->H_q % desc->H_kv != 0 || desc->H_q / desc->H_kv > kMaxHeads) return RQ_ERR_SHAPE;
  return RQ_OK;
}

// Workspace: the split records [B][H_q][splits][132] fp32.
size_t workspace_bytes(const rq_cache_desc* desc, int splits) {
  return static_cast<size_t>(desc->B) * desc->H_q * splits * kPart * sizeof(float);
}

// rq_decode_set_pattern's setting
std::atomic<int> g_decode_pattern{RQ_DECODE_BACK_TO_BACK};

void fill_args(DecodeArgs& a, const rq_cache_desc* desc, int32_t layer, const void* q,
               const void* packed, const uint8_t* bits_dev, const uint64_t* offsets_dev,
               const int8_t* signs_dev, void* ws, uint32_t* status_dev, const SplitPlan& plan) {
  a.q = q;
  a.packed = static_cast<const uint8_t*>(packed);
  a.bits = bits_dev;
  a.offsets = offsets_dev;
  a.signs = signs_dev;
  a.partial = static_cast<float*>(ws);
  a.n_rows = nullptr;
  a.status = status_dev;
  a.layer = layer;
  a.B = desc->B;
  a.H = desc->H_kv;
  a.Hq = desc->H_q;
  a.g = desc->H_q / desc->H_kv;
  a.nblk = desc->S / kTile;
  a.splits = plan.splits;
  a.bps = plan.bps;
  a.s_lo = plan.s_lo;
  a.bps_lo = plan.bps_lo;
  a.u_lo = plan.u_lo;
  a.kg = stored_grouping(desc->k_grouping);   // wide per-token groups are stored as groups of 32
  a.vg = stored_grouping(desc->v_grouping);
  a.hadamard = desc->hadamard ? 1 : 0;
  a.mix = g_decode_pattern.load(std::memory_order_relaxed) == RQ_DECODE_INTERLEAVED ? 1 : 0;
  a.kq = desc->k_quantizer;
  a.vq = desc->v_quantizer;
  if (a.kq == RQ_LLOYDMAX || a.vq == RQ_LLOYDMAX) fill_lm_book(a.lm);
}

// split kernel, then the merge kernel as its programmatic dependent
rq_status launch_decode(const DecodeArgs& a, const rq_cache_desc* desc, float* out, cudaStream_t s,
                        const void* res_layer = nullptr, int R = 0) {
  return desc->dtype == RQ_F16 ? launch_decode_f16(a, out, res_layer, R, s)
                               : launch_decode_bf16(a, out, res_layer, R, s);
}

}  // namespace
}  // namespace rq

extern "C" rq_status rq_decode_set_pattern(int32_t pattern) {
  if (pattern != RQ_DECODE_BACK_TO_BACK && pattern != RQ_DECODE_INTERLEAVED) return RQ_ERR_INVALID_ARG;
  rq::g_decode_pattern.store(pattern, std::memory_order_relaxed);
  return RQ_OK;
}

extern "C" rq_status rq_decode_workspace_bytes(const rq_cache_desc* desc, size_t* bytes) {
  using namespace rq;
  if (!bytes) return RQ_ERR_INVALID_ARG;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  int slots = 0;
  if (decode_slots(&slots) != RQ_OK) return RQ_ERR_CUDA;
  *bytes = workspace_bytes(desc, max_splits(desc, slots));
  return RQ_OK;
}

extern "C" rq_status rq_decode_attention(const rq_cache_desc* desc, int32_t layer, const void* q,
                                         const void* packed, const uint8_t* bits_dev,
                                         const uint64_t* offsets_dev, const int8_t* signs_dev,
                                         float* out, void* ws, size_t ws_bytes,
                                         uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!q || !packed || !bits_dev || !offsets_dev || !out || !ws) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || !aligned16(ws) || (reinterpret_cast<uintptr_t>(q) & 1u) ||
      (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int slots = 0;
  if (decode_slots(&slots) != RQ_OK) return RQ_ERR_CUDA;
  const SplitPlan plan = decode_plan(desc, desc->S / kTile, slots);
  if (ws_bytes < workspace_bytes(desc, plan.splits)) return RQ_ERR_WORKSPACE;
  DecodeArgs a;
  fill_args(a, desc, layer, q, packed, bits_dev, offsets_dev, signs_dev, ws, status_dev, plan);
  return launch_decode(a, desc, out, static_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// Allocation-free decode: the split-K partials live in a fixed device array
// of this library instead of a caller-supplied workspace, for callers that
// cannot allocate (runtimes whose allocator belongs to someone else, plugins
// handed only their inputs and outputs). The array is shared by every call
// on a device.
namespace rq {
namespace {

constexpr size_t kStaticScratchFloats = RQ_STATIC_SCRATCH_BYTES / sizeof(float);
static __device__ __align__(256) float g_decode_scratch[kStaticScratchFloats];

// device address of g_decode_scratch for the current device, looked up once
// per device (host code only sees a host-side stand-in for the symbol)
rq_status static_scratch_ptr(float** ptr) {
  static std::atomic<uintptr_t> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) {
    const uintptr_t c = cache[dev].load(std::memory_order_acquire);
    if (c != 0) {
      *ptr = reinterpret_cast<float*>(c);
      return RQ_OK;
    }
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return RQ_ERR_CUDA;
  if (dev >= 0 && dev < 64) cache[dev].store(reinterpret_cast<uintptr_t>(p), std::memory_order_release);
  *ptr = static_cast<float*>(p);
  return RQ_OK;
}

}  // namespace
}  // namespace rq

extern "C" rq_status rq_decode_attention_static(const rq_cache_desc* desc, int32_t layer,
                                                const void* q, const void* packed,
                                                const uint8_t* bits_dev,
                                                const uint64_t* offsets_dev,
                                                const int8_t* signs_dev, float* out,
                                                uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!q || !packed || !bits_dev || !offsets_dev || !out) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || (reinterpret_cast<uintptr_t>(q) & 1u) ||
      (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int slots = 0;
  if (decode_slots(&slots) != RQ_OK) return RQ_ERR_CUDA;
  const SplitPlan plan = decode_plan(desc, desc->S / kTile, slots);
  if (workspace_bytes(desc, plan.splits) > RQ_STATIC_SCRATCH_BYTES) return RQ_ERR_WORKSPACE;
  float* scratch = nullptr;
  if (static_scratch_ptr(&scratch) != RQ_OK) return RQ_ERR_CUDA;
  DecodeArgs a;
  fill_args(a, desc, layer, q, packed, bits_dev, offsets_dev, signs_dev, scratch, status_dev, plan);
  return launch_decode(a, desc, out, static_cast<cudaStream_t>(stream));
}

// ------------------------------------------------- decode over n_tokens ----
extern "C" rq_status rq_decode_attention_len(const rq_cache_desc* desc, int32_t layer,
                                             int32_t n_tokens, const void* q, const void* packed,
                                             const uint8_t* bits_dev, const uint64_t* offsets_dev,
                                             const int8_t* signs_dev, const void* residual,
                                             float* out, void* ws, size_t ws_bytes,
                                             uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!q || !packed || !bits_dev || !offsets_dev || !out || !ws) return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L || n_tokens < 1 || n_tokens > desc->S) return RQ_ERR_INVALID_ARG;
  const int R = n_tokens % kTile;
  if (R > 0 && !residual) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || !aligned16(ws) || (R > 0 && !aligned16(residual)) ||
      (reinterpret_cast<uintptr_t>(q) & 1u) || (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int slots = 0;
  if (decode_slots(&slots) != RQ_OK) return RQ_ERR_CUDA;
  const int nblk = n_tokens / kTile;
  const SplitPlan plan = decode_plan(desc, nblk, slots);
  if (ws_bytes < workspace_bytes(desc, plan.splits)) return RQ_ERR_WORKSPACE;
  DecodeArgs a;
  fill_args(a, desc, layer, q, packed, bits_dev, offsets_dev, signs_dev, ws, status_dev, plan);
  a.nblk = nblk;
  // this layer's residual windows: [B][H][2][32][128] values of the cache dtype
  const void* res_layer =
      R > 0 ? static_cast<const uint8_t*>(residual) +
                  static_cast<size_t>(layer) * desc->B * desc->H_kv * 2 * kTile * kD * 2
            : nullptr;
  return launch_decode(a, desc, out, static_cast<cudaStream_t>(stream), res_layer, R);
}


// --------------------------------------- decode with a token count per row ----
extern "C" rq_status rq_decode_attention_rows(const rq_cache_desc* desc, int32_t layer,
                                              const int32_t* n_dev, const void* q,
                                              const void* packed, const uint8_t* bits_dev,
                                              const uint64_t* offsets_dev, const int8_t* signs_dev,
                                              const void* residual, float* out, void* ws,
                                              size_t ws_bytes, uint32_t* status_dev, void* stream) {
  using namespace rq;
  const rq_status st = check_desc(desc);
  if (st != RQ_OK) return st;
  if (!n_dev || !q || !packed || !bits_dev || !offsets_dev || !residual || !out || !ws)
    return RQ_ERR_INVALID_ARG;
  if (layer < 0 || layer >= desc->L) return RQ_ERR_INVALID_ARG;
  if (!aligned16(packed) || !aligned16(ws) || !aligned16(residual) ||
      (reinterpret_cast<uintptr_t>(n_dev) & 3u) || (reinterpret_cast<uintptr_t>(q) & 1u) ||
      (reinterpret_cast<uintptr_t>(out) & 3u))
    return RQ_ERR_ALIGNMENT;
  if (desc->B == 0) return RQ_OK;
  int slots = 0;
  if (decode_slots(&slots) != RQ_OK) return RQ_ERR_CUDA;
  // the split plan of the capacity; each row's CTAs stop at its own length
  const int nblk = desc->S / kTile;
  const SplitPlan plan = decode_plan(desc, nblk, slots);
  if (ws_bytes < workspace_bytes(desc, plan.splits)) return RQ_ERR_WORKSPACE;
  DecodeArgs a;
  fill_args(a, desc, layer, q, packed, bits_dev, offsets_dev, signs_dev, ws, status_dev, plan);
  a.n_rows = n_dev;
  const void* res_layer = static_cast<const uint8_t*>(residual) +
                          static_cast<size_t>(layer) * desc->B * desc->H_kv * 2 * kTile * kD * 2;
  return launch_decode(a, desc, out, static_cast<cudaStream_t>(stream), res_layer, 0);
}
