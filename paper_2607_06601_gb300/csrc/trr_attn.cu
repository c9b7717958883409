// trr_attn.cu - the attention entry points: trr_decode_attn, trr_decode_step,
// trr_decode_attn_routed and trr_decode_attn_static (Sec. 3.2(A), Eq. 2; Sec. 3.8;
// Sec. 7).  The host side of a call: its launches, their shared memory and scratch
// views; the kernels are in trr_attn.cuh, instantiated by the trr_attn_*.cu files.
#include <algorithm>
#include <climits>

#include "trr_attn.cuh"

namespace trr {

// Done once per cache at creation, so that calls stay legal inside stream capture.
cudaError_t attn_configure() {
  cudaError_t (*const parts[])() = {configure_attn_cc, configure_attn_head_modes, configure_attn_mma,
                                     configure_attn_step_cc, configure_attn_step_mma};
  for (auto part : parts) {
    const cudaError_t e = part();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// The tensor-core path serves query groups (g >= 2) whose (head, group) columns fit
// one 8-wide mma tile.
static bool use_mma(const Layout& l) {  // per-head modes: one warp per query head
  return uses_mma(l.Hq, l.Hkv, l.d, l.G, l.head_modes);
}

// Ring bytes an attention call with n queries gets, or -1 when one stage of the
// widest page (one KV slice, its positions) or of the query rows would not fit.
static int attn_ring_bytes(const Layout& l, int n, int hpu, int scr_floats, int fused, int limit) {
  const int fixed = AttnSmem(0, n, scr_floats, fused).total;
  const int ring = (limit - fixed) / 128 * 128;
  const int widest = static_cast<int>(l.slice[3]) + 4 * l.P;
  const int qrows = hpu * 2 * l.d;
  if (ring < std::max(widest, qrows)) return -1;
  return ring;
}

// Queries per launch: their unit tables live in the CTAs' shared memory; a call with
// more queries is cut into launches of this many, chained on the stream.
constexpr int kMaxLaunchQueries = 1024;

static cudaError_t launch_one(const Layout& l, const AttnKernelArgs& ka, int num_sms, cudaStream_t s) {
  const bool mma = use_mma(l);
  const int ctas = mma ? kMmaCtasPerSm : cc_ctas_per_sm(l.d);
  const int ring = attn_ring_bytes(l, ka.n, ka.hpu, ka.scr_floats, ka.fused, attn_smem_limit(ctas));
  if (ring < 0) return cudaErrorInvalidConfiguration;
  AttnKernelArgs k = ka;
  k.ring_bytes = ring;
  const size_t sm = static_cast<size_t>(AttnSmem(ring, k.n, k.scr_floats, k.fused).total);
  const dim3 grid(ctas * num_sms), block(32 * (kNcw + 1));
  if (k.fused) return mma ? launch_attn_step_mma(l, grid, block, sm, s, k) : launch_attn_step_cc(l, grid, block, sm, s, k);
  if (mma) return launch_attn_mma(l, grid, block, sm, s, k);
  return l.head_modes ? launch_attn_head_modes(l, grid, block, sm, s, k) : launch_attn_cc(l, grid, block, sm, s, k);
}

// The launches of an attention call with the given scratch views in `a`; *launches
// counts them.
// `step` (a decode step: k, v, bits given) selects the decode-step kernels, which with
// `early` (the layer's cache state is settled, see cache_layer_settled) read that state
// and issue their first page copies before the previous kernel ends; the other calls
// always wait for it first.
struct StepInputs {
  const void* k;
  const void* v;
  const uint8_t* bits;
};
static cudaError_t launch_attention(const Layout& l, const LayerArgs& a, int num_sms, int n,
                                    const int32_t* seq_ids, const int32_t* q_positions, const void* q_bf16,
                                    const uint8_t* modes, const float* mode_logits, const int32_t* windows,
                                    int window_scalar, float softmax_scale, void* out_bf16, cudaStream_t s,
                                    int* launches, bool early, const StepInputs* step = nullptr) {
  *launches = 0;
  AttnKernelArgs ka;
  ka.a = a;
  ka.window_scalar = window_scalar;
  ka.early = early ? 1 : 0;
  ka.fused = step ? 1 : 0;
  ka.k = step ? static_cast<const uint16_t*>(step->k) : nullptr;
  ka.v = step ? static_cast<const uint16_t*>(step->v) : nullptr;
  ka.bits = step ? step->bits : nullptr;
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.f / sqrtf(static_cast<float>(l.d));
  ka.qscale = scale * 1.4426950408889634f;
  const bool mma = use_mma(l);
  const int g = l.Hq / l.Hkv;
  ka.hpu = mma ? kNcw * g : kNcw;
  ka.defer_merge = mma ? 1 : 0;
  // tensor-core scratch per consumer warp: the query's bf16 words (4 d floats), later
  // the unit's rows (g (d + 4) floats)
  ka.scr_floats = mma ? std::max(4 * l.d, g * (l.d + 4)) : 0;
  const int64_t row = static_cast<int64_t>(l.Hq) * l.d;  // bf16 elements per query
  for (int q0 = 0; q0 < n; q0 += kMaxLaunchQueries) {
    ka.n = std::min(kMaxLaunchQueries, n - q0);
    ka.q0 = q0;
    ka.seq_ids = seq_ids + q0;
    ka.q_positions = q_positions + q0;
    ka.modes = modes ? modes + static_cast<int64_t>(q0) * (l.head_modes ? l.Hq : 1) : nullptr;
    ka.mode_logits = mode_logits ? mode_logits + 3 * q0 : nullptr;
    ka.windows = windows ? windows + q0 : nullptr;
    ka.q = static_cast<const uint16_t*>(q_bf16) + q0 * row;
    ka.out = static_cast<uint16_t*>(out_bf16) + q0 * row;
    ka.a.cnt = a.cnt + static_cast<int64_t>(q0) * l.Hq * l.cnt_stride;
    ka.early = step && early && q0 == 0 ? 1 : 0;  // a later launch follows one on the same layer
    cudaError_t e = launch_one(l, ka, num_sms, s);
    if (e != cudaSuccess) return e;
    ++*launches;
    if (mma) {  // the tensor-core path's splits are merged by the combine kernel
      CombineArgs ca;
      ca.part = a.part;
      ca.qtab = reinterpret_cast<const int2*>(ka.a.cnt);
      ca.out = ka.out;
      ca.Hq = l.Hq;
      const dim3 cgrid(ka.n * l.Hq), cblock(32 * kCombineWarps);
      e = launch_attn_combine(l.d, cgrid, cblock, s, ca);
      if (e != cudaSuccess) return e;
      ++*launches;
    }
  }
  return cudaSuccess;
}

}  // namespace trr

using namespace trr;

extern "C" trr_status trr_decode_attn(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                      const int32_t* q_positions, const void* q_bf16, const uint8_t* modes,
                                      const int32_t* windows, int32_t window_scalar, float softmax_scale,
                                      void* out_bf16, void* stream) {
  if (!cache) return TRR_ERR_INVALID_ARG;
  const Layout& l = cache_layout(cache);
  if (layer < 0 || layer >= l.L || n < 0 || n > l.max_queries) return TRR_ERR_INVALID_ARG;
  cache_set_launches(cache, 0);
  if (n == 0) return TRR_OK;
  if (!seq_ids || !q_positions || !q_bf16 || !modes || !out_bf16) return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(q_bf16) | reinterpret_cast<uintptr_t>(out_bf16)) & 15)
    return TRR_ERR_INVALID_ARG;
  LayerArgs a = layer_args(l, cache_views(cache), layer);
  a.wait_ns = cache_wait_ns(cache);
  cache_note_call(cache, layer);
  int launches = 0;
  const cudaError_t e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, q_positions, q_bf16, modes,
                                         nullptr, windows, window_scalar, softmax_scale, out_bf16,
                                         static_cast<cudaStream_t>(stream), &launches, false);
  cache_set_launches(cache, launches);
  return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}

extern "C" trr_status trr_decode_step(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                      const int32_t* positions, const void* k_bf16, const void* v_bf16,
                                      const uint8_t* bits, const uint8_t* modes, const void* q_bf16,
                                      const int32_t* windows, int32_t window_scalar, float softmax_scale,
                                      void* out_bf16, void* stream) {
  if (!cache) return TRR_ERR_INVALID_ARG;
  const Layout& l = cache_layout(cache);
  if (layer < 0 || layer >= l.L || n < 0 || n > l.max_queries || n > l.max_append || n > kStepMax)
    return TRR_ERR_INVALID_ARG;
  cache_set_launches(cache, 0);
  if (n == 0) return TRR_OK;
  if (!seq_ids || !positions || !k_bf16 || !v_bf16 || !bits || !modes || !q_bf16 || !out_bf16)
    return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(q_bf16) | reinterpret_cast<uintptr_t>(out_bf16) |
       reinterpret_cast<uintptr_t>(k_bf16) | reinterpret_cast<uintptr_t>(v_bf16)) & 15)
    return TRR_ERR_INVALID_ARG;
  if (l.head_modes) return TRR_ERR_UNSUPPORTED;  // one mode per token
  LayerArgs a = layer_args(l, cache_views(cache), layer);
  a.wait_ns = cache_wait_ns(cache);
  const bool early = cache_layer_settled(cache, layer);
  cache_note_call(cache, layer);
  const StepInputs step{k_bf16, v_bf16, bits};
  int launches = 0;
  const cudaError_t e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, positions, q_bf16, modes, nullptr,
                                         windows, window_scalar, softmax_scale, out_bf16,
                                         static_cast<cudaStream_t>(stream), &launches, early, &step);
  cache_set_launches(cache, launches);
  return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}

extern "C" trr_status trr_decode_attn_routed(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                             const int32_t* q_positions, const void* q_bf16, const float* mode_logits,
                                             const int32_t* windows, int32_t window_scalar, float softmax_scale,
                                             void* out_bf16, void* stream) {
  if (!cache) return TRR_ERR_INVALID_ARG;
  const Layout& l = cache_layout(cache);
  if (layer < 0 || layer >= l.L || n < 0 || n > l.max_queries) return TRR_ERR_INVALID_ARG;
  cache_set_launches(cache, 0);
  if (n == 0) return TRR_OK;
  if (!seq_ids || !q_positions || !q_bf16 || !mode_logits || !out_bf16) return TRR_ERR_INVALID_ARG;
  if (((reinterpret_cast<uintptr_t>(q_bf16) | reinterpret_cast<uintptr_t>(out_bf16)) & 15) ||
      (reinterpret_cast<uintptr_t>(mode_logits) & 3))
    return TRR_ERR_INVALID_ARG;
  if (l.head_modes) return TRR_ERR_UNSUPPORTED;  // router decisions are per token
  LayerArgs a = layer_args(l, cache_views(cache), layer);
  a.wait_ns = cache_wait_ns(cache);
  cache_note_call(cache, layer);
  int launches = 0;
  const cudaError_t e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, q_positions, q_bf16, nullptr,
                                         mode_logits, windows, window_scalar, softmax_scale, out_bf16,
                                         static_cast<cudaStream_t>(stream), &launches, false);
  cache_set_launches(cache, launches);
  return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}

// ------------------------------------------------------ static-scratch variant --
//
// trr_decode_attn_static runs the same kernel as trr_decode_attn, but keeps all of its
// per-call scratch (arrival counters, fp32 partials and the call's control words) in one
// file-scope device array instead of the cache's scratch region.  Nothing is allocated
// per call or at set-up.
namespace trr {

constexpr int64_t kStaticScratchBytes = 32ll << 20;  // 32 MiB on every device using the library
static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
static void* g_static_ptr[kMaxDevices];  // device address of g_static_scratch, per device

// Address of the array on the current device, looked up once per device.
static cudaError_t static_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (!g_static_ptr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_static_scratch);
    if (e != cudaSuccess) return e;
    g_static_ptr[dev] = ptr;
  }
  *out = g_static_ptr[dev];
  return cudaSuccess;
}

// The call's attention control words sit at this offset among its control words.
constexpr int kStaticLayerCtrl = 32;

// Clears what a call needs at zero: the control words and the arrival counters.
__global__ void static_scratch_clear_kernel(int32_t* wctrl, int32_t* cnt, int ncnt) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < kCtrlInts) wctrl[i] = i == kStaticLayerCtrl + kFirstBadQuery ? INT_MAX : 0;
  for (int j = i; j < ncnt; j += gridDim.x * blockDim.x) cnt[j] = 0;
}

// Forwards the call's first error to the cache's sticky status word.
__global__ void static_scratch_status_kernel(const int32_t* wctrl, int32_t* ctrl) {
  const int st = wctrl[kStatus];
  if (st != 0) atomicCAS(ctrl + kStatus, 0, st);
}

}  // namespace trr

extern "C" trr_status trr_decode_attn_static(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                             const int32_t* q_positions, const void* q_bf16, const uint8_t* modes,
                                             const int32_t* windows, int32_t window_scalar, float softmax_scale,
                                             void* out_bf16, void* stream) {
  if (!cache) return TRR_ERR_INVALID_ARG;
  const Layout& l = cache_layout(cache);
  if (layer < 0 || layer >= l.L || n < 0) return TRR_ERR_INVALID_ARG;
  cache_set_launches(cache, 0);
  if (n == 0) return TRR_OK;
  if (!seq_ids || !q_positions || !q_bf16 || !modes || !out_bf16) return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(q_bf16) | reinterpret_cast<uintptr_t>(out_bf16)) & 15)
    return TRR_ERR_INVALID_ARG;
  // scratch of this call, carved from the static array; reject what does not fit
  auto up = [](int64_t x) { return (x + 255) / 256 * 256; };
  const int64_t b_ctrl = up(4 * kCtrlInts);
  const int64_t b_cnt = up(4ll * n * l.units * l.cnt_stride);
  const int64_t b_part = up(4ll * n * l.s_cap * l.units * (l.d + 4));
  if (b_ctrl + b_cnt + b_part > kStaticScratchBytes) return TRR_ERR_OUT_OF_MEMORY;
  void* base = nullptr;
  if (static_scratch(&base) != cudaSuccess) return TRR_ERR_CUDA;
  uint8_t* b = static_cast<uint8_t*>(base);
  LayerArgs a = layer_args(l, cache_views(cache), layer);
  a.wait_ns = cache_wait_ns(cache);
  int32_t* cache_ctrl = a.ctrl;
  a.ctrl = reinterpret_cast<int32_t*>(b);
  a.lctl = a.ctrl + kStaticLayerCtrl;
  a.cnt = reinterpret_cast<int32_t*>(b + b_ctrl);
  a.part = reinterpret_cast<float*>(b + b_ctrl + b_cnt);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int ncnt = n * l.units * l.cnt_stride;
  static_scratch_clear_kernel<<<std::max(1, std::min(256, (ncnt + 255) / 256)), 256, 0, s>>>(a.ctrl, a.cnt, ncnt);
  cudaError_t e = cudaGetLastError();
  int launches = 0;
  if (e == cudaSuccess)
    e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, q_positions, q_bf16, modes, nullptr, windows,
                         window_scalar, softmax_scale, out_bf16, s, &launches, false);
  cache_note_call(cache, layer);
  if (e != cudaSuccess) return TRR_ERR_CUDA;
  static_scratch_status_kernel<<<1, 1, 0, s>>>(a.ctrl, cache_ctrl);
  cache_set_launches(cache, launches + 2);
  return cudaGetLastError() == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}
