// trr_route.cu - trr_route_decisions: the router's hard decisions at inference
// (Sec. 3.8: arg max of the mode and width logits) and what they cost under the model
// of Sec. 3.5 (Appendix C's expected_cost at a one-hot policy).
//
// One thread per group of 4 tokens (16-byte loads and stores where the arrays allow);
// a CTA adds its partial sums to the caller's totals with four 64-bit atomics.  The
// kernel streams 32 bytes of input and writes 18 bytes per token.
#include <algorithm>

#include "trr_internal.cuh"

namespace trr {

constexpr int kRouteThreads = 256;

struct RouteArgs {
  int n;
  const float* mode_logits;  // [n][3]
  const float* bit_logits;   // [n][4]
  const int32_t* positions;  // [n], or null when no cost is asked for
  int window, Hq, d, Hkv, skip_writes_kv;
  uint8_t* modes;            // outputs, each may be null
  uint8_t* bits;
  int64_t* attn_flops;
  int64_t* kv_bits;
  unsigned long long* totals;  // [4], added to
};

// Decisions and cost of token e; adds to the thread's sums.
__device__ __forceinline__ void route_token(const RouteArgs& r, const float* zm, const float* zb, int p, int& m,
                                            int& b, long long& flops, long long& mem, long long* sum) {
  m = hard_decision<3>(zm);
  b = 2 << hard_decision<4>(zb);
  // key positions read: full p + 1, local min(p + 1, w), skip 0 (p < 0 charged as 0)
  const long long t = static_cast<long long>(max(p, 0)) + 1;
  const long long keys = m == TRR_MODE_FULL ? t : m == TRR_MODE_LOCAL ? min(t, static_cast<long long>(r.window)) : 0;
  const long long per_key = 2ll * r.Hq * r.d, per_bit = 2ll * r.Hkv * r.d;
  flops = per_key * keys;
  mem = (m == TRR_MODE_SKIP && !r.skip_writes_kv) ? 0 : per_bit * b;
  sum[0] += flops;
  sum[1] += mem;
  sum[2] += per_key * t;
  sum[3] += per_bit * 16;
}

// One thread per group of 4 tokens.  VEC: every array is aligned for 16-byte loads of
// a group's logits (48 + 64 bytes) and positions and for 4-byte / 16-byte stores of its
// decisions and costs; a partial last group and the unaligned case go token by token.
template <bool VEC>
__global__ void __launch_bounds__(kRouteThreads) route_kernel(RouteArgs r) {
  __shared__ long long s_sum[kRouteThreads / 32][4];
  // The logits may come from the kernel just before this one: wait for it first.
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool cost = r.positions != nullptr;
  long long sum[4] = {0, 0, 0, 0};
  const int groups = (r.n + 3) >> 2;
  for (int g = blockIdx.x * kRouteThreads + threadIdx.x; g < groups; g += gridDim.x * kRouteThreads) {
    const int e0 = g << 2;
    if (VEC && e0 + 4 <= r.n) {
      float zm[12], zb[16];
      const float4* m4 = reinterpret_cast<const float4*>(r.mode_logits) + 3 * static_cast<int64_t>(g);
      const float4* b4 = reinterpret_cast<const float4*>(r.bit_logits) + 4 * static_cast<int64_t>(g);
#pragma unroll
      for (int i = 0; i < 3; ++i) reinterpret_cast<float4*>(zm)[i] = __ldcs(m4 + i);
#pragma unroll
      for (int i = 0; i < 4; ++i) reinterpret_cast<float4*>(zb)[i] = __ldcs(b4 + i);
      int p[4] = {0, 0, 0, 0};
      if (cost) {
        const int4 pv = __ldcs(reinterpret_cast<const int4*>(r.positions) + g);
        p[0] = pv.x; p[1] = pv.y; p[2] = pv.z; p[3] = pv.w;
      }
      uint32_t mw = 0, bw = 0;
      long long fl[4], mb[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        int m, b;
        route_token(r, zm + 3 * i, zb + 4 * i, p[i], m, b, fl[i], mb[i], sum);
        mw |= static_cast<uint32_t>(m) << (8 * i);
        bw |= static_cast<uint32_t>(b) << (8 * i);
      }
      if (r.modes) __stcs(reinterpret_cast<unsigned int*>(r.modes) + g, mw);
      if (r.bits) __stcs(reinterpret_cast<unsigned int*>(r.bits) + g, bw);
      if (r.attn_flops) {
        longlong2* o = reinterpret_cast<longlong2*>(r.attn_flops) + 2 * static_cast<int64_t>(g);
        __stcs(o, make_longlong2(fl[0], fl[1]));
        __stcs(o + 1, make_longlong2(fl[2], fl[3]));
      }
      if (r.kv_bits) {
        longlong2* o = reinterpret_cast<longlong2*>(r.kv_bits) + 2 * static_cast<int64_t>(g);
        __stcs(o, make_longlong2(mb[0], mb[1]));
        __stcs(o + 1, make_longlong2(mb[2], mb[3]));
      }
    } else {
      for (int e = e0; e < min(e0 + 4, r.n); ++e) {
        int m, b;
        long long fl, mb;
        route_token(r, r.mode_logits + 3 * static_cast<int64_t>(e), r.bit_logits + 4 * static_cast<int64_t>(e),
                    cost ? r.positions[e] : 0, m, b, fl, mb, sum);
        if (r.modes) r.modes[e] = static_cast<uint8_t>(m);
        if (r.bits) r.bits[e] = static_cast<uint8_t>(b);
        if (r.attn_flops) r.attn_flops[e] = fl;
        if (r.kv_bits) r.kv_bits[e] = mb;
      }
    }
  }
  if (!r.totals || !cost) return;
#pragma unroll
  for (int k = 0; k < 4; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum[k] += __shfl_xor_sync(0xffffffffu, sum[k], o);
  if (lane == 0)
#pragma unroll
    for (int k = 0; k < 4; ++k) s_sum[warp][k] = sum[k];
  __syncthreads();
  if (threadIdx.x < 4) {
    long long v = 0;
    for (int w = 0; w < kRouteThreads / 32; ++w) v += s_sum[w][threadIdx.x];
    if (v) atomicAdd(r.totals + threadIdx.x, static_cast<unsigned long long>(v));
  }
}

}  // namespace trr

using namespace trr;

extern "C" trr_status trr_route_decisions(int32_t n, const float* mode_logits, const float* bit_logits,
                                          const int32_t* positions, int32_t window, int32_t num_q_heads,
                                          int32_t head_dim, int32_t num_kv_heads, int32_t skip_writes_kv,
                                          uint8_t* modes, uint8_t* bits, int64_t* attn_flops, int64_t* kv_bits,
                                          int64_t* totals, void* stream) {
  if (n < 0) return TRR_ERR_INVALID_ARG;
  if (n == 0) return TRR_OK;
  if (!mode_logits || !bit_logits) return TRR_ERR_INVALID_ARG;
  const bool cost = attn_flops || kv_bits || totals;
  if (cost && (!positions || window < 1 || num_q_heads < 1 || head_dim < 1 || num_kv_heads < 1))
    return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(mode_logits) | reinterpret_cast<uintptr_t>(bit_logits) |
       reinterpret_cast<uintptr_t>(positions)) & 3)
    return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(attn_flops) | reinterpret_cast<uintptr_t>(kv_bits) |
       reinterpret_cast<uintptr_t>(totals)) & 7)
    return TRR_ERR_INVALID_ARG;
  RouteArgs r;
  r.n = n;
  r.mode_logits = mode_logits;
  r.bit_logits = bit_logits;
  r.positions = cost ? positions : nullptr;
  r.window = window;
  r.Hq = num_q_heads;
  r.d = head_dim;
  r.Hkv = num_kv_heads;
  r.skip_writes_kv = skip_writes_kv ? 1 : 0;
  r.modes = modes;
  r.bits = bits;
  r.attn_flops = attn_flops;
  r.kv_bits = kv_bits;
  r.totals = reinterpret_cast<unsigned long long*>(totals);
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const auto al = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
  const bool vec = al(mode_logits, 16) && al(bit_logits, 16) && al(r.positions, 16) && al(modes, 4) &&
                   al(bits, 4) && al(attn_flops, 16) && al(kv_bits, 16);
  const int64_t want = (static_cast<int64_t>(n) + 4ll * kRouteThreads - 1) / (4ll * kRouteThreads);
  const unsigned grid = static_cast<unsigned>(std::max<int64_t>(1, std::min<int64_t>(want, 8ll * sms)));
  const cudaError_t e =
      vec ? launch_pdl(route_kernel<true>, dim3(grid), dim3(kRouteThreads), 0, static_cast<cudaStream_t>(stream), r)
          : launch_pdl(route_kernel<false>, dim3(grid), dim3(kRouteThreads), 0, static_cast<cudaStream_t>(stream), r);
  return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}
