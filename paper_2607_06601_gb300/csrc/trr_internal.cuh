// trr_internal.cuh - layout arithmetic, kernel argument blocks and PTX helpers shared
// by the library's translation units (trr_cache.cu, trr_append.cu, trr_attn.cu).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/trr.h"

namespace trr {

constexpr int kClasses = 4;
__host__ __device__ constexpr int bits_of_class(int c) { return c == 0 ? 2 : c == 1 ? 4 : c == 2 ? 8 : 16; }

// Control words (int32) at the start of the cache memory.
enum Ctrl : int {
  kStatus = 0,        // sticky first error since the last trr_get_status
  kNextPage = 4,      // [4] pages handed out per class
  kAppendOk = 10,     // append: 1 when the plan kernel committed the call
  kAppendDone = 11,   // one-kernel append: CTAs finished (the last one commits)
  kCtrlInts = 64
};

// Control words of the attention kernels, one set per layer (an attention or decode-step
// kernel of one layer may start while the previous layer's kernel still runs).
enum LayerCtrl : int {
  kNextUnit = 0,      // next work unit to hand out
  kDoneCtas = 1,      // CTAs finished (the last one records the status)
  kFirstBadQuery = 2, // min of (query index * 16 + error) over failing queries (INT_MAX = none)
  kAborted = 3,       // 1 when a CTA gave up a wait (a decode step then commits nothing)
  kLayerCtrlInts = 4
};

// Splits of one attention work unit are sized to hold at most this many pages (+ one
// partial page per class), so that a warp holds an item's page ids one per lane.
constexpr int kItemMaxPages = 28;

// Split partials are merged in groups of this many (then the groups): a query with
// ns splits per head has 1 + ceil(ns / kMergeGroup) arrival counters per head.
constexpr int kMergeGroup = 16;

// Byte layout of one cache (see include/trr.h for the documented part).
struct Layout {
  int L, S, Hq, Hkv, d, G, P, maxctx, MP, W32;
  int cap[kClasses];
  int max_append, max_queries, split_bytes, skip_writes_kv, head_modes;
  int swz;        // 8- and 16-bit code rows stored swizzled (caches of the CUDA-core consumer)
  int units;      // attention work units per query split (one per query head)
  int pos_split;  // key positions per split at least (split_bytes of 8-bit tokens)
  int s_cap;      // most splits one query is cut into
  int cnt_stride; // arrival counters per (query, head): 1 + ceil(s_cap / kMergeGroup)
  int64_t max_items;
  int64_t hdr, tokb[kClasses], slice[kClasses], maskb, page_bytes[kClasses];
  int64_t off_ctrl, off_lctl, off_last_pos, off_ntok, off_presence, off_pt, off_pfirst, off_plast, off_lastpg;
  int64_t off_aplan, off_cnt, off_part, off_pool[kClasses], total;
};

// Splits of a query whose key range spans `range` positions: at least pos_split
// positions each, enough that no split holds more than kItemMaxPages + 4 pages, at most
// s_cap (which covers the page bound for any range up to max_context).
__host__ __device__ inline int splits_of(int range, int pos_split, int P, int s_cap) {
  if (range <= 0) return 1;
  const int by_len = (range + pos_split - 1) / pos_split;
  const int by_pages = ((range + P - 1) / P + 2 * kClasses + kItemMaxPages - 1) / kItemMaxPages;
  const int ns = by_len > by_pages ? by_len : by_pages;
  return ns < s_cap ? ns : s_cap;
}

// The tensor-core consumer serves query groups (g >= 2) whose (head, group) columns fit
// one 8-wide mma tile, without per-head modes; every other cache is read by the
// CUDA-core consumer, whose lanes read 8- and 16-bit code rows in a pattern that the
// swizzle below makes free of shared-memory bank conflicts.
__host__ __device__ inline bool uses_mma(int Hq, int Hkv, int d, int G, int head_modes) {
  const int g = Hq / Hkv, ng = d / G;
  return !head_modes && g >= 2 && g * ng <= 8;
}

// Where byte o of a KV slice's K or V code region (o counted from the slice's start)
// is stored in a swizzled cache, for 8- and 16-bit pages: each 128-byte line keeps its
// 16-byte chunks in the order chunk ^ (line % 8).  Both regions start on a line of the
// slice.  2- and 4-bit rows, scales, positions and masks are stored plainly.
__host__ __device__ inline int64_t swz_off(int64_t o) {
  return (o & ~static_cast<int64_t>(127)) | ((((o >> 4) ^ (o >> 7)) & 7) << 4) | (o & 15);
}

// Per-entry plan written by the append plan kernel.
struct AppendPlan {
  int page;   // page id, -1 = nothing stored
  int slot;   // slot in the page
  int cls;    // width class
  int pos;    // position
};

struct Views {  // typed device pointers into the cache memory
  int32_t* ctrl;
  int32_t* lctl;
  int32_t* last_pos;
  int32_t* ntok;
  uint32_t* presence;
  int32_t* pt;
  int32_t* pfirst;
  int32_t* plast;
  int32_t* lastpg;
  AppendPlan* aplan;
  int32_t* cnt;
  float* part;
  uint8_t* pool[kClasses];
};

inline Views make_views(const Layout& l, void* base) {
  uint8_t* b = static_cast<uint8_t*>(base);
  Views v;
  v.ctrl = reinterpret_cast<int32_t*>(b + l.off_ctrl);
  v.lctl = reinterpret_cast<int32_t*>(b + l.off_lctl);
  v.last_pos = reinterpret_cast<int32_t*>(b + l.off_last_pos);
  v.ntok = reinterpret_cast<int32_t*>(b + l.off_ntok);
  v.presence = reinterpret_cast<uint32_t*>(b + l.off_presence);
  v.pt = reinterpret_cast<int32_t*>(b + l.off_pt);
  v.pfirst = reinterpret_cast<int32_t*>(b + l.off_pfirst);
  v.plast = reinterpret_cast<int32_t*>(b + l.off_plast);
  v.lastpg = reinterpret_cast<int32_t*>(b + l.off_lastpg);
  v.aplan = reinterpret_cast<AppendPlan*>(b + l.off_aplan);
  v.cnt = reinterpret_cast<int32_t*>(b + l.off_cnt);
  v.part = reinterpret_cast<float*>(b + l.off_part);
  for (int c = 0; c < kClasses; ++c) v.pool[c] = b + l.off_pool[c];
  return v;
}

// Everything a kernel needs about one layer of one cache, passed by value.
struct LayerArgs {
  int layer, S, Hq, Hkv, d, G, P, maxctx, MP, W32, units, pos_split, s_cap, cnt_stride, split_bytes, skip_writes_kv;
  int head_modes;      // modes are [n][Hq]; each KV head's slice ends with its presence mask
  int swz;             // 8- and 16-bit code rows stored swizzled (see swz_off)
  uint64_t wait_ns;    // bound of an in-kernel wait before the kernel reports TRR_ERR_TIMEOUT
  int maskb;           // bytes that end a slice for its presence mask (16, or 0 without head_modes)
  int cap[kClasses];
  int hdr;
  int slice[kClasses];
  int64_t page_bytes[kClasses];
  int32_t* ctrl;
  int32_t* lctl;       // this layer's attention control words [kLayerCtrlInts]
  int32_t* last_pos;   // this layer: [S]
  int32_t* ntok;       // this layer: [S][4]
  uint32_t* presence;  // this layer: [S][W32]
  int32_t* pt;         // this layer: [S][4][MP]
  int32_t* pfirst;
  int32_t* plast;
  int32_t* lastpg;     // this layer: [S][4] id of the page holding token ntok-1 (internal)
  AppendPlan* aplan;
  int32_t* cnt;        // [max_queries][Hq][cnt_stride] split arrivals (zero between calls)
  float* part;         // [max_queries * s_cap * Hq][d + 4] fp32 partials: acc, M, L
  uint8_t* pool[kClasses];
};

LayerArgs layer_args(const Layout& l, const Views& v, int layer);

// Accessors of the opaque cache (defined in trr_cache.cu).
const Layout& cache_layout(const trr_cache* c);
const Views& cache_views(const trr_cache* c);
int cache_num_sms(const trr_cache* c);
void cache_set_launches(trr_cache* c, int n);
// Whether a kernel of a call on `layer` may read that layer's cache state before the
// previous kernel of the stream has finished: true when neither of the two calls
// enqueued before it on this cache touched the layer (with programmatic dependent
// launch, a kernel starts only once its predecessor has passed its own wait, so every
// kernel before that one has finished).  cache_note_call records a call.
bool cache_layer_settled(const trr_cache* c, int layer);
void cache_note_call(trr_cache* c, int layer);
uint64_t cache_wait_ns(const trr_cache* c);

// One-time kernel attribute setup (defined in trr_attn.cu).
cudaError_t attn_configure();

// ------------------------------------------------------------------ PTX helpers --

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

// 1-D bulk copy global -> shared (this CTA), completion counted on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// The global nanosecond timer.
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Default bound of an in-kernel wait (trr_set_wait_limit changes it per cache).
constexpr uint64_t kDefaultWaitNs = 2000000000ull;

// One try at phase `parity` of `bar`: parks the thread until the phase completes or
// about hint_ns pass (the hint is an upper bound: a try may return sooner), so that a
// waiting warp does not take issue slots.
__device__ __forceinline__ bool mbar_try(uint32_t addr, uint32_t parity, uint32_t hint_ns) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(addr), "r"(parity), "r"(hint_ns)
      : "memory");
  return done != 0;
}

// Whether phase `parity` has completed, without suspending.
__device__ __forceinline__ bool mbar_test_at(uint32_t addr, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(addr), "r"(parity)
      : "memory");
  return done != 0;
}

// One try of a wait bounded by limit_ns: a suspending try (a try may last until the
// phase completes), or, for a limit below the 20 us hint, a test that returns at once,
// so that a short limit is kept.
__device__ __forceinline__ bool mbar_poll(uint32_t addr, uint32_t parity, uint64_t limit_ns) {
  return limit_ns >= 20000 ? mbar_try(addr, parity, 20000u) : mbar_test_at(addr, parity);
}

// Bounded wait for phase `parity` of `bar`: returns false once limit_ns have passed
// (measured on the global timer) without the phase completing.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns = kDefaultWaitNs) {
  const uint32_t addr = smem_u32(bar);
  if (mbar_poll(addr, parity, limit_ns)) return true;
  const uint64_t t0 = global_ns();
  for (;;) {
    if (mbar_poll(addr, parity, limit_ns)) return true;
    if (global_ns() - t0 >= limit_ns) return false;
  }
}

// atomic add with release (of what this thread has seen written) and acquire (of what
// the threads that released the same counter wrote) at GPU scope
__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// The hard decision of one controller head (Sec. 3.8: at inference the router takes
// the arg max of its logits): the index of the largest of K logits, the first of equal
// ones; a NaN is never taken, and a row of NaN gives 0.
template <int K>
__device__ __forceinline__ int hard_decision(const float* z) {
  int best = 0;
  float top = z[0];
#pragma unroll
  for (int i = 1; i < K; ++i) {
    const float v = z[i];
    if (v > top || (top != top && v == v)) {
      top = v;
      best = i;
    }
  }
  return best;
}

// ---------------------------------------------------------------- quantiser --
// Eq. 4 of Sec. 3.2(C), shared by the append kernels and the decode-step kernel so that
// both store the same bytes.

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// round((x - z) / s) of Eq. 4 on the exact quotient, ties to even, clamped to [0, levels].
// u = fl32(fl32(x - z) * rs) with rs = fl32(1 / s) is within 3 binary32 roundings, under
// 2^-21 |u|, of the exact quotient, so rint(u) is exact unless u lies that close to a
// half-way point c + 1/2.  There the midpoint z + (c + 1/2) s is formed in binary64,
// where it is exact (z and s are binary16: a multiple of 2^-25 below 2^18), and compared
// with x (a bf16 value).  Only half-way points inside [0, levels] matter: the clamp
// settles the others.
__device__ __forceinline__ int code_of(float x, float z, float s, float rs, int levels) {
  const float u = __fmul_rn(__fsub_rn(x, z), rs);
  const float fl = floorf(u);
  if (fabsf(__fsub_rn(u, fl + 0.5f)) <= fabsf(u) * 0x1p-21f && fl >= 0.f && fl < static_cast<float>(levels)) {
    const double mid = __dadd_rn(static_cast<double>(z), __dmul_rn(static_cast<double>(fl) + 0.5, static_cast<double>(s)));
    const double xd = static_cast<double>(x);
    const int c = static_cast<int>(fl);
    return (xd > mid || (xd == mid && (c & 1))) ? c + 1 : c;
  }
  return min(max(__float2int_rn(u), 0), levels);
}

// One row of D values (a token's K or V for one KV head) quantised by a warp at b < 16
// bits: lane l holds values EPL*l .. EPL*l + EPL-1 (EPL = D/32) as bf16 in raw; a group's
// min / max by shuffles over its G/EPL lanes; codes packed LSB-first.  The lane writes
// code word `code_idx` (of the row's D*b/32 words) when code_idx >= 0 and the group's
// (s, z) word `sz_idx` when sz_idx >= 0.  A group holding a value binary16 cannot carry
// (non-finite or |x| > 65504) gets zero codes and a zero (s, z) word, and bad = true.
struct RowCodes {
  uint32_t code_word, sz_word;
  int code_idx, sz_idx;
  bool bad;
};
template <int D>
__device__ __forceinline__ RowCodes quantise_row_codes(const uint2 w, int b, int G, int lane) {
  constexpr int EPL = D / 32;
  float x[EPL];
  x[0] = bf16lo(w.x);
  x[1] = bf16hi(w.x);
  if (EPL == 4) {
    x[EPL > 2 ? 2 : 0] = bf16lo(w.y);
    x[EPL > 3 ? 3 : 1] = bf16hi(w.y);
  }
  const int lgl = __ffs(G) - 1 - (EPL == 4 ? 2 : 1), GL = 1 << lgl;  // lanes of one group (powers of two:
                                                                      // shifts and masks, no division)
  float mn = x[0], mx = x[0];
  bool bad = false;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    bad |= !(fabsf(x[i]) <= 65504.f);  // also true for NaN
    mn = fminf(mn, x[i]);
    mx = fmaxf(mx, x[i]);
  }
  for (int o = 1; o < GL; o <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    bad |= __shfl_xor_sync(0xffffffffu, static_cast<int>(bad), o) != 0;
  }
  const int levels = (1 << b) - 1;
  uint32_t val = 0, szw = 0;
  if (!bad) {
    const __half z16 = __float2half_rn(mn);                                                    // z = min(x)
    const __half s16 = __float2half_rn(__fdiv_rn(__fsub_rn(mx, mn), static_cast<float>(levels)));  // s
    const float z = __half2float(z16), s = __half2float(s16), rs = __frcp_rn(s);
#pragma unroll
    for (int i = 0; i < EPL; ++i)
      val |= static_cast<uint32_t>(s != 0.f ? code_of(x[i], z, s, rs, levels) : 0) << (i * b);
    szw = static_cast<uint32_t>(__half_as_ushort(s16)) | (static_cast<uint32_t>(__half_as_ushort(z16)) << 16);
  }
  const int lpw = 5 - (__ffs(EPL * b) - 1), LPW = 1 << lpw;  // lanes sharing one 32-bit word of codes
  val <<= (lane & (LPW - 1)) * EPL * b;
  for (int o = 1; o < LPW; o <<= 1) val |= __shfl_xor_sync(0xffffffffu, val, o);
  RowCodes r;
  r.code_word = val;
  r.sz_word = szw;
  r.code_idx = (lane & (LPW - 1)) == 0 ? lane >> lpw : -1;
  r.sz_idx = (lane & (GL - 1)) == 0 ? lane >> lgl : -1;
  r.bad = bad;
  return r;
}

__device__ __forceinline__ void set_status(int32_t* ctrl, int code) {
  atomicCAS(ctrl + kStatus, 0, code);
}

// Programmatic dependent launch: a kernel launched with launch_pdl may start while the
// previous kernel of the stream is still running; it must call pdl_wait() before it
// touches memory that kernel writes, and calls pdl_trigger() to let its own successor
// start early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... Args>
inline cudaError_t launch_pdl(void (*kern)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

}  // namespace trr
