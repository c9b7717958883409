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
  kFirstBadQuery = 12,// attention: min of (query index * 16 + error) over failing queries
                      // (INT_MAX = none)
  kDoneCtas = 14,     // attention: CTAs finished (the last one records the status)
  kNextUnit = 15,     // attention: next work unit to hand out
  kCtrlInts = 64
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
  int units;      // attention work units per query split (one per query head)
  int pos_split;  // key positions per split at least (split_bytes of 8-bit tokens)
  int s_cap;      // most splits one query is cut into
  int cnt_stride; // arrival counters per (query, head): 1 + ceil(s_cap / kMergeGroup)
  int64_t max_items;
  int64_t hdr, tokb[kClasses], slice[kClasses], maskb, page_bytes[kClasses];
  int64_t off_ctrl, off_last_pos, off_ntok, off_presence, off_pt, off_pfirst, off_plast, off_lastpg;
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

// Per-entry plan written by the append plan kernel.
struct AppendPlan {
  int page;   // page id, -1 = nothing stored
  int slot;   // slot in the page
  int cls;    // width class
  int pos;    // position
};

struct Views {  // typed device pointers into the cache memory
  int32_t* ctrl;
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
  int maskb;           // bytes that end a slice for its presence mask (16, or 0 without head_modes)
  int cap[kClasses];
  int hdr;
  int slice[kClasses];
  int64_t page_bytes[kClasses];
  int32_t* ctrl;
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

// Bounded wait for phase `parity` of `bar`: returns false when it gave up.  Each try
// parks the thread until the phase completes or about 20 us pass, so a waiting warp
// does not take issue slots; at most max_tries tries (about a second).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t max_tries = 50000) {
  uint32_t addr = smem_u32(bar);
  for (uint32_t i = 0; i < max_tries; ++i) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(addr), "r"(parity), "r"(20000)
        : "memory");
    if (done) return true;
  }
  return false;
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
