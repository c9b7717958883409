// trr_cache.cu - cache creation, layout, status and inspection entry points.
//
// The cache is one block of device memory: control words, per-(layer, sequence)
// metadata, scratch for the two hot-path calls, then one page pool per width class
// (Sec. 7: tokens grouped by precision, one bit-width class per page).
#include <algorithm>
#include <climits>
#include <cstdlib>
#include <cstring>
#include <new>

#include "trr_internal.cuh"

namespace trr {

LayerArgs layer_args(const Layout& l, const Views& v, int layer) {
  LayerArgs a;
  a.layer = layer;
  a.S = l.S; a.Hq = l.Hq; a.Hkv = l.Hkv; a.d = l.d; a.G = l.G; a.P = l.P;
  a.maxctx = l.maxctx; a.MP = l.MP; a.W32 = l.W32; a.units = l.units; a.pos_split = l.pos_split;
  a.s_cap = l.s_cap;
  a.split_bytes = l.split_bytes; a.skip_writes_kv = l.skip_writes_kv;
  a.head_modes = l.head_modes; a.maskb = static_cast<int>(l.maskb); a.swz = l.swz;
  a.hdr = static_cast<int>(l.hdr);
  for (int c = 0; c < kClasses; ++c) {
    a.cap[c] = l.cap[c];
    a.slice[c] = static_cast<int>(l.slice[c]);
    a.page_bytes[c] = l.page_bytes[c];
    a.pool[c] = v.pool[c];
  }
  const int64_t ls = static_cast<int64_t>(layer) * l.S;
  a.wait_ns = kDefaultWaitNs;
  a.ctrl = v.ctrl;
  a.lctl = v.lctl + static_cast<int64_t>(layer) * kLayerCtrlInts;
  a.last_pos = v.last_pos + ls;
  a.ntok = v.ntok + ls * 4;
  a.presence = v.presence + ls * l.W32;
  a.pt = v.pt + ls * 4 * l.MP;
  a.pfirst = v.pfirst + ls * 4 * l.MP;
  a.plast = v.plast + ls * 4 * l.MP;
  a.lastpg = v.lastpg + ls * 4;
  a.aplan = v.aplan;
  a.cnt = v.cnt;
  a.cnt_stride = l.cnt_stride;
  a.part = v.part;
  return a;
}

static int64_t roundup(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// Validates the configuration and fills every size and offset.
static trr_status make_layout(const trr_cache_config* c, Layout* l) {
  if (!c || !l) return TRR_ERR_INVALID_ARG;
  if (c->num_layers < 1 || c->max_seqs < 1 || c->num_kv_heads < 1 || c->num_q_heads < 1 ||
      c->max_context < 1 || c->max_append < 1 || c->max_queries < 1 || c->split_bytes < 0)
    return TRR_ERR_INVALID_ARG;
  if (c->num_q_heads % c->num_kv_heads) return TRR_ERR_UNSUPPORTED;
  if (c->head_dim != 64 && c->head_dim != 128) return TRR_ERR_UNSUPPORTED;
  if ((c->group_size != 32 && c->group_size != 64 && c->group_size != 128) ||
      c->group_size > c->head_dim)
    return TRR_ERR_UNSUPPORTED;
  if (c->page_size != 16 && c->page_size != 32 && c->page_size != 64) return TRR_ERR_UNSUPPORTED;
  if (c->max_append > 1024 || c->max_queries > 4096 || c->skip_writes_kv < 0 ||
      c->skip_writes_kv > 1 || c->head_modes < 0 || c->head_modes > 1 || c->max_context > (1 << 24) ||
      c->max_seqs > (1 << 20))
    return TRR_ERR_UNSUPPORTED;
  for (int k = 0; k < kClasses; ++k)
    if (c->pages_per_class[k] < 0) return TRR_ERR_INVALID_ARG;

  l->L = c->num_layers; l->S = c->max_seqs; l->Hq = c->num_q_heads; l->Hkv = c->num_kv_heads;
  l->d = c->head_dim; l->G = c->group_size; l->P = c->page_size; l->maxctx = c->max_context;
  l->MP = (l->maxctx + l->P - 1) / l->P;
  l->W32 = (l->maxctx + 31) / 32;
  for (int k = 0; k < kClasses; ++k) l->cap[k] = c->pages_per_class[k];
  l->max_append = c->max_append;
  l->max_queries = c->max_queries;
  l->split_bytes = c->split_bytes ? c->split_bytes : 24576;
  l->skip_writes_kv = c->skip_writes_kv;
  l->head_modes = c->head_modes;
  l->swz = uses_mma(l->Hq, l->Hkv, l->d, l->G, l->head_modes) ? 0 : 1;
  l->hdr = roundup(4 * static_cast<int64_t>(l->P), 128);
  // per-head modes: each KV head's slice of a page ends with 16 bytes holding its 64-bit
  // presence mask, so that the copy of a slice brings its mask
  l->maskb = l->head_modes ? 16 : 0;
  for (int k = 0; k < kClasses; ++k) {
    const int b = bits_of_class(k);
    l->tokb[k] = b < 16 ? 2 * (l->d * b / 8) + 2 * (l->d / l->G) * 4 : 4 * l->d;
    l->slice[k] = l->P * l->tokb[k] + l->maskb;
    l->page_bytes[k] = roundup(l->hdr + l->Hkv * l->slice[k], 128);
  }
  l->units = l->Hq;
  // splits per query: at least pos_split key positions each (split_bytes of 8-bit
  // tokens), and few enough pages per split for any range up to max_context
  l->pos_split = static_cast<int>(std::max<int64_t>(l->P, l->split_bytes / l->tokb[2]));
  l->s_cap = 1 << 30;
  l->s_cap = std::max(splits_of(l->maxctx, l->pos_split, l->P, l->s_cap), 1);
  l->cnt_stride = 1 + (l->s_cap + kMergeGroup - 1) / kMergeGroup;
  l->max_items = static_cast<int64_t>(l->max_queries) * l->units * l->s_cap;

  const int64_t nls = static_cast<int64_t>(l->L) * l->S;
  int64_t off = 0;
  auto take = [&](int64_t bytes) {
    const int64_t o = off;
    off = roundup(off + bytes, 256);
    return o;
  };
  l->off_ctrl = take(4 * kCtrlInts);
  l->off_lctl = take(4 * static_cast<int64_t>(kLayerCtrlInts) * l->L);
  l->off_last_pos = take(4 * nls);
  l->off_ntok = take(16 * nls);
  l->off_presence = take(4 * nls * l->W32);
  l->off_pt = take(16 * nls * l->MP);
  l->off_pfirst = take(16 * nls * l->MP);
  l->off_plast = take(16 * nls * l->MP);
  l->off_lastpg = take(16 * nls);
  l->off_aplan = take(static_cast<int64_t>(sizeof(AppendPlan)) * l->max_append);
  l->off_cnt = take(4 * static_cast<int64_t>(l->max_queries) * l->units * l->cnt_stride);
  l->off_part = take(4 * l->max_items * (l->Hq / l->units) * (l->d + 4));
  for (int k = 0; k < kClasses; ++k) l->off_pool[k] = take(l->cap[k] * l->page_bytes[k]);
  l->total = off;
  return TRR_OK;
}

}  // namespace trr

struct trr_cache {
  trr::Layout lay;
  trr::Views views;
  void* base;
  bool owned;
  int device;
  int num_sms;
  int last_launches;
  int recent[2];  // layers of the last two calls enqueued (-1: none; -2: every layer)
  uint64_t wait_ns;  // bound of an in-kernel wait
};

using namespace trr;

extern "C" trr_status trr_cache_required_bytes(const trr_cache_config* cfg, uint64_t* bytes) {
  if (!bytes) return TRR_ERR_INVALID_ARG;
  Layout l;
  trr_status st = make_layout(cfg, &l);
  if (st != TRR_OK) return st;
  *bytes = static_cast<uint64_t>(l.total);
  return TRR_OK;
}

__global__ void init_ctrl_kernel(int32_t* ctrl, int32_t* lctl, int nl) {
  if (ctrl && threadIdx.x < kCtrlInts) ctrl[threadIdx.x] = 0;
  for (int i = threadIdx.x; i < nl * kLayerCtrlInts; i += blockDim.x)
    lctl[i] = i % kLayerCtrlInts == kFirstBadQuery ? INT_MAX : 0;
}

// Metadata to its empty state, stream-ordered.
static trr_status clear_metadata(trr_cache* c, cudaStream_t s) {
  const Layout& l = c->lay;
  uint8_t* b = static_cast<uint8_t*>(c->base);
  const int64_t nls = static_cast<int64_t>(l.L) * l.S;
  init_ctrl_kernel<<<1, 256, 0, s>>>(reinterpret_cast<int32_t*>(b + l.off_ctrl),
                                     reinterpret_cast<int32_t*>(b + l.off_lctl), l.L);
  c->recent[0] = c->recent[1] = -2;  // state changed by something other than a layer's call
  bool ok = cudaGetLastError() == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_last_pos, 0xFF, 4 * nls, s) == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_ntok, 0, 16 * nls, s) == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_presence, 0, 4 * nls * l.W32, s) == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_pt, 0xFF, 3 * (l.off_pfirst - l.off_pt), s) == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_lastpg, 0xFF, 16 * nls, s) == cudaSuccess;
  ok = ok && cudaMemsetAsync(b + l.off_cnt, 0, 4 * static_cast<int64_t>(l.max_queries) * l.units * l.cnt_stride, s) ==
                  cudaSuccess;
  return ok ? TRR_OK : TRR_ERR_CUDA;
}

extern "C" trr_status trr_create_cache(const trr_cache_config* cfg, trr_cache** out) {
  if (!cfg || !out) return TRR_ERR_INVALID_ARG;
  *out = nullptr;
  Layout l;
  trr_status st = make_layout(cfg, &l);
  if (st != TRR_OK) return st;
  trr_cache* c = new (std::nothrow) trr_cache();
  if (!c) return TRR_ERR_OUT_OF_MEMORY;
  c->lay = l;
  if (cudaGetDevice(&c->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess) {
    delete c;
    return TRR_ERR_CUDA;
  }
  if (cfg->pool) {
    if (cfg->pool_bytes < static_cast<uint64_t>(l.total) ||
        (reinterpret_cast<uintptr_t>(cfg->pool) & 255)) {
      delete c;
      return TRR_ERR_OUT_OF_MEMORY;
    }
    c->base = cfg->pool;
    c->owned = false;
  } else {
    if (cudaMalloc(&c->base, l.total) != cudaSuccess) {
      cudaGetLastError();
      delete c;
      return TRR_ERR_OUT_OF_MEMORY;
    }
    c->owned = true;
  }
  if (attn_configure() != cudaSuccess) {
    if (c->owned) cudaFree(c->base);
    delete c;
    return TRR_ERR_CUDA;
  }
  c->views = make_views(l, c->base);
  c->last_launches = 0;
  c->wait_ns = kDefaultWaitNs;
  st = clear_metadata(c, nullptr);
  if (st == TRR_OK && cudaStreamSynchronize(nullptr) != cudaSuccess) st = TRR_ERR_CUDA;
  c->recent[0] = c->recent[1] = -1;  // the cleared state is complete on the device
  if (st != TRR_OK) {
    if (c->owned) cudaFree(c->base);
    delete c;
    return st;
  }
  *out = c;
  return TRR_OK;
}

extern "C" trr_status trr_destroy(trr_cache* c) {
  if (!c) return TRR_OK;
  trr_status st = TRR_OK;
  if (cudaDeviceSynchronize() != cudaSuccess) st = TRR_ERR_CUDA;
  if (c->owned && cudaFree(c->base) != cudaSuccess) st = TRR_ERR_CUDA;
  delete c;
  return st;
}

__global__ void take_status_kernel(int32_t* ctrl, int32_t* out) {
  *out = atomicExch(ctrl + kStatus, 0);
}

extern "C" trr_status trr_get_status(trr_cache* c, void* stream) {
  if (!c) return TRR_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the taken value lands in the last control word, then comes back to the host
  int32_t* slot = c->views.ctrl + kCtrlInts - 1;
  take_status_kernel<<<1, 1, 0, s>>>(c->views.ctrl, slot);
  int32_t v = 0;
  if (cudaGetLastError() != cudaSuccess ||
      cudaMemcpyAsync(&v, slot, 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return TRR_ERR_CUDA;
  if (v == TRR_ERR_TIMEOUT) {
    // a call gave up a wait and may have left split counters and the layers' work
    // counters mid-count: back to their start values, so that the cache serves again
    const Layout& l = c->lay;
    uint8_t* b = static_cast<uint8_t*>(c->base);
    init_ctrl_kernel<<<1, 256, 0, s>>>(nullptr, reinterpret_cast<int32_t*>(b + l.off_lctl), l.L);
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemsetAsync(b + l.off_cnt, 0, 4 * static_cast<int64_t>(l.max_queries) * l.units * l.cnt_stride, s) !=
            cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return TRR_ERR_CUDA;
    c->recent[0] = c->recent[1] = -2;
  }
  return static_cast<trr_status>(v);
}

extern "C" trr_status trr_set_wait_limit(trr_cache* c, uint64_t nanoseconds) {
  if (!c) return TRR_ERR_INVALID_ARG;
  c->wait_ns = nanoseconds ? nanoseconds : kDefaultWaitNs;
  return TRR_OK;
}

extern "C" trr_status trr_reset(trr_cache* c, void* stream) {
  if (!c) return TRR_ERR_INVALID_ARG;
  return clear_metadata(c, static_cast<cudaStream_t>(stream));
}

extern "C" trr_status trr_get_region(const trr_cache* c, int32_t region, void** ptr, uint64_t* bytes) {
  if (!c || !ptr || !bytes) return TRR_ERR_INVALID_ARG;
  const Layout& l = c->lay;
  uint8_t* b = static_cast<uint8_t*>(c->base);
  const int64_t nls = static_cast<int64_t>(l.L) * l.S;
  switch (region) {
    case 0: *ptr = b + l.off_last_pos; *bytes = 4 * nls; break;
    case 1: *ptr = b + l.off_ntok; *bytes = 16 * nls; break;
    case 2: *ptr = b + l.off_presence; *bytes = 4 * nls * l.W32; break;
    case 3: *ptr = b + l.off_pt; *bytes = 16 * nls * l.MP; break;
    case 4: *ptr = b + l.off_pfirst; *bytes = 16 * nls * l.MP; break;
    case 5: *ptr = b + l.off_plast; *bytes = 16 * nls * l.MP; break;
    case 6: *ptr = b + l.off_ctrl + 4 * kNextPage; *bytes = 16; break;
    case 7: case 8: case 9: case 10:
      *ptr = b + l.off_pool[region - 7];
      *bytes = static_cast<uint64_t>(l.cap[region - 7]) * l.page_bytes[region - 7];
      break;
    default: return TRR_ERR_INVALID_ARG;
  }
  return TRR_OK;
}

extern "C" int32_t trr_last_launch_count(const trr_cache* c) { return c ? c->last_launches : 0; }

// Accessors used by the other translation units.
namespace trr {
const Layout& cache_layout(const trr_cache* c) { return c->lay; }
const Views& cache_views(const trr_cache* c) { return c->views; }
int cache_num_sms(const trr_cache* c) { return c->num_sms; }
void cache_set_launches(trr_cache* c, int n) { c->last_launches = n; }
bool cache_layer_settled(const trr_cache* c, int layer) {
  return c->recent[0] != -2 && c->recent[1] != -2 && c->recent[0] != layer && c->recent[1] != layer;
}
uint64_t cache_wait_ns(const trr_cache* c) { return c->wait_ns; }
void cache_note_call(trr_cache* c, int layer) {
  c->recent[1] = c->recent[0];
  c->recent[0] = layer;
}
}  // namespace trr
