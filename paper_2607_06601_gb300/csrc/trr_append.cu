// trr_append.cu - trr_kv_append: quantise-on-write into the width-class page pools.
//
// Calls of up to 256 entries (decode steps) run as one kernel, append_fused_kernel
// (below); larger ones as two:
//   append_plan_kernel   one CTA, one thread per entry.  Validates every entry, ranks
//                        it among the earlier entries of its (sequence, class), hands
//                        out page ids in entry order, and commits the metadata only
//                        when the whole call is valid (Sec. 3.8: each token's KV is
//                        stored at its chosen width in a paged cache).
//   append_write_kernel  one thread per (entry, KV head, K|V, group): the quantiser
//                        Q_b of Sec. 3.2(C), Eq. 4, or a bf16 copy for b = 16.
#include <climits>

#include "trr_internal.cuh"

namespace trr {

__device__ __forceinline__ int class_of_bits(int b) {
  return b == 2 ? 0 : b == 4 ? 1 : b == 8 ? 2 : b == 16 ? 3 : -1;
}

// An entry's attention mode and bit-width: the caller's, or the hard decisions of its
// router logits (Sec. 3.8), taken here in the append's own planning step.  With
// per-head modes (modes[n][Hq]) the largest of the entry's head modes: skip only when
// every head skips, above full when any head's value is not a mode.
__device__ __forceinline__ int entry_mode(const LayerArgs& a, const uint8_t* modes, const float* mode_logits, int e) {
  if (mode_logits) return hard_decision<3>(mode_logits + 3 * e);
  if (!a.head_modes) return modes[e];
  int m = 0;
  const uint8_t* row = modes + static_cast<int64_t>(e) * a.Hq;
  for (int h = 0; h < a.Hq; ++h) m = max(m, static_cast<int>(row[h]));
  return m;
}

// Per-head modes: whether entry e stores KV head j, i.e. whether a query head reading it
// (h / (Hq / Hkv) == j) does not skip, or skip tokens store KV.
__device__ __forceinline__ bool head_stores(const LayerArgs& a, const uint8_t* modes, int e, int j) {
  if (a.skip_writes_kv) return true;
  const int g = a.Hq / a.Hkv;
  const uint8_t* row = modes + static_cast<int64_t>(e) * a.Hq + j * g;
  for (int h = 0; h < g; ++h)
    if (row[h] != TRR_MODE_SKIP) return true;
  return false;
}

// Per-head modes: KV head j's presence mask in a page, the first 8 of the 16 bytes that
// end its slice.
__device__ __forceinline__ unsigned long long* head_mask(const LayerArgs& a, int c, int pid, int j) {
  return reinterpret_cast<unsigned long long*>(a.pool[c] + static_cast<int64_t>(pid) * a.page_bytes[c] + a.hdr +
                                               static_cast<int64_t>(j + 1) * a.slice[c] - a.maskb);
}
__device__ __forceinline__ int entry_bits(const uint8_t* bits, const float* bit_logits, int e) {
  return bit_logits ? 2 << hard_decision<4>(bit_logits + 4 * e) : bits[e];
}

__global__ void __launch_bounds__(1024) append_plan_kernel(LayerArgs a, int n, const int32_t* __restrict__ seq_ids,
                                                           const int32_t* __restrict__ positions,
                                                           const uint8_t* __restrict__ bits,
                                                           const uint8_t* __restrict__ modes,
                                                           const float* __restrict__ bit_logits,
                                                           const float* __restrict__ mode_logits) {
  __shared__ int s_seq[1024];
  __shared__ int s_pos[1024];
  __shared__ int s_cls[1024];   // width class when the entry stores KV, else -1
  __shared__ int s_open[1024];  // class of the page the entry opens, else -1
  __shared__ int s_first_err;
  __shared__ int s_nopen[kClasses];

  pdl_wait();
  pdl_trigger();
  const int e = threadIdx.x;
  const bool act = e < n;
  int seq = -1, pos = 0, c = -1, err = 0;
  bool writes = false;
  if (act) {
    seq = seq_ids[e];
    pos = positions[e];
    const int m = entry_mode(a, modes, mode_logits, e);
    if (seq < 0 || seq >= a.S) {
      err = TRR_ERR_INVALID_ARG;
    } else {
      c = class_of_bits(entry_bits(bits, bit_logits, e));
      if (c < 0 || m > TRR_MODE_FULL) err = TRR_ERR_INVALID_ARG;
      else if (pos < 0 || pos >= a.maxctx) err = TRR_ERR_BAD_POSITION;
    }
    writes = !err && (m != TRR_MODE_SKIP || a.skip_writes_kv);
  }
  s_seq[e] = (act && seq >= 0 && seq < a.S) ? seq : -1;
  s_pos[e] = pos;
  s_cls[e] = writes ? c : -1;
  if (e == 0) s_first_err = INT_MAX;
  if (e < kClasses) s_nopen[e] = 0;
  __syncthreads();

  // Earlier entries of the same sequence: the largest position and, per class, how
  // many store KV.  Later ones: whether this entry is the sequence's / class's last.
  int prev_max = -1, rank = 0;
  bool later_seq = false, later_cls = false;
  if (act && s_seq[e] >= 0) {
    for (int j = 0; j < n; ++j) {
      if (s_seq[j] != seq) continue;
      if (j < e) {
        prev_max = max(prev_max, s_pos[j]);
        rank += (writes && s_cls[j] == c);
      } else if (j > e) {
        later_seq = true;
        later_cls |= (writes && s_cls[j] == c);
      }
    }
  }
  int k = 0, slot = 0, kidx = 0;
  bool opens = false;
  if (act && !err && pos <= max(prev_max, a.last_pos[seq])) err = TRR_ERR_BAD_POSITION;
  if (act && !err && writes) {
    k = a.ntok[seq * 4 + c] + rank;
    slot = k % a.P;
    kidx = k / a.P;
    opens = slot == 0;
  }
  s_open[e] = opens ? c : -1;
  __syncthreads();

  int pid = -1;
  if (opens) {  // page ids in entry order: next_page + openers of this class before e
    int before = 0;
    for (int j = 0; j < e; ++j) before += (s_open[j] == c);
    pid = a.ctrl[kNextPage + c] + before;
    if (pid >= a.cap[c]) err = TRR_ERR_OUT_OF_PAGES;
  }
  if (act && err) atomicMin(&s_first_err, e);
  __syncthreads();
  if (s_first_err != INT_MAX) {  // the call is a no-op; record the lowest failing entry
    if (e == s_first_err) set_status(a.ctrl, err);
    if (e == 0) a.ctrl[kAppendOk] = 0;
    return;
  }

  // Commit.  Openers first, so that later entries of the same page can read its id.
  const int64_t row = (static_cast<int64_t>(seq) * 4 + c) * a.MP + kidx;
  if (opens) {
    a.pt[row] = pid;
    a.pfirst[row] = pos;
    atomicAdd(&s_nopen[c], 1);
    if (a.head_modes)  // a new page starts with every presence bit (and the padding) clear
      for (int j = 0; j < a.Hkv; ++j) {
        head_mask(a, c, pid, j)[0] = 0ull;
        head_mask(a, c, pid, j)[1] = 0ull;
      }
  }
  __syncthreads();
  if (act) {
    AppendPlan p{-1, 0, 0, pos};
    if (writes) {
      if (!opens) pid = a.pt[row];
      p.page = pid;
      p.slot = slot;
      p.cls = c;
      if (!later_cls || slot == a.P - 1) a.plast[row] = pos;
      if (!later_cls) {
        a.ntok[seq * 4 + c] = k + 1;
        a.lastpg[seq * 4 + c] = pid;
      }
      reinterpret_cast<int32_t*>(a.pool[c] + pid * a.page_bytes[c])[slot] = pos;
      atomicOr(&a.presence[static_cast<int64_t>(seq) * a.W32 + pos / 32], 1u << (pos % 32));
      if (a.head_modes)  // the slot's bit for every KV head the entry stores
        for (int j = 0; j < a.Hkv; ++j)
          if (head_stores(a, modes, e, j)) atomicOr(head_mask(a, c, pid, j), 1ull << slot);
    }
    a.aplan[e] = p;
    if (!later_seq) a.last_pos[seq] = pos;
  }
  __syncthreads();
  if (e < kClasses) a.ctrl[kNextPage + e] += s_nopen[e];
  if (e == 0) a.ctrl[kAppendOk] = 1;
}

// Eq. 4 on 32 consecutive values (one chunk of a group): codes packed LSB-first.
template <int B>
__device__ __forceinline__ void quantise_chunk(const uint4* src, float z, float s, float rs, uint8_t* sl, int64_t off,
                                               bool sw) {
  constexpr int levels = (1 << B) - 1;
  constexpr int per_word = 32 / B;
  uint32_t words[B];
#pragma unroll
  for (int w = 0; w < B; ++w) words[w] = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint4 u = src[q];
    const uint32_t wv[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int h = 0; h < 8; ++h) {
      const float x = (h & 1) ? bf16hi(wv[h >> 1]) : bf16lo(wv[h >> 1]);
      const int code = s != 0.f ? code_of(x, z, s, rs, levels) : 0;
      const int j = q * 8 + h;
      words[j / per_word] |= static_cast<uint32_t>(code) << ((j % per_word) * B);
    }
  }
#pragma unroll
  for (int w = 0; w < B; ++w) {  // word w at byte off + 4 w of the slice (swizzled: sw)
    const int64_t o = off + 4 * w;
    *reinterpret_cast<uint32_t*>(sl + (sw ? swz_off(o) : o)) = words[w];
  }
}

__global__ void __launch_bounds__(256) append_write_kernel(LayerArgs a, int n, const uint16_t* __restrict__ k,
                                                           const uint16_t* __restrict__ v) {
  pdl_wait();
  pdl_trigger();
  if (a.ctrl[kAppendOk] == 0) return;
  const int ng = a.d / a.G;
  const int per_entry = a.Hkv * 2 * ng;
  const int64_t gid = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (gid >= static_cast<int64_t>(n) * per_entry) return;
  const int e = static_cast<int>(gid / per_entry);
  const int r = static_cast<int>(gid % per_entry);
  const int h = r / (2 * ng);
  const int which = (r / ng) & 1;  // 0 = K, 1 = V
  const int g = r % ng;
  const AppendPlan p = a.aplan[e];
  if (p.page < 0) return;
  const int b = bits_of_class(p.cls);
  const uint16_t* src = (which ? v : k) + (static_cast<int64_t>(e) * a.Hkv + h) * a.d + g * a.G;
  uint8_t* sl = a.pool[p.cls] + p.page * a.page_bytes[p.cls] + a.hdr + static_cast<int64_t>(h) * a.slice[p.cls];
  const uint4* s4 = reinterpret_cast<const uint4*>(src);
  if (b == 16) {  // native precision: copy the bf16 bits, 16 bytes (one chunk) at a time
    const int64_t off = static_cast<int64_t>(which) * a.P * a.d * 2 + static_cast<int64_t>(p.slot) * a.d * 2 + g * a.G * 2;
    for (int i = 0; i < a.G / 8; ++i) {
      const int64_t o = off + 16 * i;
      *reinterpret_cast<uint4*>(sl + (a.swz ? swz_off(o) : o)) = s4[i];
    }
    return;
  }
  // min / max of the group; values binary16 cannot carry make the group all zeros
  float mn = __int_as_float(0x7f800000), mx = -mn;
  bool bad = false;
  for (int i = 0; i < a.G / 8; ++i) {
    const uint4 u = s4[i];
    const uint32_t wv[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int h2 = 0; h2 < 8; ++h2) {
      const float x = (h2 & 1) ? bf16hi(wv[h2 >> 1]) : bf16lo(wv[h2 >> 1]);
      bad |= !(fabsf(x) <= 65504.f);  // also true for NaN
      mn = fminf(mn, x);
      mx = fmaxf(mx, x);
    }
  }
  const int rowb = a.d * b / 8;
  const bool sw = a.swz && b == 8;  // 8-bit rows of a swizzled cache
  const int64_t coff = static_cast<int64_t>(which) * a.P * rowb + static_cast<int64_t>(p.slot) * rowb + g * a.G * b / 8;
  uint32_t* sz = reinterpret_cast<uint32_t*>(sl + 2 * static_cast<int64_t>(a.P) * rowb +
                                             static_cast<int64_t>(which) * a.P * ng * 4 +
                                             static_cast<int64_t>(p.slot) * ng * 4 + g * 4);
  if (bad) {
    for (int i = 0; i < a.G * b / 32; ++i) {
      const int64_t o = coff + 4 * i;
      *reinterpret_cast<uint32_t*>(sl + (sw ? swz_off(o) : o)) = 0;
    }
    *sz = 0;
    set_status(a.ctrl, TRR_ERR_BAD_VALUE);
    return;
  }
  const __half z16 = __float2half_rn(mn);                                   // z = min(x)
  const float levels = static_cast<float>((1 << b) - 1);
  const __half s16 = __float2half_rn(__fdiv_rn(__fsub_rn(mx, mn), levels));  // s
  const float z = __half2float(z16), s = __half2float(s16), rs = __frcp_rn(s);
  for (int q = 0; q < a.G / 32; ++q) {
    const int64_t off = coff + 4 * q * b;  // 32 codes of b bits = b words
    if (b == 2) quantise_chunk<2>(s4 + 4 * q, z, s, rs, sl, off, false);
    else if (b == 4) quantise_chunk<4>(s4 + 4 * q, z, s, rs, sl, off, false);
    else quantise_chunk<8>(s4 + 4 * q, z, s, rs, sl, off, sw);
  }
  *sz = static_cast<uint32_t>(__half_as_ushort(s16)) | (static_cast<uint32_t>(__half_as_ushort(z16)) << 16);
}

// ------------------------------------------------------------ one-kernel append --
//
// For calls of up to kFusedMax entries (a decode step) one kernel does the whole append.
// Every CTA plans every entry (the same deterministic plan as append_plan_kernel, from
// the metadata as the call found it), each warp quantises one (entry, KV head, K|V) row,
// and the last CTA to finish commits the metadata: no CTA reads metadata after the
// commit, since every other CTA has finished by then.

constexpr int kFusedMax = 256;

// One row of d values (entry, KV head, K or V) by a warp, written to its slot.
// The codes go to byte row_off of the slice sl (swizzled when sw).
template <int D>
__device__ __forceinline__ void quantise_row(const uint2 w, uint8_t* sl, int64_t row_off, bool sw, uint32_t* sz_row,
                                             int b, int G, int lane, int32_t* ctrl) {
  const RowCodes r = quantise_row_codes<D>(w, b, G, lane);
  if (r.bad && r.sz_idx >= 0) set_status(ctrl, TRR_ERR_BAD_VALUE);
  if (r.code_idx >= 0) {
    const int64_t o = row_off + 4 * r.code_idx;
    *reinterpret_cast<uint32_t*>(sl + (sw ? swz_off(o) : o)) = r.code_word;
  }
  if (r.sz_idx >= 0) sz_row[r.sz_idx] = r.sz_word;
}

template <int D>
__global__ void __launch_bounds__(256) append_fused_kernel(LayerArgs a, int n, const int32_t* __restrict__ seq_ids,
                                                           const int32_t* __restrict__ positions,
                                                           const uint8_t* __restrict__ bits,
                                                           const uint8_t* __restrict__ modes,
                                                           const float* __restrict__ bit_logits,
                                                           const float* __restrict__ mode_logits,
                                                           const uint16_t* __restrict__ k,
                                                           const uint16_t* __restrict__ v) {
  __shared__ int s_seq[kFusedMax];
  __shared__ int s_pos[kFusedMax];
  __shared__ int s_cls[kFusedMax];   // width class when the entry stores KV, else -1
  __shared__ int s_k[kFusedMax];     // token index in the (sequence, class) list
  __shared__ int s_pid[kFusedMax];   // page of the token (openers: the new page)
  __shared__ int s_wopen[8][kClasses];
  __shared__ int s_next[kClasses];
  __shared__ int s_first_err;
  __shared__ int s_last;

  const int e = threadIdx.x, lane = e & 31, warp = e >> 5;
  const bool act = e < n;
  // The call's own inputs (entries, K/V rows) are read first: no kernel of this library
  // writes them, so this overlaps the previous kernel of the stream.  Cache metadata and
  // control words come after the wait.
  // this warp's row (entry, KV head, K|V), loaded while the entries are planned
  const int row = blockIdx.x * (blockDim.x >> 5) + warp;
  const bool has_row = row < n * a.Hkv * 2;
  const int re = row / (2 * a.Hkv), rh = (row >> 1) % a.Hkv, which = row & 1;
  uint2 raw = make_uint2(0, 0);
  if (has_row) {
    const uint16_t* src = (which ? v : k) + (static_cast<int64_t>(re) * a.Hkv + rh) * D;
    if (D == 64) raw.x = reinterpret_cast<const uint32_t*>(src)[lane];
    else raw = reinterpret_cast<const uint2*>(src)[lane];
  }
  int seq = -1, pos = 0, c = -1, err = 0;
  bool writes = false;
  if (act) {
    seq = seq_ids[e];
    pos = positions[e];
    const int m = entry_mode(a, modes, mode_logits, e);
    if (seq < 0 || seq >= a.S) {
      err = TRR_ERR_INVALID_ARG;
    } else {
      c = class_of_bits(entry_bits(bits, bit_logits, e));
      if (c < 0 || m > TRR_MODE_FULL) err = TRR_ERR_INVALID_ARG;
      else if (pos < 0 || pos >= a.maxctx) err = TRR_ERR_BAD_POSITION;
    }
    writes = !err && (m != TRR_MODE_SKIP || a.skip_writes_kv);
  }
  s_seq[e] = (act && seq >= 0 && seq < a.S) ? seq : -1;
  s_pos[e] = pos;
  s_cls[e] = writes ? c : -1;
  pdl_wait();
  pdl_trigger();
  if (e < kClasses) s_next[e] = a.ctrl[kNextPage + e];
  if (e == 0) s_first_err = INT_MAX;
  __syncthreads();

  // earlier entries of the same sequence: the largest position and, per class, how many
  // store KV; later ones: whether this entry is the sequence's / class's last
  int prev_max = -1, rank = 0;
  bool later_seq = false, later_cls = false;
  if (act && s_seq[e] >= 0) {
    for (int j = 0; j < n; ++j) {
      if (s_seq[j] != seq) continue;
      if (j < e) {
        prev_max = max(prev_max, s_pos[j]);
        rank += (writes && s_cls[j] == c);
      } else if (j > e) {
        later_seq = true;
        later_cls |= (writes && s_cls[j] == c);
      }
    }
  }
  int tok = 0, nt_old = 0, last_page = -1;
  bool opens = false;
  if (act && !err) {
    const int lp = a.last_pos[seq];
    if (writes) {
      nt_old = a.ntok[seq * 4 + c];
      last_page = a.lastpg[seq * 4 + c];
    }
    if (pos <= max(prev_max, lp)) err = TRR_ERR_BAD_POSITION;
    if (writes) {
      tok = nt_old + rank;
      opens = tok % a.P == 0;
    }
  }
  // page ids in entry order: next_page + openers of the same class before e
  int before = 0;
#pragma unroll
  for (int cc = 0; cc < kClasses; ++cc) {
    const unsigned bal = __ballot_sync(0xffffffffu, !err && opens && c == cc);
    if (lane == 0) s_wopen[warp][cc] = __popc(bal);
    if (c == cc) before = __popc(bal & ((1u << lane) - 1u));
  }
  __syncthreads();
  int pid = -1;
  if (opens) {
    for (int w = 0; w < warp; ++w) before += s_wopen[w][c];
    pid = s_next[c] + before;
    if (pid >= a.cap[c]) err = TRR_ERR_OUT_OF_PAGES;
  }
  if (act && err) atomicMin(&s_first_err, e);
  s_k[e] = tok;
  s_pid[e] = pid;
  __syncthreads();
  if (s_first_err != INT_MAX) {  // the call is a no-op; record the lowest failing entry
    if (blockIdx.x == 0 && e == s_first_err) set_status(a.ctrl, err);
    return;
  }
  const int kidx = tok / a.P;
  const int64_t prow = (static_cast<int64_t>(seq) * 4 + c) * a.MP + kidx;
  if (writes && !opens) {  // a page opened earlier: by a previous call (then the class's
                           // last page), or by an earlier entry of this call
    if (kidx * a.P < nt_old) {
      pid = last_page;
    } else {
      for (int j = 0; j < e; ++j)
        if (s_seq[j] == seq && s_cls[j] == c && s_k[j] == kidx * a.P) pid = s_pid[j];
    }
    s_pid[e] = pid;
  }
  __syncthreads();

  if (has_row) {
    const int rc = s_cls[re];
    if (rc >= 0) {
      const int b = bits_of_class(rc), slot = s_k[re] % a.P;
      uint8_t* sl = a.pool[rc] + static_cast<int64_t>(s_pid[re]) * a.page_bytes[rc] + a.hdr +
                    static_cast<int64_t>(rh) * a.slice[rc];
      if (b == 16) {  // this lane's D/32 values (4 or 8 bytes: inside one 16-byte chunk)
        const int64_t o = (static_cast<int64_t>(which) * a.P + slot) * D * 2 + lane * (D / 16);
        uint8_t* dst = sl + (a.swz ? swz_off(o) : o);
        if (D == 64) *reinterpret_cast<uint32_t*>(dst) = raw.x;
        else *reinterpret_cast<uint2*>(dst) = raw;
      } else {
        const int rowb = D * b / 8, ng = D / a.G;
        uint32_t* sz_row = reinterpret_cast<uint32_t*>(sl + 2 * static_cast<int64_t>(a.P) * rowb +
                                                      (static_cast<int64_t>(which) * a.P + slot) * ng * 4);
        quantise_row<D>(raw, sl, (static_cast<int64_t>(which) * a.P + slot) * rowb, a.swz && b == 8, sz_row, b, a.G,
                        lane, a.ctrl);
      }
    }
  }

  // the last CTA to finish commits the metadata of every entry: its acquire follows the
  // release of every other CTA, after all of their reads of the old metadata
  __syncthreads();
  if (e == 0) s_last = atom_add_acq_rel(&a.ctrl[kAppendDone], 1) == static_cast<int>(gridDim.x) - 1;
  __syncthreads();
  if (!s_last) return;
  if (act) {
    if (writes) {
      const int slot = tok % a.P;
      if (opens) {
        a.pt[prow] = pid;
        a.pfirst[prow] = pos;
      }
      if (!later_cls || slot == a.P - 1) a.plast[prow] = pos;
      if (!later_cls) {
        a.ntok[seq * 4 + c] = tok + 1;
        a.lastpg[seq * 4 + c] = pid;
      }
      reinterpret_cast<int32_t*>(a.pool[c] + static_cast<int64_t>(pid) * a.page_bytes[c])[slot] = pos;
      atomicOr(&a.presence[static_cast<int64_t>(seq) * a.W32 + pos / 32], 1u << (pos % 32));
    }
    if (!later_seq) a.last_pos[seq] = pos;
  }
  if (a.head_modes) {  // presence masks: openers clear their new pages, then every entry
                       // sets its slot's bit for the KV heads it stores
    const bool mine = act && writes;
    if (mine && opens)
      for (int j = 0; j < a.Hkv; ++j) {
        head_mask(a, c, pid, j)[0] = 0ull;
        head_mask(a, c, pid, j)[1] = 0ull;
      }
    __syncthreads();
    if (mine)
      for (int j = 0; j < a.Hkv; ++j)
        if (head_stores(a, modes, e, j)) atomicOr(head_mask(a, c, pid, j), 1ull << (tok % a.P));
  }
  if (e < kClasses) {
    int opened = 0;
    for (int w = 0; w < 8; ++w) opened += s_wopen[w][e];
    a.ctrl[kNextPage + e] = s_next[e] + opened;
  }
  if (e == 0) a.ctrl[kAppendDone] = 0;
}

}  // namespace trr

using namespace trr;

// One append call: the entries' modes and widths come from `bits` / `modes`, or (with
// those null) from the router logits.
static trr_status append_call(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                              const int32_t* positions, const void* k_bf16, const void* v_bf16, const uint8_t* bits,
                              const uint8_t* modes, const float* bit_logits, const float* mode_logits,
                              void* stream) {
  if (!cache) return TRR_ERR_INVALID_ARG;
  const Layout& l = cache_layout(cache);
  if (layer < 0 || layer >= l.L || n < 0 || n > l.max_append) return TRR_ERR_INVALID_ARG;
  cache_set_launches(cache, 0);
  if (n == 0) return TRR_OK;
  if (!seq_ids || !positions || !k_bf16 || !v_bf16 || !(bits || bit_logits) || !(modes || mode_logits))
    return TRR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(k_bf16) | reinterpret_cast<uintptr_t>(v_bf16)) & 15)
    return TRR_ERR_INVALID_ARG;  // rows are read 16 bytes at a time
  if ((reinterpret_cast<uintptr_t>(bit_logits) | reinterpret_cast<uintptr_t>(mode_logits)) & 3)
    return TRR_ERR_INVALID_ARG;
  if (mode_logits && l.head_modes) return TRR_ERR_UNSUPPORTED;  // router decisions are per token
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const LayerArgs a = layer_args(l, cache_views(cache), layer);
  cache_note_call(cache, layer);
  const uint16_t* k = static_cast<const uint16_t*>(k_bf16);
  const uint16_t* v = static_cast<const uint16_t*>(v_bf16);
  if (n <= kFusedMax) {  // one kernel: 256 threads plan, one warp per (entry, head, K|V) row
    const unsigned blocks = static_cast<unsigned>((static_cast<int64_t>(n) * l.Hkv * 2 + 7) / 8);
    const cudaError_t e =
        l.d == 64 ? launch_pdl(append_fused_kernel<64>, dim3(blocks), dim3(256), 0, s, a, n, seq_ids, positions, bits,
                               modes, bit_logits, mode_logits, k, v)
                  : launch_pdl(append_fused_kernel<128>, dim3(blocks), dim3(256), 0, s, a, n, seq_ids, positions,
                               bits, modes, bit_logits, mode_logits, k, v);
    cache_set_launches(cache, 1);
    return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
  }
  const int threads = (n + 31) / 32 * 32;
  cudaError_t e = launch_pdl(append_plan_kernel, dim3(1), dim3(threads), 0, s, a, n, seq_ids, positions, bits, modes,
                             bit_logits, mode_logits);
  if (e != cudaSuccess) return TRR_ERR_CUDA;
  const int64_t work = static_cast<int64_t>(n) * l.Hkv * 2 * (l.d / l.G);
  e = launch_pdl(append_write_kernel, dim3(static_cast<unsigned>((work + 255) / 256)), dim3(256), 0, s, a, n, k, v);
  cache_set_launches(cache, 2);
  return e == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}

extern "C" trr_status trr_kv_append(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                    const int32_t* positions, const void* k_bf16, const void* v_bf16,
                                    const uint8_t* bits, const uint8_t* modes, void* stream) {
  return append_call(cache, layer, n, seq_ids, positions, k_bf16, v_bf16, bits, modes, nullptr, nullptr, stream);
}

extern "C" trr_status trr_kv_append_routed(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                           const int32_t* positions, const void* k_bf16, const void* v_bf16,
                                           const float* bit_logits, const float* mode_logits, void* stream) {
  return append_call(cache, layer, n, seq_ids, positions, k_bf16, v_bf16, nullptr, nullptr, bit_logits, mode_logits,
                     stream);
}
