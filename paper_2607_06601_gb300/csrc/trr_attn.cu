// trr_attn.cu - trr_decode_attn: mode-routed split-K decode attention over the
// mixed-precision paged cache (Sec. 3.2(A), Eq. 2; Sec. 3.8; Sec. 7).
//
// One persistent kernel per call (two CTAs per SM, every warp an independent worker):
//   1. Every CTA cuts the call into work units: query q gets ns_q splits from the
//      length of its key range (full: [0, t]; local: [t-w+1, t]; skip or invalid: one
//      unit that writes the zero row) and a prefix sum numbers the units.  The same
//      deterministic computation in every CTA takes the place of a planning kernel.
//   2. Work items (unit, query head) are dealt round-robin to the warps.  A warp plans
//      its item itself: the sequence's per-class token counts, a 32-way search of the
//      pages' first / last positions at window edges, and the split's share of every
//      class's pages in range (one page id per lane).  It streams those pages' slices
//      of the head through a private ring of shared memory filled by 1-D bulk copies
//      (cp.async.bulk + mbarrier), the query row riding on the first copy of each
//      item, so items follow each other without a pipeline drain.  Lane pair (key,
//      half) of a 64-wide head (four lanes for 128) dequantises in registers and keeps
//      its own online softmax; lanes merge with shuffles.
//   3. A query with one split gets its bf16 row from that item.  Otherwise each split
//      writes an fp32 partial and counts its arrival; the last split of the (query,
//      head) to arrive merges the partials, writes the row and resets the counter.
//   4. The last CTA to finish records the error of the lowest failing query.
//
// Dequantisation: k = z + c*s, so q.k = s * sum(q_i c_i) + z * sum(q_i).  A code is
// masked in place (no shift) and its bits read as a binary32 subnormal, c * 2^(e-149)
// where e is its bit offset; the query is pre-scaled per width class by 2^(100-e) so
// that q_i * x_i = q_i c_i 2^-49 exactly as an fp32 product.  V is accumulated in a
// domain scaled by 2^-49 with the per-offset factor folded into the key's weight.
#include <algorithm>
#include <climits>

#include "trr_internal.cuh"

namespace trr {

#define kNegInf (-__int_as_float(0x7f800000))
constexpr float kTau = 8.f;    // lazy rescale threshold (log2 units)


// ----------------------------------------------------------------------- plan --

// For NS increasing arrays arr_i = base + i * stride of n[i] entries: the count of
// entries below x, searched by the whole warp.  The first round probes the last 32
// entries: decode queries look at the end of the page lists, so that round almost always
// settles it.  Otherwise 32 probes per round narrow the rest.  Every search advances in
// the same round.
template <int NS>
__device__ __forceinline__ void warp_count_below(const int* base, int64_t stride, const int (&n)[NS], int x,
                                                 int (&out)[NS], int lane) {
  int lo[NS], hi[NS];
#pragma unroll
  for (int i = 0; i < NS; ++i) {
    const int idx = max(0, n[i] - 32) + lane;
    const int v = idx < n[i] ? base[i * stride + idx] : INT_MAX;
    const unsigned below = __ballot_sync(0xffffffffu, idx < n[i] && v < x);
    const int b = max(0, n[i] - 32);
    if (n[i] <= 32 || (below & 1u)) {  // arr[b] < x: everything before it is too
      lo[i] = hi[i] = b + __popc(below);
    } else {
      lo[i] = 0;
      hi[i] = b;
    }
  }
  for (int round = 0; round < 6; ++round) {
    bool any = false;
#pragma unroll
    for (int i = 0; i < NS; ++i) any |= hi[i] > lo[i];
    if (!any) break;
#pragma unroll
    for (int i = 0; i < NS; ++i) {
      const int span = hi[i] - lo[i];
      const int step = span <= 32 ? 1 : (span + 31) / 32;
      const int idx = lo[i] + lane * step;
      const int v = (span > 0 && idx < hi[i]) ? base[i * stride + idx] : INT_MAX;
      const int cnt = __popc(__ballot_sync(0xffffffffu, idx < hi[i] && v < x));
      if (span <= 0) continue;
      if (span <= 32 || cnt == 0) {
        lo[i] = hi[i] = lo[i] + (span <= 32 ? cnt : 0);
      } else {
        const int last = lo[i] + (cnt - 1) * step;  // last probe below x
        hi[i] = min(hi[i], lo[i] + cnt * step);
        lo[i] = last + 1;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < NS; ++i) out[i] = lo[i];
}

// ------------------------------------------------------------------ dequant --

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// exact 2^e, -126 <= e <= 127 (folds to a constant for constant e)
__device__ __forceinline__ float pow2f(int e) { return __int_as_float((127 + e) << 23); }

// Bit offset of element i (of a lane's 32) inside the word it is extracted from.
__host__ __device__ constexpr int ex_of(int B, int i) {
  return B == 2 ? ((i % 16) < 11 ? 2 * (i % 16) : 2 * (i % 16 - 11))
                : B == 4 ? ((i % 8) < 5 ? 4 * (i % 8) : 4 * (i % 8 - 5)) : 0;
}
// Pre-scale exponent of the query in class B.
__host__ __device__ constexpr int qe_of(int B, int i) { return B == 16 ? 0 : 100 - ex_of(B, i); }

// Element i as c * 2^(ex-149): the code left in place, read as a subnormal.
template <int B>
__device__ __forceinline__ float code_at(const uint32_t* w, const uint32_t* h, int i) {
  if (B == 2) {
    const int j = i % 16;
    return __uint_as_float(j < 11 ? (w[i / 16] & (3u << (2 * j))) : (h[i / 16] & (3u << (2 * (j - 11)))));
  } else if (B == 4) {
    const int j = i % 8;
    return __uint_as_float(j < 5 ? (w[i / 8] & (15u << (4 * j))) : (h[i / 8] & (15u << (4 * (j - 5)))));
  } else {
    return __uint_as_float(__byte_perm(w[i / 4], 0u, 0x4440u | (i % 4)));
  }
}
// d = a * b + c on two fp32 lanes at once (packed fp32 FMA, round to nearest).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }

template <int B>
__device__ __forceinline__ void high_parts(const uint32_t* w, uint32_t* h) {
  constexpr int sh = B == 2 ? 22 : B == 4 ? 20 : 16;
#pragma unroll
  for (int k = 0; k < B; ++k) h[k] = w[k] >> sh;
}

// x *= f on pairs of fp32 lanes (packed multiply)
__device__ __forceinline__ void fmul2_inplace(float& x0, float& x1, float f0, float f1) {
  const float2 r = __fmul2_rn(make_float2(x0, x1), make_float2(f0, f1));
  x0 = r.x;
  x1 = r.y;
}

template <int BFROM, int BTO>
__device__ __forceinline__ void rescale_q(float (&qp)[32]) {
#pragma unroll
  for (int i = 0; i < 32; i += 2)
    fmul2_inplace(qp[i], qp[i + 1], pow2f(qe_of(BTO, i) - qe_of(BFROM, i)),
                  pow2f(qe_of(BTO, i + 1) - qe_of(BFROM, i + 1)));
}

// V is accumulated as acc_i * 2^(ex_i(B) - 49) while class B's pages are consumed
// (B = 16: ex = 0), so that every element of a key takes the same weight p*s*2^100.
template <int BFROM, int BTO>
__device__ __forceinline__ void rescale_acc(float (&acc)[32]) {
#pragma unroll
  for (int i = 0; i < 32; i += 2)
    fmul2_inplace(acc[i], acc[i + 1],
                  pow2f((BTO == 16 ? 0 : ex_of(BTO, i)) - (BFROM == 16 ? 0 : ex_of(BFROM, i))),
                  pow2f((BTO == 16 ? 0 : ex_of(BTO, i + 1)) - (BFROM == 16 ? 0 : ex_of(BFROM, i + 1))));
}

// qp from the domain of class `from` to that of class `to` (from < to, or from = 16).
__device__ __forceinline__ void rescale_dyn(float (&qp)[32], float (&acc)[32], int from, int to) {
  switch (from * 4 + to) {
    case 1: rescale_q<2, 4>(qp); rescale_acc<2, 4>(acc); break;
    case 2: rescale_q<2, 8>(qp); rescale_acc<2, 8>(acc); break;
    case 3: rescale_q<2, 16>(qp); rescale_acc<2, 16>(acc); break;
    case 6: rescale_q<4, 8>(qp); rescale_acc<4, 8>(acc); break;
    case 7: rescale_q<4, 16>(qp); rescale_acc<4, 16>(acc); break;
    case 11: rescale_q<8, 16>(qp); rescale_acc<8, 16>(acc); break;
    case 12: rescale_q<16, 2>(qp); rescale_acc<16, 2>(acc); break;
    case 13: rescale_q<16, 4>(qp); rescale_acc<16, 4>(acc); break;
    case 14: rescale_q<16, 8>(qp); rescale_acc<16, 8>(acc); break;
    default: break;
  }
}
// acc from class `from`'s domain back to class 16's (the common one of the merge)
__device__ __forceinline__ void acc_to_neutral(float (&acc)[32], int from) {
  switch (from) {
    case 0: rescale_acc<2, 16>(acc); break;
    case 1: rescale_acc<4, 16>(acc); break;
    case 2: rescale_acc<8, 16>(acc); break;
    default: break;
  }
}

// 2^x with the hardware approximation (relative error about 2^-22; results below the
// binary32 normal range flush to zero, far below a softmax sum's resolution).
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct LaneState {
  float m, l, zacc;  // running max (log2), sum of weights, sum of p*z (V zero points)
  float acc[32];     // sum of p*v over the lane's 32 dims, scaled by 2^-49
};

__device__ __forceinline__ float softmax_step(LaneState& st, float score) {
  if (score > st.m + kTau) {
    const float alpha = fast_exp2(st.m - score);  // 0 when m = -inf
#pragma unroll
    for (int j = 0; j < 32; ++j) st.acc[j] *= alpha;
    st.l *= alpha;
    st.zacc *= alpha;
    st.m = score;
  }
  const float p = fast_exp2(score - st.m);
  st.l += p;
  return p;
}

// Shared-memory loads at 32-bit shared addresses.  Volatile: they stay after the
// mbarrier wait that makes the bytes valid.
__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
__device__ __forceinline__ uint2 lds64(uint32_t a) {
  uint2 v;
  asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
  return v;
}
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
  return v;
}

// The B words of 32 B-bit codes at shared address a (4B-byte aligned), in as few loads as
// possible (one 8- or 16-byte load per row part keeps the warp's request conflict-free).
template <int B>
__device__ __forceinline__ void lds_codes(uint32_t a, uint32_t* w) {
  if (B == 2) {
    const uint2 u = lds64(a);
    w[0] = u.x; w[1] = u.y;
  } else {
#pragma unroll
    for (int k = 0; k < B; k += 4) {
      const uint4 u = lds128(a + 4 * k);
      w[k] = u.x; w[k + 1] = u.y; w[k + 2] = u.z; w[k + 3] = u.w;
    }
  }
}

// One page of width class B (P = NIT * keys per iteration tokens) at shared address s0;
// lane -> (key kl, 32-dim part).  Keys past `fill` are empty slots; with positions at
// spos (masked pages), keys outside [lo, hi] are masked too.
template <int D, int B, int NIT>
__device__ __forceinline__ void consume_page(uint32_t s0, uint32_t spos, bool masked, int G, int fill, int lo,
                                             int hi, const float (&qp)[32], float sumq, LaneState& st, int lane) {
  constexpr int LPK = D / 32;
  constexpr int KPI = 32 / LPK;
  constexpr int P = NIT * KPI;
  constexpr int rowb = B == 16 ? 2 * D : D * B / 8;  // bytes of one key's row of K (or V)
  const int part = lane % LPK, kl = lane / LPK;
  const int ng = D / G;
  const int grp = part * 32 / G;
  const uint32_t krow = s0 + kl * rowb + part * (B == 16 ? 64 : 4 * B);   // this lane's K bytes, key kl
  const uint32_t ksz = s0 + 2 * P * rowb + (kl * ng + grp) * 4;           // its (s, z), key kl
  const uint32_t szstep = KPI * ng * 4;
#pragma unroll 1
  for (int it = 0; it < NIT; ++it) {
    const int key = it * KPI + kl;
    bool valid = key < fill;
    if (masked) {
      const int pos = static_cast<int>(lds32(spos + 4 * key));
      valid = valid && pos >= lo && pos <= hi;
    }
    const uint32_t ka = krow + it * KPI * rowb, va = ka + P * rowb;
    float dot;
    if (B == 16) {
      float2 d2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 u = lds128(ka + 16 * q);
        d2[0] = ffma2(make_float2(qp[8 * q + 0], qp[8 * q + 1]), make_float2(bf_lo(u.x), bf_hi(u.x)), d2[0]);
        d2[1] = ffma2(make_float2(qp[8 * q + 2], qp[8 * q + 3]), make_float2(bf_lo(u.y), bf_hi(u.y)), d2[1]);
        d2[0] = ffma2(make_float2(qp[8 * q + 4], qp[8 * q + 5]), make_float2(bf_lo(u.z), bf_hi(u.z)), d2[0]);
        d2[1] = ffma2(make_float2(qp[8 * q + 6], qp[8 * q + 7]), make_float2(bf_lo(u.w), bf_hi(u.w)), d2[1]);
      }
      dot = (d2[0].x + d2[0].y) + (d2[1].x + d2[1].y);
    } else {
      uint32_t w[B], h[B];
      lds_codes<B>(ka, w);
      if (B != 8) high_parts<B>(w, h);
      const uint32_t szw = lds32(ksz + it * szstep);
      float2 d2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
      for (int i = 0; i < 16; ++i)
        d2[i & 1] = ffma2(make_float2(qp[2 * i], qp[2 * i + 1]),
                          make_float2(code_at<B>(w, h, 2 * i), code_at<B>(w, h, 2 * i + 1)), d2[i & 1]);
      const float2 sz = __half22float2(*reinterpret_cast<const __half2*>(&szw));  // (s, z)
      dot = fmaf(sz.x * pow2f(49), (d2[0].x + d2[0].y) + (d2[1].x + d2[1].y), sz.y * sumq);
    }
#pragma unroll
    for (int o = 1; o < LPK; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    if (valid) {
      const float p = softmax_step(st, dot);
      if (B == 16) {
        const float wv = p * pow2f(-49);
        const float2 w2 = make_float2(wv, wv);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 u = lds128(va + 16 * q);
          const uint32_t uw[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const int i = 8 * q + 2 * h;
            const float2 r = ffma2(w2, make_float2(bf_lo(uw[h]), bf_hi(uw[h])), make_float2(st.acc[i], st.acc[i + 1]));
            st.acc[i] = r.x;
            st.acc[i + 1] = r.y;
          }
        }
      } else {
        uint32_t w[B], h[B];
        lds_codes<B>(va, w);
        if (B != 8) high_parts<B>(w, h);
        const uint32_t szw = lds32(ksz + it * szstep + P * ng * 4);
        const float2 sz = __half22float2(*reinterpret_cast<const __half2*>(&szw));  // (s, z)
        const float wb = p * sz.x * pow2f(100);
        const float2 w2 = make_float2(wb, wb);
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float2 r = ffma2(w2, make_float2(code_at<B>(w, h, i), code_at<B>(w, h, i + 1)),
                                 make_float2(st.acc[i], st.acc[i + 1]));
          st.acc[i] = r.x;
          st.acc[i + 1] = r.y;
        }
        st.zacc = fmaf(p, sz.y, st.zacc);
      }
    }
  }
}

// -------------------------------------------------------------------- kernel --

constexpr int kSlots = 8;          // pages a warp may have in flight (one mbarrier each)
constexpr int kItemsPerWarp = 3;   // splits are made small enough for about this many
                                   // items per warp (never below the cache's pos_split)

struct AttnKernelArgs {
  LayerArgs a;
  int n;                       // queries of the call
  const int32_t* seq_ids;
  const int32_t* q_positions;
  const uint8_t* modes;
  const int32_t* windows;      // per-query windows, or null: window_scalar
  int window_scalar;
  const uint16_t* q;
  uint16_t* out;
  float qscale;      // softmax scale * log2(e)
  int ring_bytes;    // bytes of one warp's ring of shared memory
};

// Error of a query's arguments, 0 when it is valid.
__device__ __forceinline__ int query_error(const LayerArgs& a, int seq, int t, int mode, int w) {
  if (seq < 0 || seq >= a.S || mode > TRR_MODE_FULL) return TRR_ERR_INVALID_ARG;
  if (t < 0 || t >= a.maxctx) return TRR_ERR_BAD_POSITION;
  if (mode == TRR_MODE_LOCAL && w < 1) return TRR_ERR_INVALID_ARG;
  return 0;
}

// Key positions in range (Eq. 2): full [0, t]; local the last w positions up to t.
__device__ __forceinline__ int query_range(int t, int mode, int w) {
  return mode == TRR_MODE_FULL ? t + 1 : mode == TRR_MODE_LOCAL ? min(w, t + 1) : 0;
}

// Per-page record the producer writes for the consumer: meta = class | fill << 2 |
// mask << 9 | flags << 10 (1 first, 2 last, 4 no page) | item entry << 13, the ring
// offset of the page's slice (then its positions when masked, then the query row on the
// first page of an item) and the ring bytes to release after the page.  The item's own
// fields sit once in the warp's item table (kItemSlots entries of 8 words: lo, hi, item,
// query, head, splits, unit of split 0, KV head); an entry is rewritten only after every
// record of its previous item has been consumed (at most kSlots records are in flight).
constexpr int kItemSlots = 8;
static_assert(kItemSlots >= kSlots, "an item entry outlives the records in flight");

// Shared-memory carve-up of one attention CTA; every region starts 16-byte aligned
// (mbarriers need 8, bulk-copy destinations 16).
__host__ __device__ constexpr int align16(int x) { return (x + 15) & ~15; }
constexpr int kWarpWords = kItemSlots * 8 + 8;  // per-warp shared words: item table, merge
struct AttnSmem {
  int rings, recs, bars, words, pre, red, total;
  __host__ __device__ AttnSmem(int nwarps, int ring_bytes, int n)
      : rings(0),
        recs(align16(nwarps * ring_bytes)),
        bars(recs + align16(nwarps * kSlots * 16)),
        words(bars + align16(nwarps * kSlots * 8)),
        pre(words + nwarps * kWarpWords * 4),
        red(pre + align16(4 * (n + 1))),
        total(red + 16 * 8) {}
};

// The plan of one work item as the producer needs it: lane j holds page j's id and meta
// in registers; the item's fields sit in the warp's shared words (written by lane 0):
// [0] lo [1] hi [2] item [3] query [4] query head [5] splits [6] unit of split 0 [7] KV head.
template <int D>
__device__ __forceinline__ int plan_next_item(const AttnKernelArgs& ka, const int* pre, int n, int wstride, int lane,
                                           int* next_item, int* wplan, int& wid, int& wmeta, int& kvh) {
  const LayerArgs& a = ka.a;
  const int total = pre[n] * a.Hq;
  while (*next_item < total) {
    const int i = *next_item;
    *next_item += wstride;
    const int u = i / a.Hq, h = i - u * a.Hq;
    int lo_q = 0, hi_q = n;  // the query of unit u: pre[q] <= u < pre[q + 1]
    while (hi_q - lo_q > 1) {
      const int mid = (lo_q + hi_q) >> 1;
      if (pre[mid] <= u) lo_q = mid;
      else hi_q = mid;
    }
    const int q = lo_q, sp = u - pre[q], ns = pre[q + 1] - pre[q];
    const int seq = ka.seq_ids[q], t = ka.q_positions[q], mode = ka.modes[q];
    const int w = ka.windows ? ka.windows[q] : ka.window_scalar;
    const int err = query_error(a, seq, t, mode, w);
    if (err || mode == TRR_MODE_SKIP) {  // a zero row; the error of the lowest query
      uint4* o = reinterpret_cast<uint4*>(ka.out + (static_cast<int64_t>(q) * a.Hq + h) * D);
      if (lane < D / 8) o[lane] = make_uint4(0, 0, 0, 0);
      if (err && h == 0 && lane == 0) atomicMin(&a.ctrl[kFirstBadQuery], q * 16 + err);
      continue;
    }
    const int lo = mode == TRR_MODE_FULL ? 0 : max(0, t - w + 1);
    // per class: pages ending before lo, pages starting at or before t
    int nt[kClasses];
#pragma unroll
    for (int c = 0; c < kClasses; ++c) nt[c] = a.ntok[seq * 4 + c];
    const bool upper_mask = t < a.last_pos[seq];  // keys after t may be stored
    int pages[kClasses], first[kClasses], end[kClasses];
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      pages[c] = (nt[c] + a.P - 1) / a.P;
      first[c] = 0;
      end[c] = pages[c];
    }
    const int64_t row0 = static_cast<int64_t>(seq) * 4 * a.MP;
    // a window's pages are almost always among the last 32 of each class: their ids are
    // loaded together with the search's first probes
    int tb[kClasses], ptail[kClasses];
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      tb[c] = max(0, pages[c] - 32);
      ptail[c] = (lo > 0 && tb[c] + lane < pages[c]) ? a.pt[row0 + c * a.MP + tb[c] + lane] : -1;
    }
    if (lo > 0) warp_count_below<kClasses>(a.plast + row0, a.MP, pages, lo, first, lane);
    if (upper_mask) warp_count_below<kClasses>(a.pfirst + row0, a.MP, pages, t + 1, end, lane);
    // this split's share of each class's pages in range, then one page per lane
    // split sp of ns takes np / ns pages of the class, one more when sp < np % ns
    int beg[kClasses], tc[kClasses], npr[kClasses];
    int T = 0;
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      npr[c] = max(0, end[c] - first[c]);
      const unsigned each = static_cast<unsigned>(npr[c]) / static_cast<unsigned>(ns);
      const int extra = npr[c] - static_cast<int>(each) * ns;
      beg[c] = first[c] + sp * static_cast<int>(each) + min(sp, extra);
      tc[c] = static_cast<int>(each) + (sp < extra ? 1 : 0);
      T += tc[c];
    }
    T = min(T, kItemMaxPages + kClasses);  // the split bound keeps T within this
    wid = -1;
    wmeta = 0;
    const int t1 = tc[0], t2 = t1 + tc[1], t3 = t2 + tc[2];
    const int c = (lane >= t1) + (lane >= t2) + (lane >= t3);
    auto pick = [c](const int (&v)[kClasses]) { return c == 0 ? v[0] : c == 1 ? v[1] : c == 2 ? v[2] : v[3]; };
    const int kid = pick(beg) + lane - (c == 0 ? 0 : c == 1 ? t1 : c == 2 ? t2 : t3);
    int from_tail = -1;
#pragma unroll
    for (int cc = 0; cc < kClasses; ++cc) {
      const int v = __shfl_sync(0xffffffffu, ptail[cc], (kid - tb[cc]) & 31);
      if (c == cc && kid >= tb[cc]) from_tail = v;
    }
    if (lane < T) {
      const int f = pick(first);
      wid = from_tail >= 0 ? from_tail : a.pt[static_cast<int64_t>(seq * 4 + c) * a.MP + kid];
      const int fill = min(a.P, pick(nt) - kid * a.P);
      // slot positions are needed on a page that may hold keys outside [lo, t]
      const bool mask = (lo > 0 && kid == f) || (upper_mask && kid == f + pick(npr) - 1);
      wmeta = c | (fill << 2) | (mask ? 512 : 0);
    }
    kvh = h / (a.Hq / a.Hkv);
    if (lane == 0) {
      reinterpret_cast<int4*>(wplan)[0] = make_int4(lo, t, i, q);
      reinterpret_cast<int4*>(wplan)[1] = make_int4(h, ns, pre[q], kvh);
    }
    __syncwarp();
    return T;
  }
  return -1;
}

template <int D, int P>
__global__ void __launch_bounds__(256, 2) attn_kernel(const __grid_constant__ AttnKernelArgs ka) {
  constexpr int LPK = D / 32;  // lanes per key
  constexpr int KPI = 32 / LPK;  // keys per warp iteration
  constexpr int DPL = D / 32;  // dimensions per lane after the merge
  const LayerArgs& a = ka.a;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int n = ka.n;
  const int qrow = D * 2;  // bytes of one query row
  const int R = ka.ring_bytes;
  const AttnSmem lay(nwarps, R, n);  // [rings][slot records][mbarriers][unit prefix][scratch]
  uint8_t* ring = smem + lay.rings + warp * R;
  int4* recs = reinterpret_cast<int4*>(smem + lay.recs) + warp * kSlots;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + lay.bars) + warp * kSlots;
  int* pre = reinterpret_cast<int*>(smem + lay.pre);
  int* witems = reinterpret_cast<int*>(smem + lay.words) + warp * kWarpWords;  // item table
  int* wmerge = witems + kItemSlots * 8;
  long long* red = reinterpret_cast<long long*>(smem + lay.red);

  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kSlots; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
  }
  pdl_wait();
  pdl_trigger();

  // ---------------------------------------------------------- work units --
  // Every CTA computes the same split of the call: query q gets ns_q splits from its key
  // range; pre[q] numbers its first unit, pre[n] counts them all.
  long long rsum = 0;
  for (int q = threadIdx.x; q < n; q += blockDim.x) {
    const int seq = ka.seq_ids[q], t = ka.q_positions[q], mode = ka.modes[q];
    const int w = ka.windows ? ka.windows[q] : ka.window_scalar;
    const int r = query_error(a, seq, t, mode, w) ? 0 : query_range(t, mode, w);
    pre[q] = r;
    rsum += r;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
  if (lane == 0) red[warp] = rsum;
  __syncthreads();
  rsum = 0;
  for (int k = 0; k < nwarps; ++k) rsum += red[k];
  // splits small enough for about kItemsPerWarp items per warp, never below pos_split
  // (binary32 arithmetic: the same result in every CTA, and it only sizes the splits)
  const float want = static_cast<float>(gridDim.x * nwarps * kItemsPerWarp);
  const float by_work = ceilf(static_cast<float>(rsum) * static_cast<float>(a.Hq) / want);
  const int pos_split = by_work > static_cast<float>(a.pos_split) ? static_cast<int>(fminf(by_work, 1073741824.f))
                                                                   : a.pos_split;
  {
    const int chunk = (n + blockDim.x - 1) / blockDim.x;
    const int q0 = min(n, static_cast<int>(threadIdx.x) * chunk), q1 = min(n, q0 + chunk);
    int mine = 0;
    for (int q = q0; q < q1; ++q) mine += splits_of(pre[q], pos_split, a.P, a.s_cap);
    int incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    __syncthreads();  // every read of red above is done
    if (lane == 31) red[8 + warp] = incl;
    __syncthreads();
    int off = incl - mine;
    for (int k = 0; k < warp; ++k) off += static_cast<int>(red[8 + k]);
    for (int q = q0; q < q1; ++q) {
      const int ns = splits_of(pre[q], pos_split, a.P, a.s_cap);
      pre[q] = off;
      off += ns;
    }
    if (threadIdx.x == blockDim.x - 1) pre[n] = off;
    __syncthreads();
  }
  const int wstride = gridDim.x * nwarps;

  // ------------------------------------------------------------ producer --
  // Items are dealt round-robin; consecutive warps take consecutive heads of one unit,
  // so the planning loads of a unit mostly hit in L1.
  int next_item = blockIdx.x * nwarps + warp;
  int wid = -1, wmeta = 0;             // the producer's item: page id / meta of page `lane`
  int p_T = 0;                         // pages of the producer's item
  int p_kvh = 0;                       // its KV head
  int pf = 0;                          // next page of the producer's item
  bool pvalid = false;
  uint32_t issued = 0, consumed = 0;   // pages issued / consumed by this warp
  uint32_t started = 0;                // items started by this warp (item table index)
  int head = 0, used = 0;              // ring: next free offset, bytes held

  auto start_item = [&]() -> bool {
    p_T = plan_next_item<D>(ka, pre, n, wstride, lane, &next_item, witems + (started % kItemSlots) * 8, wid,
                            wmeta, p_kvh);
    pf = 0;
    if (p_T < 0) return false;
    ++started;
    return true;
  };
  // start the copies of the producer's next page if a slot and ring space are free
  auto try_issue = [&]() -> bool {
    if (issued - consumed >= kSlots) return false;  // first: an item entry is reused only
                                                    // once fewer records are in flight
    if (!pvalid) {
      pvalid = start_item();
      if (!pvalid) return false;
    }
    const bool first = pf == 0;
    int meta = 0, id = -1, bytes_page = 0;
    if (p_T > 0) {
      id = __shfl_sync(0xffffffffu, wid, pf);
      meta = __shfl_sync(0xffffffffu, wmeta, pf);
      bytes_page = a.slice[meta & 3] + ((meta & 512) ? 4 * P : 0);
    }
    const int need = bytes_page + (first ? qrow : 0);
    if (used == 0) head = 0;  // an empty ring can start anywhere
    int off = head, waste = 0;
    if (off + need > R) {
      waste = R - off;
      off = 0;
    }
    if (used + waste + need > R) return false;
    head = off + need;
    used += waste + need;
    const uint32_t slot = issued % kSlots;
    const int flags = (first ? 1 : 0) | (pf + 1 >= p_T ? 2 : 0) | (p_T == 0 ? 4 : 0);
    // The record, then the arrival.  The ring is written only by bulk copies; the warp's
    // earlier reads of these bytes have completed (their values were consumed), and the
    // record reaches the consumer through the mbarrier's release / acquire, so no proxy
    // fence is needed here.
    if (lane == 0) {
      const int entry = (started - 1) % kItemSlots;
      recs[slot] = make_int4(meta | (flags << 10) | (entry << 13), off, waste + need, 0);
      mbar_arrive_expect_tx(&bars[slot], need);
      const int c = meta & 3;
      if (p_T > 0) {
        const uint8_t* page = a.pool[c] + static_cast<int64_t>(id) * a.page_bytes[c];
        bulk_g2s(ring + off, page + a.hdr + static_cast<int64_t>(p_kvh) * a.slice[c], a.slice[c], &bars[slot]);
        if (meta & 512) bulk_g2s(ring + off + a.slice[c], page, 4 * P, &bars[slot]);
      }
      if (first) {
        const int* it = witems + entry * 8;
        bulk_g2s(ring + off + bytes_page, ka.q + (static_cast<int64_t>(it[3]) * a.Hq + it[4]) * D, qrow, &bars[slot]);
      }
    }
    __syncwarp();
    ++issued;
    ++pf;
    if (pf >= p_T) pvalid = false;
    return true;
  };

  // ------------------------------------------------------------ consumer --
  const int part = lane % LPK, kl = lane / LPK;
  LaneState st;
  float qp[32];
  float sumq = 0.f;
  int cur_cls = 3;
  st.m = kNegInf;
  st.l = 0.f;
  st.zacc = 0.f;
  // The merge of an item's lanes and splits, once its last page is consumed.
  bool merge_pending = false;
  auto merge_item = [&]() {
    const int4 mr = reinterpret_cast<const int4*>(wmerge)[0];  // item, query, head, splits
    const int m_item = mr.x, m_qi = mr.y, m_qh = mr.z, m_nsplit = mr.w, m_base = wmerge[4];
    // merge the lanes that share a part.  Rescale to the common maximum, then
    // reduce-scatter over the key lanes: each halving step keeps half of the 32 dims
    // and sends the other half to the partner lane.
    acc_to_neutral(st.acc, cur_cls);
    float M = st.m;
#pragma unroll
    for (int o = LPK; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float f = (st.m == kNegInf) ? 0.f : fast_exp2(st.m - M);
    float L = st.l * f;
#pragma unroll
    for (int o = LPK; o < 32; o <<= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
    {
      const float2 s49 = make_float2(pow2f(49) * f, pow2f(49) * f), zf = make_float2(st.zacc * f, st.zacc * f);
#pragma unroll
      for (int j = 0; j < 32; j += 2) {
        const float2 r = __ffma2_rn(make_float2(st.acc[j], st.acc[j + 1]), s49, zf);
        st.acc[j] = r.x;
        st.acc[j + 1] = r.y;
      }
    }
#pragma unroll
    for (int width = 16, o = 16; o >= LPK; width >>= 1, o >>= 1) {
      const bool upper = lane & o;
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (i < width) {
          const float keep = upper ? st.acc[width + i] : st.acc[i];
          const float give = upper ? st.acc[i] : st.acc[width + i];
          st.acc[i] = keep + __shfl_xor_sync(0xffffffffu, give, o);
        }
      }
    }
    // lane (kl, part) now holds dims part*32 + DPL*kl .. + DPL-1 in acc[0 .. DPL-1]
    const int dim0 = part * 32 + DPL * kl;
    const int64_t orow = (static_cast<int64_t>(m_qi) * a.Hq + m_qh) * D;
    if (m_nsplit == 1) {
      const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
      for (int j = 0; j < DPL; j += 2)
        *reinterpret_cast<__nv_bfloat162*>(ka.out + orow + dim0 + j) =
            __floats2bfloat162_rn(st.acc[j] * inv, st.acc[j + 1] * inv);
      return;
    }
    // a partial at the item's index; the last split of (query, head) to arrive merges
    float* pp = a.part + static_cast<int64_t>(m_item) * (D + 4);
#pragma unroll
    for (int j = 0; j < DPL; j += 2)
      *reinterpret_cast<float2*>(pp + dim0 + j) = make_float2(st.acc[j], st.acc[j + 1]);
    if (lane == 0) *reinterpret_cast<float2*>(pp + D) = make_float2(M, L);
    // the warp's partial stores happen before lane 0's release; the last arriver's
    // acquire happens before its lanes read the other splits' partials
    __syncwarp();
    int arrivals = 0;
    int* counter = a.cnt + static_cast<int64_t>(m_qi) * a.Hq + m_qh;
    if (lane == 0) arrivals = atom_add_acq_rel(counter, 1);
    __syncwarp();
    arrivals = __shfl_sync(0xffffffffu, arrivals, 0);
    if (arrivals != m_nsplit - 1) return;
    const float* p0 = a.part + (static_cast<int64_t>(m_base) * a.Hq + m_qh) * (D + 4);
    const int64_t sstride = static_cast<int64_t>(a.Hq) * (D + 4);
    float Mx = kNegInf;
    for (int s = lane; s < m_nsplit; s += 32) Mx = fmaxf(Mx, __ldcg(p0 + s * sstride + D));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) Mx = fmaxf(Mx, __shfl_xor_sync(0xffffffffu, Mx, o));
    float Ls = 0.f, acc_o[DPL];
#pragma unroll
    for (int j = 0; j < DPL; ++j) acc_o[j] = 0.f;
#pragma unroll 4
    for (int s = 0; s < m_nsplit; ++s) {
      const float* ps = p0 + s * sstride;
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(ps + D));
      const float wgt = (ml.x == kNegInf) ? 0.f : fast_exp2(ml.x - Mx);
      Ls = fmaf(wgt, ml.y, Ls);
#pragma unroll
      for (int j = 0; j < DPL; ++j) acc_o[j] = fmaf(wgt, __ldcg(ps + lane * DPL + j), acc_o[j]);
    }
    const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
    for (int j = 0; j < DPL; j += 2)
      *reinterpret_cast<__nv_bfloat162*>(ka.out + orow + lane * DPL + j) =
          __floats2bfloat162_rn(acc_o[j] * inv, acc_o[j + 1] * inv);
    if (lane == 0) *counter = 0;  // ready for the next call
  };

  for (;;) {
    // refill first, so that the next item's copies fly while this one merges; the one
    // place the producer plans items
    while (try_issue()) {
    }
    if (merge_pending) {
      merge_pending = false;
      merge_item();
    }
    if (consumed == issued) break;
    const uint32_t g = consumed;
    const uint32_t slot = g % kSlots;
    const bool arrived = mbar_wait(&bars[slot], (g / kSlots) & 1);
    if (!__all_sync(0xffffffffu, arrived)) {  // give up together, never half a warp
      for (uint32_t r = g + 1; r < issued; ++r) mbar_wait(&bars[r % kSlots], (r / kSlots) & 1);
      if (lane == 0) set_status(a.ctrl, TRR_ERR_TIMEOUT);
      break;
    }
    const int4 r0 = recs[slot];
    const int meta = r0.x, flags = (meta >> 10) & 7;
    const int* item_words = witems + (meta >> 13) * 8;  // lo, hi, item, query, head, splits, base
    if (flags & 1) {  // first page of an item: query row and a fresh state
      const int qoff = r0.y + ((flags & 4) ? 0 : a.slice[meta & 3] + ((meta & 512) ? 4 * P : 0));
      const uint32_t qa = smem_u32(ring + qoff + part * 64);
      const float2 qs2 = make_float2(ka.qscale, ka.qscale);
      float2 sq2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 u = lds128(qa + 16 * q);
        const uint32_t wv[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const float2 r = __fmul2_rn(make_float2(bf_lo(wv[h]), bf_hi(wv[h])), qs2);
          qp[8 * q + 2 * h] = r.x;
          qp[8 * q + 2 * h + 1] = r.y;
          sq2 = __fadd2_rn(sq2, r);
        }
      }
      sumq = sq2.x + sq2.y;
      cur_cls = 3;  // the neutral scale is class 16's
      st.m = kNegInf;
      st.l = 0.f;
      st.zacc = 0.f;
#pragma unroll
      for (int j = 0; j < 32; ++j) st.acc[j] = 0.f;
    }
    if (!(flags & 4)) {
      const int cls = meta & 3, fill = (meta >> 2) & 127;
      if (cls != cur_cls) {
        rescale_dyn(qp, st.acc, cur_cls, cls);
        cur_cls = cls;
      }
      const uint32_t s0 = smem_u32(ring + r0.y);
      const uint32_t sp = s0 + a.slice[cls];  // slot positions, on masked pages
      const bool masked = meta & 512;
      const int c_lo = item_words[0], c_hi = item_words[1];  // key range
      switch (cls) {
        case 0: consume_page<D, 2, P / KPI>(s0, sp, masked, a.G, fill, c_lo, c_hi, qp, sumq, st, lane); break;
        case 1: consume_page<D, 4, P / KPI>(s0, sp, masked, a.G, fill, c_lo, c_hi, qp, sumq, st, lane); break;
        case 2: consume_page<D, 8, P / KPI>(s0, sp, masked, a.G, fill, c_lo, c_hi, qp, sumq, st, lane); break;
        default: consume_page<D, 16, P / KPI>(s0, sp, masked, a.G, fill, c_lo, c_hi, qp, sumq, st, lane); break;
      }
    }
    if (flags & 2) {  // last page of the item: its merge follows the refill
      if (lane == 0) {
        reinterpret_cast<int4*>(wmerge)[0] = make_int4(item_words[2], item_words[3], item_words[4], item_words[5]);
        wmerge[4] = item_words[6];
      }
      merge_pending = true;
    }
    __syncwarp();
    used -= r0.z;  // release the slot's ring bytes (the record is read)
    consumed = g + 1;
  }

  // The last CTA to finish records the error of the lowest failing query.
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&a.ctrl[kDoneCtas], 1) == static_cast<int>(gridDim.x) - 1) {
      __threadfence();
      const int bad = atomicExch(&a.ctrl[kFirstBadQuery], INT_MAX);
      if (bad != INT_MAX) set_status(a.ctrl, bad & 15);
      atomicExch(&a.ctrl[kDoneCtas], 0);
    }
  }
}

constexpr int kAttnSmemLimit = 113 * 1024;  // dynamic shared memory of one attention CTA

// Done once per cache at creation, so that calls stay legal inside stream capture.
cudaError_t attn_configure() {
  const void* kernels[] = {
      reinterpret_cast<const void*>(attn_kernel<64, 16>), reinterpret_cast<const void*>(attn_kernel<64, 32>),
      reinterpret_cast<const void*>(attn_kernel<64, 64>), reinterpret_cast<const void*>(attn_kernel<128, 16>),
      reinterpret_cast<const void*>(attn_kernel<128, 32>), reinterpret_cast<const void*>(attn_kernel<128, 64>)};
  for (const void* k : kernels) {
    const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmemLimit);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// The one launch of an attention call with the given scratch views in `a`.
static cudaError_t launch_attention(const Layout& l, const LayerArgs& a, int num_sms, int n,
                                    const int32_t* seq_ids, const int32_t* q_positions, const void* q_bf16,
                                    const uint8_t* modes, const int32_t* windows, int window_scalar,
                                    float softmax_scale, void* out_bf16, cudaStream_t s) {
  AttnKernelArgs ka;
  ka.a = a;
  ka.n = n;
  ka.seq_ids = seq_ids;
  ka.q_positions = q_positions;
  ka.modes = modes;
  ka.windows = windows;
  ka.window_scalar = window_scalar;
  ka.q = static_cast<const uint16_t*>(q_bf16);
  ka.out = static_cast<uint16_t*>(out_bf16);
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.f / sqrtf(static_cast<float>(l.d));
  ka.qscale = scale * 1.4426950408889634f;
  // a ring holds at least one page of the widest class with its positions and a query
  // row; up to 12 KB when shared memory allows
  const int widest = (static_cast<int>(l.slice[3]) + 4 * l.P + 2 * l.d + 127) / 128 * 128;
  int nwarps = 8, ring = 0;
  for (; nwarps > 0; --nwarps) {
    const int fixed = AttnSmem(nwarps, 0, n).total;
    ring = std::min(std::max(12 * 1024, widest), (kAttnSmemLimit - fixed) / nwarps / 128 * 128);
    if (ring >= widest) break;
  }
  if (nwarps < 1) return cudaErrorInvalidConfiguration;
  ka.ring_bytes = ring;
  const int smem = AttnSmem(nwarps, ring, n).total;
  // one kernel per head size and page size: the page loop unrolls, and a kernel's code
  // holds only the four width classes it can meet
  const dim3 grid(2 * num_sms), block(nwarps * 32);
  const size_t sm = static_cast<size_t>(smem);
  if (l.d == 64) {
    if (l.P == 16) return launch_pdl(attn_kernel<64, 16>, grid, block, sm, s, ka);
    if (l.P == 32) return launch_pdl(attn_kernel<64, 32>, grid, block, sm, s, ka);
    return launch_pdl(attn_kernel<64, 64>, grid, block, sm, s, ka);
  }
  if (l.P == 16) return launch_pdl(attn_kernel<128, 16>, grid, block, sm, s, ka);
  if (l.P == 32) return launch_pdl(attn_kernel<128, 32>, grid, block, sm, s, ka);
  return launch_pdl(attn_kernel<128, 64>, grid, block, sm, s, ka);
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
  const LayerArgs a = layer_args(l, cache_views(cache), layer);
  const cudaError_t e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, q_positions, q_bf16, modes,
                                         windows, window_scalar, softmax_scale, out_bf16,
                                         static_cast<cudaStream_t>(stream));
  cache_set_launches(cache, 1);
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

// Clears what a call needs at zero: the control words and the arrival counters.
__global__ void static_scratch_clear_kernel(int32_t* wctrl, int32_t* cnt, int ncnt) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < kCtrlInts) wctrl[i] = i == kFirstBadQuery ? INT_MAX : 0;
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
  const int64_t b_cnt = up(4ll * n * l.units);
  const int64_t b_part = up(4ll * n * l.s_cap * l.units * (l.d + 4));
  if (b_ctrl + b_cnt + b_part > kStaticScratchBytes) return TRR_ERR_OUT_OF_MEMORY;
  void* base = nullptr;
  if (static_scratch(&base) != cudaSuccess) return TRR_ERR_CUDA;
  uint8_t* b = static_cast<uint8_t*>(base);
  LayerArgs a = layer_args(l, cache_views(cache), layer);
  int32_t* cache_ctrl = a.ctrl;
  a.ctrl = reinterpret_cast<int32_t*>(b);
  a.cnt = reinterpret_cast<int32_t*>(b + b_ctrl);
  a.part = reinterpret_cast<float*>(b + b_ctrl + b_cnt);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int ncnt = n * l.units;
  static_scratch_clear_kernel<<<std::max(1, std::min(256, (ncnt + 255) / 256)), 256, 0, s>>>(a.ctrl, a.cnt, ncnt);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess)
    e = launch_attention(l, a, cache_num_sms(cache), n, seq_ids, q_positions, q_bf16, modes, windows,
                         window_scalar, softmax_scale, out_bf16, s);
  if (e != cudaSuccess) return TRR_ERR_CUDA;
  static_scratch_status_kernel<<<1, 1, 0, s>>>(a.ctrl, cache_ctrl);
  cache_set_launches(cache, 3);
  return cudaGetLastError() == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}
