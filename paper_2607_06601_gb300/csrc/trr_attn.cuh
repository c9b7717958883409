#pragma once
// trr_attn.cuh - the attention kernels of trr_decode_attn and trr_decode_step: mode-routed
// split-K decode attention over the mixed-precision paged cache (Sec. 3.2(A), Eq. 2; Sec. 3.8; Sec. 7).
//
// One persistent kernel per call: three CTAs per SM, each one producer warp and four
// consumer warps around a ring of shared memory.
//   1. Every CTA cuts the call into work units: query q gets ns_q splits from the
//      length of its key range (full: [0, t]; local: [t-w+1, t]; skip or invalid: one
//      split that writes the zero rows), and a unit is a split and a block of query
//      heads.  The same deterministic computation in every CTA takes the place of a
//      planning kernel.  Splits are sized for about one unit per CTA on a small call
//      and up to three on a large one.
//   2. The producer warp takes units (on a small call from a call-wide counter as its
//      CTA starts and finishes them; on a large one its CTA's own first, then from the
//      counter) and plans each once: the sequence's per-class token counts, a 32-way
//      search of the pages' first / last positions at window edges, the split's share
//      of every class's pages in range.  It pushes the unit through the ring as stages
//      filled by 1-D bulk copies (cp.async.bulk + mbarrier): the block's query rows,
//      then per page the slices of the KV heads the block reads (slot positions too
//      when the page straddles the key range).
//   3. Consumer warps read the stages in order and release each one.  Two consumers:
//        - CUDA cores (one query head per warp; MHA and wide query groups): lane pair
//          (key, half) of a 64-wide head (four lanes for 128) dequantises in registers
//          and keeps its own online softmax; lanes merge with shuffles;
//        - tensor cores (one KV head and its whole query group per warp, g >= 2 with
//          g * d/G <= 8): q.k and P.V as mma.sync m16n8k16 with f32 accumulation.
//   4. A query with one split gets its bf16 rows from that unit.  Otherwise each split
//      writes fp32 partials; partials merge in two levels (groups of kMergeGroup, then
//      the groups), each by the last arrival, which resets its counter.
//   5. The last CTA to finish records the error of the lowest failing query.
//
// Per-head modes (a cache with head_modes): the query's widest head mode sizes its
// splits; a unit reads the pages of its head block's widest mode (a block of local and
// skip heads only its window's splits); every slice of a page ends with its KV head's
// presence mask, which the consumer applies per key; pages before the window come only
// for the KV heads a full head of the block reads; a skip head writes its zero row.
//
// CUDA-core dequantisation: k = z + c*s, so q.k = s * sum(q_i c_i) + z * sum(q_i).  A
// code is masked in place (no shift) and its bits read as a binary32 subnormal,
// c * 2^(e-149) where e is its bit offset; the query is pre-scaled per width class by
// 2^(100-e) so that q_i * x_i = q_i c_i 2^-49 exactly as an fp32 product.  V is
// accumulated in a domain scaled by 2^-49 with the per-offset factor folded into the
// key's weight.
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

// Bit offset of element i (of a lane's 16 or 32) inside the word it is extracted from.
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

// The words' high parts (codes past the binary32 mantissa, shifted down); NW words.
template <int B, int NW>
__device__ __forceinline__ void high_parts(const uint32_t* w, uint32_t* h) {
  constexpr int sh = B == 2 ? 22 : B == 4 ? 20 : 16;
#pragma unroll
  for (int k = 0; k < NW; ++k) h[k] = w[k] >> sh;
}

// x *= f on pairs of fp32 lanes (packed multiply)
__device__ __forceinline__ void fmul2_inplace(float& x0, float& x1, float f0, float f1) {
  const float2 r = __fmul2_rn(make_float2(x0, x1), make_float2(f0, f1));
  x0 = r.x;
  x1 = r.y;
}

// 2^x with the hardware approximation (relative error about 2^-22; results below the
// binary32 normal range flush to zero, far below a softmax sum's resolution).
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int E>
struct LaneState {
  float m, l, zacc;  // running max (log2), sum of weights, sum of p*z (V zero points)
  float acc[E];      // sum of p*v over the lane's E dims, scaled by 2^-49
};

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
__device__ __forceinline__ int4 lds128i(uint32_t a) {
  int4 v;
  asm volatile("ld.shared.v4.s32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
__device__ __forceinline__ void sts32(uint32_t a, uint32_t v) {
  asm volatile("st.shared.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
  return v;
}

// The factors that move a lane's query and V accumulators between the domains of two
// width classes, element by element (E = 32 elements per lane): row from * 4 + to.  One
// table read by every class change keeps a single copy of the code in the consumer's
// loop (a switch over templated copies made the loop several kilobytes larger).  Each
// CTA of the CUDA-core kernels writes the table into its shared memory before the wait
// on the previous kernel, and a class change reads its row with warp-wide broadcast
// loads (from constant memory, whose cache misses, a switch took about 470 cycles).
struct RescaleTable {
  float q[16][32];    // query: 2^(qe(to, i) - qe(from, i))
  float acc[16][32];  // V accumulators: 2^(ex(to, i) - ex(from, i)), ex = 0 at width 16
};
constexpr int kRescaleFloats = static_cast<int>(sizeof(RescaleTable) / 4);

// Entry k of the table (k < kRescaleFloats), as the struct lays it out.
__device__ __forceinline__ float rescale_entry(int k) {
  const bool is_acc = k >= 16 * 32;
  const int row = (k >> 5) & 15, i = k & 31, bf = bits_of_class(row >> 2), bt = bits_of_class(row & 3);
  const int e = is_acc ? (bt == 16 ? 0 : ex_of(bt, i)) - (bf == 16 ? 0 : ex_of(bf, i)) : qe_of(bt, i) - qe_of(bf, i);
  return pow2f(e);
}

// qp and acc from the domain of class `from` to that of class `to`; tbl: the table's
// shared-memory address.
template <int E>
__device__ __forceinline__ void rescale_dyn(float (&qp)[E], float (&acc)[E], int from, int to, uint32_t tbl) {
  static_assert(E == 32, "one factor per element of a lane's 32");
  const uint32_t qf = tbl + (from * 4 + to) * 128, af = qf + 16 * 32 * 4;
#pragma unroll
  for (int i = 0; i < E; i += 4) {
    const uint4 fq = lds128(qf + 4 * i), fa = lds128(af + 4 * i);
    fmul2_inplace(qp[i], qp[i + 1], __uint_as_float(fq.x), __uint_as_float(fq.y));
    fmul2_inplace(qp[i + 2], qp[i + 3], __uint_as_float(fq.z), __uint_as_float(fq.w));
    fmul2_inplace(acc[i], acc[i + 1], __uint_as_float(fa.x), __uint_as_float(fa.y));
    fmul2_inplace(acc[i + 2], acc[i + 3], __uint_as_float(fa.z), __uint_as_float(fa.w));
  }
}
// acc from class `from`'s domain back to class 16's (the common one of the merge)
template <int E>
__device__ __forceinline__ void acc_to_neutral(float (&acc)[E], int from, uint32_t tbl) {
  const uint32_t af = tbl + 16 * 32 * 4 + (from * 4 + 3) * 128;
#pragma unroll
  for (int i = 0; i < E; i += 4) {
    const uint4 fa = lds128(af + 4 * i);
    fmul2_inplace(acc[i], acc[i + 1], __uint_as_float(fa.x), __uint_as_float(fa.y));
    fmul2_inplace(acc[i + 2], acc[i + 3], __uint_as_float(fa.z), __uint_as_float(fa.w));
  }
}


// The NW words of a lane's codes at shared address a (4 NW-byte aligned), in as few
// loads as possible (one 4-, 8- or 16-byte load per row part keeps the warp's request
// conflict-free).
template <int NW>
__device__ __forceinline__ void lds_codes(uint32_t a, uint32_t* w) {
  if (NW == 1) {
    w[0] = lds32(a);
  } else if (NW == 2) {
    const uint2 u = lds64(a);
    w[0] = u.x; w[1] = u.y;
  } else {
#pragma unroll
    for (int k = 0; k < NW; k += 4) {
      const uint4 u = lds128(a + 4 * k);
      w[k] = u.x; w[k + 1] = u.y; w[k + 2] = u.z; w[k + 3] = u.w;
    }
  }
}

// One page of width class B (P = NIT * keys per iteration tokens) at shared address s0;
// lane -> (key kl, 32-dim part).  Keys past `fill` are empty slots; with positions at
// spos (masked pages), keys outside [lo, hi] are masked too.
// A lane's q-th 16-byte chunk of a key's 8- or 16-bit row in a swizzled slice: the row
// part it reads starts at chunk c0 of its 128-byte line, whose chunks are stored in the
// order chunk ^ xm (xm: the line's index mod 8; see swz_off).
__device__ __forceinline__ uint32_t swz_chunk(uint32_t a, int c0, int xm, int q) {
  return a + static_cast<uint32_t>((((c0 + q) ^ xm) - c0) * 16);
}

// q.k of one key at shared address ka (this lane's E dims) in class B, with its (s, z)
// word at kszaddr for B < 16: s * sum(q_i c_i) + z * sum(q_i) in the domain of qp.
template <int B, int E>
__device__ __forceinline__ float k_dot(uint32_t ka, uint32_t kszaddr, const float (&qp)[E], float sumq, int c0, int xm) {
  float2 d2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  if (B == 16) {
#pragma unroll
    for (int q = 0; q < E / 8; ++q) {
      const uint4 u = lds128(swz_chunk(ka, c0, xm, q));
      d2[0] = ffma2(make_float2(qp[8 * q + 0], qp[8 * q + 1]), make_float2(bf_lo(u.x), bf_hi(u.x)), d2[0]);
      d2[1] = ffma2(make_float2(qp[8 * q + 2], qp[8 * q + 3]), make_float2(bf_lo(u.y), bf_hi(u.y)), d2[1]);
      d2[0] = ffma2(make_float2(qp[8 * q + 4], qp[8 * q + 5]), make_float2(bf_lo(u.z), bf_hi(u.z)), d2[0]);
      d2[1] = ffma2(make_float2(qp[8 * q + 6], qp[8 * q + 7]), make_float2(bf_lo(u.w), bf_hi(u.w)), d2[1]);
    }
    return (d2[0].x + d2[0].y) + (d2[1].x + d2[1].y);
  }
  constexpr int NW = E * B / 32;
  uint32_t w[NW], h[NW];
  if (B == 8) {  // two chunks of the swizzled row
#pragma unroll
    for (int q = 0; q < NW / 4; ++q) {
      const uint4 u = lds128(swz_chunk(ka, c0, xm, q));
      w[4 * q] = u.x; w[4 * q + 1] = u.y; w[4 * q + 2] = u.z; w[4 * q + 3] = u.w;
    }
  } else {
    lds_codes<NW>(ka, w);
  }
  if (B != 8) high_parts<B, NW>(w, h);
  const uint32_t szw = lds32(kszaddr);
#pragma unroll
  for (int i = 0; i < E / 2; ++i)
    d2[i & 1] = ffma2(make_float2(qp[2 * i], qp[2 * i + 1]),
                      make_float2(code_at<B>(w, h, 2 * i), code_at<B>(w, h, 2 * i + 1)), d2[i & 1]);
  const float2 sz = __half22float2(*reinterpret_cast<const __half2*>(&szw));  // (s, z)
  return fmaf(sz.x * pow2f(49), (d2[0].x + d2[0].y) + (d2[1].x + d2[1].y), sz.y * sumq);
}

// acc += p * v for one key's V at shared address va (this lane's E dims) in class B,
// with its (s, z) word at vszaddr for B < 16.
template <int B, int E>
__device__ __forceinline__ void v_acc(uint32_t va, uint32_t vszaddr, float p, LaneState<E>& st, int c0, int xm) {
  if (B == 16) {
    const float wv = p * pow2f(-49);
    const float2 w2 = make_float2(wv, wv);
#pragma unroll
    for (int q = 0; q < E / 8; ++q) {
      const uint4 u = lds128(swz_chunk(va, c0, xm, q));
      const uint32_t uw[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const int i = 8 * q + 2 * h;
        const float2 r = ffma2(w2, make_float2(bf_lo(uw[h]), bf_hi(uw[h])), make_float2(st.acc[i], st.acc[i + 1]));
        st.acc[i] = r.x;
        st.acc[i + 1] = r.y;
      }
    }
    return;
  }
  constexpr int NW = E * B / 32;
  uint32_t w[NW], h[NW];
  if (B == 8) {  // two chunks of the swizzled row
#pragma unroll
    for (int q = 0; q < NW / 4; ++q) {
      const uint4 u = lds128(swz_chunk(va, c0, xm, q));
      w[4 * q] = u.x; w[4 * q + 1] = u.y; w[4 * q + 2] = u.z; w[4 * q + 3] = u.w;
    }
  } else {
    lds_codes<NW>(va, w);
  }
  if (B != 8) high_parts<B, NW>(w, h);
  const uint32_t szw = lds32(vszaddr);
  const float2 sz = __half22float2(*reinterpret_cast<const __half2*>(&szw));  // (s, z)
  const float wb = p * sz.x * pow2f(100);
  const float2 w2 = make_float2(wb, wb);
#pragma unroll
  for (int i = 0; i < E; i += 2) {
    const float2 r = ffma2(w2, make_float2(code_at<B>(w, h, i), code_at<B>(w, h, i + 1)),
                           make_float2(st.acc[i], st.acc[i + 1]));
    st.acc[i] = r.x;
    st.acc[i + 1] = r.y;
  }
  st.zacc = fmaf(p, sz.y, st.zacc);
}

// One page of width class B (P = NIT * keys per iteration tokens) at shared address s0;
// lane -> (key kl, E-dim part), and two keys per lane per iteration (kl and kl + KPI)
// when NIT is even, so that their dependency chains overlap.  Keys past `fill` are
// empty slots; with positions at spos (masked pages), keys outside [lo, hi] are masked,
// and with HM (per-head modes) the slots whose bit in pm is clear (the token does not
// store this KV head).
template <int D, int B, int NIT, int E, bool HM>
__device__ __forceinline__ void consume_page(uint32_t s0, uint32_t spos, bool masked, uint64_t pm, int G, int fill,
                                             int lo, int hi, const float (&qp)[E], float sumq, LaneState<E>& st,
                                             int lane) {
  constexpr int LPK = D / E;
  constexpr int KPI = 32 / LPK;
  constexpr int P = NIT * KPI;
  constexpr int KP = 1;  // keys per lane per iteration (one: half the code of two, which the
                         // instruction cache favours over the second key's overlap)
  constexpr int rowb = B == 16 ? 2 * D : D * B / 8;  // bytes of one key's row of K (or V)
  const int part = lane % LPK, kl = lane / LPK;
  const int lg = __ffs(G) - 1;  // G is a power of two: shifts, not divisions
  const int ng = D >> lg;
  const int grp = (part * E) >> lg;
  const uint32_t krow = s0 + kl * rowb + part * (E * B / 8);   // this lane's K bytes, key kl
  // 8- and 16-bit rows are swizzled (every cache of this consumer): the lane's first chunk
  // in its line and the line's index mod 8 (the same for every key it reads, as a key
  // group spans a multiple of 8 lines, and for the V rows, which start on such a line)
  const int o0 = kl * rowb + part * (E * B / 8);
  const int c0 = (o0 >> 4) & 7, xm = B >= 8 ? (o0 >> 7) & 7 : 0;
  const uint32_t ksz = s0 + 2 * P * rowb + (kl * ng + grp) * 4;  // its (s, z), key kl
  const uint32_t szstep = KPI * ng * 4;
#pragma unroll 1
  for (int it = 0; it < NIT && it * KPI < fill; it += KP) {  // key groups past the fill hold nothing
    bool valid[KP];
    float dot[KP];
#pragma unroll
    for (int k = 0; k < KP; ++k) {
      const int key = (it + k) * KPI + kl;
      valid[k] = key < fill;
      if (HM) valid[k] = valid[k] && ((pm >> key) & 1ull);
      if (masked) {
        const int pos = static_cast<int>(lds32(spos + 4 * key));
        valid[k] = valid[k] && pos >= lo && pos <= hi;
      }
      dot[k] = k_dot<B, E>(krow + (it + k) * KPI * rowb, ksz + (it + k) * szstep, qp, sumq, c0, xm);
    }
#pragma unroll
    for (int k = 0; k < KP; ++k) {
#pragma unroll
      for (int o = 1; o < LPK; o <<= 1) dot[k] += __shfl_xor_sync(0xffffffffu, dot[k], o);
    }
    // online softmax over the lane's keys: one lazy rescale for both
    float top = kNegInf;
#pragma unroll
    for (int k = 0; k < KP; ++k)
      if (valid[k]) top = fmaxf(top, dot[k]);
    if (top > st.m + kTau) {
      const float alpha = fast_exp2(st.m - top);  // 0 when m = -inf
#pragma unroll
      for (int j = 0; j < E; ++j) st.acc[j] *= alpha;
      st.l *= alpha;
      st.zacc *= alpha;
      st.m = top;
    }
#pragma unroll
    for (int k = 0; k < KP; ++k) {
      if (valid[k]) {
        const float p = fast_exp2(dot[k] - st.m);
        st.l += p;
        const uint32_t va = krow + (it + k) * KPI * rowb + P * rowb;
        v_acc<B, E>(va, ksz + (it + k) * szstep + P * ng * 4, p, st, c0, xm);
      }
    }
  }
}

// -------------------------------------------------------------------- kernel --
//
// One CTA = one producer warp + kNcw consumer warps.  A work unit is (query, split,
// block of query heads).  The producer plans each unit once (the key range, every
// class's pages in range, the split's share) and streams it through the CTA's ring of
// shared memory as stages: the unit's query rows, then for every page the slices of
// the KV heads the block reads, with the page's slot positions when the page straddles
// the key range.  Consumers read the stages in order and release each one.

constexpr int kNcw = 4;           // consumer warps per CTA
constexpr int kStages = 16;       // stage records a CTA may have in flight
constexpr int kUnitsPerCta = 3;   // units per CTA of a large call, at most
constexpr float kMinUnitPositions = 512.f;  // key positions of a large call's unit, at least
constexpr int kCtasPerSm = 3;     // CTAs per SM
constexpr int kMmaCtasPerSm = 3;  // CTAs per SM of the tensor-core kernels

// Dims per lane of the CUDA-core consumer (E = 16 would use four lanes per key at d = 64
// and half the registers, but it issues twice the instructions per key), and its CTAs
// per SM.
__host__ __device__ constexpr int cc_elems(int) { return 32; }
__host__ __device__ constexpr int cc_ctas_per_sm(int) { return kCtasPerSm; }
// dynamic shared memory of one attention CTA with `ctas` CTAs per SM (228 KB per SM,
// 1 KB of it reserved per CTA)
__host__ __device__ constexpr int attn_smem_limit(int ctas) {
  return ctas >= 5 ? 44 * 1024 : ctas == 2 ? 110 * 1024 : 72 * 1024;
}

// Stage record, three int4 words written by the producer before it arrives on the
// stage's full barrier:
//   a = {meta, ring offset of the stage's bytes, query, lo}
//   b = {hi (= t), split, splits, unit number of split 0}
//   c = {first KV slice of the stage (block-relative), KV slices per page | pages of the
//        stage << 8, ring offset of the page's slot positions or -1, bytes of one KV
//        slice}; a stage of several pages holds full pages of one class, each page's
//        slices after the previous page's (the last page's fill is in meta); in a query-rows
//        stage {the block's head modes, 2 bits per head (per-head modes), the local
//        window's first position, -1, 0}
// meta = class | fill << 2 | flags | head block << 16.
// A decode step's new-token stage has c.z = kNewRows: it arrives with no bytes, and each
// consumer warp first writes its KV head's slot 0 into it (and into the cache's page).
enum : int {
  kMask = 1 << 9,     // the page may hold keys outside [lo, hi]: positions follow the slices
  kFirst = 1 << 10,   // first stage of a unit (its query rows)
  kLast = 1 << 11,    // last stage of a unit
  kNoPage = 1 << 12,  // the unit has no page in range
  kEnd = 1 << 13,     // no more units
  kQRows = 1 << 14,   // the stage holds the unit's query rows
  kEarly = 1 << 15    // per-head modes: the page ends before the local window
};

constexpr int kNewRows = -2;

struct AttnKernelArgs {
  LayerArgs a;
  int n;                       // queries of the call
  const int32_t* seq_ids;
  const int32_t* q_positions;
  const uint8_t* modes;        // per-query modes, or null: mode_logits
  const float* mode_logits;    // [n][3] router logits (skip, local, full), or null
  const int32_t* windows;      // per-query windows, or null: window_scalar
  int window_scalar;
  const uint16_t* q;
  uint16_t* out;
  float qscale;      // softmax scale * log2(e)
  int q0;            // index of the launch's first query in the call (error reports)
  int ring_bytes;    // bytes of the CTA's ring of shared memory
  int hpu;           // query heads per work unit
  int scr_floats;    // per-consumer-warp scratch (floats) of the tensor-core path
  int defer_merge;   // 1: split partials are merged by the combine kernel (tensor-core path)
  int early;         // 1: the layer's cache state may be read before the previous kernel ends
  int fused;         // 1: a decode step: entry i appends its token (k, v, bits), then query i
                     // attends at the same position with the same mode
  const uint16_t* k;      // fused: K rows [n][Hkv][d] (bf16)
  const uint16_t* v;      // fused: V rows [n][Hkv][d] (bf16)
  const uint8_t* bits;    // fused: bit-widths [n]
};

// Fused decode step: the per-entry table every CTA builds in shared memory (2 ints per
// entry: the entry's token index in its (sequence, class) list, or -1 when it stores
// nothing; class | opens << 2 | openers of the class before it << 3), a hash of the
// entries' sequences (2 slots per entry: sequence + 1, lowest entry index; once the
// entries are checked, its first n ints hold the page of each token that goes into its
// class's last page), then the call's scalars.
constexpr int kStepMax = 256;  // entries of one decode-step call, at most
enum StepScalar : int {
  kSNextPage = 0,   // [4] pages handed out per class before the call (read after the wait)
  kSOpeners = 4,    // [4] entries opening a page, per class
  kSErr = 8,        // lowest failing entry * 16 + error, INT_MAX = none
  kSScalars = 16
};
__host__ __device__ constexpr int step_ints(int n) { return 2 * n + 4 * n + kSScalars; }

// Mode of query q: the caller's, or the hard decision of its mode logits.  With
// per-head modes (modes[n][Hq]) the largest of its heads' modes, which sets the query's
// key range (above full when a head's value is not a mode); any_local tells whether a
// head is local (its window must then be valid).
__device__ __forceinline__ int query_mode(const AttnKernelArgs& ka, int q, bool& any_local) {
  if (ka.mode_logits) {
    const int m = hard_decision<3>(ka.mode_logits + 3 * q);
    any_local = m == TRR_MODE_LOCAL;
    return m;
  }
  if (!ka.a.head_modes) {
    const int m = ka.modes[q];
    any_local = m == TRR_MODE_LOCAL;
    return m;
  }
  const uint8_t* row = ka.modes + static_cast<int64_t>(q) * ka.a.Hq;
  int m = 0;
  any_local = false;
  for (int h = 0; h < ka.a.Hq; ++h) {
    const int v = row[h];
    m = max(m, v);
    any_local |= v == TRR_MODE_LOCAL;
  }
  return m;
}

// Error of a query's arguments, 0 when it is valid.
__device__ __forceinline__ int query_error(const LayerArgs& a, int seq, int t, int mode, bool any_local, int w) {
  if (seq < 0 || seq >= a.S || mode > TRR_MODE_FULL) return TRR_ERR_INVALID_ARG;
  if (t < 0 || t >= a.maxctx) return TRR_ERR_BAD_POSITION;
  if (any_local && w < 1) return TRR_ERR_INVALID_ARG;
  return 0;
}

// Key positions in range (Eq. 2): full [0, t]; local the last w positions up to t.
__device__ __forceinline__ int query_range(int t, int mode, int w) {
  return mode == TRR_MODE_FULL ? t + 1 : mode == TRR_MODE_LOCAL ? min(w, t + 1) : 0;
}

// Shared-memory carve-up of one attention CTA; every region starts 16-byte aligned
// (mbarriers need 8, bulk-copy destinations 16).
__host__ __device__ constexpr int align16(int x) { return (x + 15) & ~15; }
struct AttnSmem {
  int ring, recs, sbytes, full, empty, scr, pre, ent, red, resc, flag, total;
  __host__ __device__ AttnSmem(int ring_bytes, int n, int scr_floats, int fused)
      : ring(0),
        recs(align16(ring_bytes)),
        sbytes(recs + kStages * 48),
        full(sbytes + align16(kStages * 4)),
        empty(full + kStages * 8),
        scr(empty + kStages * 8),
        pre(scr + align16(kNcw * scr_floats * 4)),
        ent(pre + align16(4 * (n + 2))),
        red(ent + (fused ? align16(4 * step_ints(n)) : 0)),
        resc(red + 16 * 8),  // the class-change factors (CUDA-core consumers, which have no scratch)
        flag(resc + (scr_floats == 0 ? 4 * kRescaleFloats : 0)),  // the abort flag; at flag + 8
                                                                    // the entry table's readiness mbarrier
        total(flag + 16) {}
};

// Bounded wait (limit_ns on the global timer) that also gives up once *abort is set (by
// a warp that gave up).
__device__ __forceinline__ bool mbar_wait_or(uint64_t* bar, uint32_t parity, volatile int* abort, uint64_t limit_ns) {
  const uint32_t addr = smem_u32(bar), aaddr = smem_u32(const_cast<int*>(abort));
  if (mbar_poll(addr, parity, limit_ns)) return true;
  const uint64_t t0 = global_ns();
  for (;;) {
    if (mbar_poll(addr, parity, limit_ns)) return true;
    if (lds32(aaddr)) return false;
    if (global_ns() - t0 >= limit_ns) return false;
  }
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Whether phase `parity` of `bar` has completed, without waiting.
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// Pages of split sp (of ns) of a query of sequence seq over key positions [lo, t]:
// returns their number T (<= kItemMaxPages + 4); lane j < T gets page j's id in wid,
// class | fill << 2 | kMask in wmeta and, when wfirst / wlast are given, the page's first
// and last positions.  Pages are listed class by class, each class's in
// position order; split sp of ns takes np / ns of a class's np pages in range, one more
// when sp < np % ns.
__device__ __forceinline__ int plan_split(const LayerArgs& a, int P, int seq, int lo, int t, int sp, int ns,
                                          int lane, int& wid, int& wmeta, int* wfirst = nullptr,
                                          int* wlast = nullptr) {
  int nt[kClasses];
#pragma unroll
  for (int c = 0; c < kClasses; ++c) nt[c] = a.ntok[seq * 4 + c];
  const bool upper_mask = t < a.last_pos[seq];  // keys after t may be stored
  int pages[kClasses], first[kClasses], end[kClasses];
#pragma unroll
  for (int c = 0; c < kClasses; ++c) {
    pages[c] = (nt[c] + P - 1) / P;
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
    ptail[c] = tb[c] + lane < pages[c] ? a.pt[row0 + c * a.MP + tb[c] + lane] : -1;
  }
  if (lo > 0) warp_count_below<kClasses>(a.plast + row0, a.MP, pages, lo, first, lane);
  if (upper_mask) warp_count_below<kClasses>(a.pfirst + row0, a.MP, pages, t + 1, end, lane);
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
  // lanes take the pages class by class from the widest (bf16) down: the largest copies
  // are issued first, while the ring is empty (before the wait on the previous kernel),
  // and the small ones stream in behind them as the consumers free the ring
  const int t1 = tc[3], t2 = t1 + tc[2], t3 = t2 + tc[1];
  const int r = (lane >= t1) + (lane >= t2) + (lane >= t3);  // rank in that order
  const int c = 3 - r;
  auto pick = [c](const int (&v)[kClasses]) { return c == 0 ? v[0] : c == 1 ? v[1] : c == 2 ? v[2] : v[3]; };
  const int kid = pick(beg) + lane - (r == 0 ? 0 : r == 1 ? t1 : r == 2 ? t2 : t3);
  int from_tail = -1;
#pragma unroll
  for (int cc = 0; cc < kClasses; ++cc) {
    const int v = __shfl_sync(0xffffffffu, ptail[cc], (kid - tb[cc]) & 31);
    if (c == cc && kid >= tb[cc]) from_tail = v;
  }
  if (lane < T) {
    const int f = pick(first);
    wid = from_tail >= 0 ? from_tail : a.pt[static_cast<int64_t>(seq * 4 + c) * a.MP + kid];
    if (wfirst) {  // the page's first and last positions
      *wfirst = a.pfirst[static_cast<int64_t>(seq * 4 + c) * a.MP + kid];
      *wlast = a.plast[static_cast<int64_t>(seq * 4 + c) * a.MP + kid];
    }
    const int fill = min(P, pick(nt) - kid * P);
    // slot positions are needed on a page that may hold keys outside [lo, t]
    const bool mask = (lo > 0 && kid == f) || (upper_mask && kid == f + pick(npr) - 1);
    wmeta = c | (fill << 2) | (mask ? kMask : 0);
  }
  return T;
}

// Key positions that query q's head blocks read in all (r: its widest head's range):
// NQB times r, or with per-head modes each block its own widest head's range, the heads
// assigned to blocks as the producer assigns them (ranked by mode when Hq <= 32, in index
// order otherwise).  It sizes the splits only.
__device__ __forceinline__ long long query_block_work(const AttnKernelArgs& ka, int q, int t, int w, int r,
                                                      int NQB) {
  const LayerArgs& a = ka.a;
  if (!a.head_modes || ka.mode_logits || r == 0) return static_cast<long long>(r) * NQB;
  const uint8_t* row = ka.modes + static_cast<int64_t>(q) * a.Hq;
  if (a.Hq <= 32) {
    int nf = 0, nl = 0;
    for (int h = 0; h < a.Hq; ++h) {
      nf += row[h] == TRR_MODE_FULL;
      nl += row[h] == TRR_MODE_LOCAL;
    }
    const int bf = (nf + ka.hpu - 1) / ka.hpu;               // blocks holding a full head
    const int bl = (nf + nl + ka.hpu - 1) / ka.hpu - bf;     // blocks led by a local head
    return static_cast<long long>(bf) * query_range(t, TRR_MODE_FULL, w) +
           (bl > 0 ? static_cast<long long>(bl) * query_range(t, TRR_MODE_LOCAL, w) : 0ll);
  }
  long long s = 0;
  for (int h0 = 0; h0 < a.Hq; h0 += ka.hpu) {
    int m = 0;
    for (int h = h0; h < min(a.Hq, h0 + ka.hpu); ++h) m = max(m, static_cast<int>(row[h]));
    s += query_range(t, m, w);
  }
  return s;
}

// The work units of a call, computed the same way by every CTA: query q gets ns_q
// splits from its key range (per-head modes: its widest head's); pre[q] numbers its
// first split, pre[n] counts them all, pre[n + 1] is the call's key positions per split.
__device__ __forceinline__ void plan_units(const AttnKernelArgs& ka, int P, int NQB, int* pre, long long* red) {
  const LayerArgs& a = ka.a;
  const int n = ka.n, lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  long long rsum = 0;
  for (int q = threadIdx.x; q < n; q += blockDim.x) {
    bool any_local;
    const int seq = ka.seq_ids[q], t = ka.q_positions[q], mode = query_mode(ka, q, any_local);
    const int w = ka.windows ? ka.windows[q] : ka.window_scalar;
    const int r = query_error(a, seq, t, mode, any_local, w) ? 0 : query_range(t, mode, w);
    pre[q] = r;
    rsum += query_block_work(ka, q, t, w, r, NQB);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
  if (lane == 0) red[warp] = rsum;
  __syncthreads();
  rsum = 0;
  for (int k = 0; k < nwarps; ++k) rsum += red[k];
  // Split size: a small call gets about one unit per CTA (its units are latency-bound
  // chains, and a second unit on a CTA doubles the call); a large one up to
  // kUnitsPerCta per CTA, each of at least kMinUnitPositions positions per head block
  // (the producer plans the next unit while the consumers work on this one); never
  // below pos_split.  The work counts each head block's own range, so that per-head
  // modes, whose blocks past the full heads read only a window or nothing, size their
  // units by the blocks that read pages.  Binary32 arithmetic: the same result in every
  // CTA, and it only sizes the splits.
  const float ctas = static_cast<float>(gridDim.x);
  const float rs = static_cast<float>(rsum);
  const float want = fmaxf(0.8f * ctas, fminf(static_cast<float>(kUnitsPerCta) * ctas, rs / kMinUnitPositions));
  const float by_work = ceilf(rs / want);
  const int pos_split = by_work > static_cast<float>(a.pos_split) ? static_cast<int>(fminf(by_work, 1073741824.f))
                                                                   : a.pos_split;
  const int chunk = (n + blockDim.x - 1) / blockDim.x;
  const int q0 = min(n, static_cast<int>(threadIdx.x) * chunk), q1 = min(n, q0 + chunk);
  int mine = 0;
  for (int q = q0; q < q1; ++q) {  // pre[q] becomes the query's split count
    const int ns = splits_of(pre[q], pos_split, P, a.s_cap);
    pre[q] = ns;
    mine += ns;
  }
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
    const int ns = pre[q];
    pre[q] = off;
    off += ns;
  }
  if (threadIdx.x == blockDim.x - 1) {
    pre[n] = off;
    pre[n + 1] = pos_split;  // for per-block split counts (per-head modes)
  }
  __syncthreads();
}

// ------------------------------------------------------------ decode step --
//
// A decode-step call (trr_decode_step) appends entry i's token (Sec. 3.2(C), Eq. 4: K and
// V stored at the entry's bit-width; nothing for a skip token unless skip tokens store
// KV) and attends with query i at the same position in the same mode (Eq. 2), in one
// kernel.  The attention reads the cache as the call finds it and takes each query's own
// new token from a stage the producer fills in shared memory; the token's bytes are
// written to its slot in the page; the last CTA to finish commits the metadata.  The
// entries name distinct sequences (one token per sequence).

__device__ __forceinline__ unsigned seq_hash(int seq, int slots) {
  return (static_cast<unsigned>(seq) * 2654435761u) % static_cast<unsigned>(slots);
}

// Every CTA: validates the entries and plans where each token goes (the same plan as the
// append kernels: the token takes index ntok of its (sequence, class) list; index % P == 0
// opens a page, whose id is next_page + the class's openers before it).  Errors, lowest
// entry first: sequence id, bit-width or mode not allowed, or a sequence named by an
// earlier entry (INVALID_ARG); position outside [0, max_context) or not above the
// sequence's last one (BAD_POSITION); a local query with a window below 1 (INVALID_ARG).
// Run by the kNcw consumer warps (threads 32 .. 32 * (kNcw + 1) - 1) while the producer
// plans its first unit; they synchronise among themselves on named barrier 1.
__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(32 * kNcw) : "memory");
}
static __device__ void plan_entries(const AttnKernelArgs& ka, int* ent) {
  const LayerArgs& a = ka.a;
  const int n = ka.n, tid = threadIdx.x - 32, nt = 32 * kNcw, H = 2 * n;
  int* hs = ent + 2 * n;  // [H][2]: sequence + 1, lowest entry index naming it
  int* sc = ent + 6 * n;
  for (int i = tid; i < 2 * H; i += nt) hs[i] = (i & 1) ? INT_MAX : 0;
  for (int i = tid; i < kSScalars; i += nt) sc[i] = i == kSErr ? INT_MAX : 0;
  consumers_sync();
  for (int e = tid; e < n; e += nt) {
    const int seq = ka.seq_ids[e];
    if (seq < 0 || seq >= a.S) continue;
    unsigned h = seq_hash(seq, H);
    for (int probe = 0; probe < H; ++probe) {
      const int old = atomicCAS(&hs[2 * h], 0, seq + 1);
      if (old == 0 || old == seq + 1) {
        atomicMin(&hs[2 * h + 1], e);
        break;
      }
      h = h + 1 == static_cast<unsigned>(H) ? 0u : h + 1;
    }
  }
  consumers_sync();
  int lp[(kStepMax + 32 * kNcw - 1) / (32 * kNcw)];  // page of each of this thread's tokens
                                                        // that goes into its class's last page
#pragma unroll
  for (int k = 0; k < (kStepMax + 32 * kNcw - 1) / (32 * kNcw); ++k) lp[k] = -1;
  for (int e = tid, k = 0; e < n; e += nt, ++k) {
    const int seq = ka.seq_ids[e], pos = ka.q_positions[e], m = ka.modes[e], b = ka.bits[e];
    const int c = b == 2 ? 0 : b == 4 ? 1 : b == 8 ? 2 : b == 16 ? 3 : -1;
    const int w = ka.windows ? ka.windows[e] : ka.window_scalar;
    int err = 0;
    if (seq < 0 || seq >= a.S || c < 0 || m > TRR_MODE_FULL) {
      err = TRR_ERR_INVALID_ARG;
    } else if (pos < 0 || pos >= a.maxctx) {
      err = TRR_ERR_BAD_POSITION;
    } else {
      unsigned h = seq_hash(seq, H);
      for (int probe = 0; probe < H && hs[2 * h] != seq + 1; ++probe) h = h + 1 == static_cast<unsigned>(H) ? 0u : h + 1;
      if (hs[2 * h + 1] != e) err = TRR_ERR_INVALID_ARG;
      else if (pos <= a.last_pos[seq]) err = TRR_ERR_BAD_POSITION;
      else if (m == TRR_MODE_LOCAL && w < 1) err = TRR_ERR_INVALID_ARG;
    }
    int tok = -1, info = 0;
    if (!err && (m != TRR_MODE_SKIP || a.skip_writes_kv)) {
      tok = a.ntok[seq * 4 + c];
      info = c | (tok % a.P == 0 ? 4 : 0);
      if (tok % a.P != 0) {
#pragma unroll
        for (int kk = 0; kk < (kStepMax + 32 * kNcw - 1) / (32 * kNcw); ++kk)
          if (kk == k) lp[kk] = a.lastpg[seq * 4 + c];
      }
    }
    ent[2 * e] = tok;
    ent[2 * e + 1] = info;
    if (err) atomicMin(&sc[kSErr], e * 16 + err);
  }
  consumers_sync();  // the hash is read no more: its first n ints take the last pages
  for (int e = tid, k = 0; e < n; e += nt, ++k) {
#pragma unroll
    for (int kk = 0; kk < (kStepMax + 32 * kNcw - 1) / (32 * kNcw); ++kk)
      if (kk == k) hs[e] = lp[kk];
  }
  if (tid < 32) {  // openers of the same class before each entry, 32 entries at a time
    int run0 = 0, run1 = 0, run2 = 0, run3 = 0;
    for (int e0 = 0; e0 < n; e0 += 32) {
      const int e = e0 + tid;
      const int tok = e < n ? ent[2 * e] : -1, info = e < n ? ent[2 * e + 1] : 0;
      const bool op = tok >= 0 && (info & 4);
      const int c = info & 3;
      const unsigned below = (1u << tid) - 1u;
      const unsigned b0 = __ballot_sync(0xffffffffu, op && c == 0), b1 = __ballot_sync(0xffffffffu, op && c == 1);
      const unsigned b2 = __ballot_sync(0xffffffffu, op && c == 2), b3 = __ballot_sync(0xffffffffu, op && c == 3);
      const int before = c == 0 ? run0 + __popc(b0 & below) : c == 1 ? run1 + __popc(b1 & below)
                       : c == 2 ? run2 + __popc(b2 & below) : run3 + __popc(b3 & below);
      if (e < n) ent[2 * e + 1] = info | ((op ? before : 0) << 3);
      run0 += __popc(b0); run1 += __popc(b1); run2 += __popc(b2); run3 += __popc(b3);
    }
    if (tid < 4) sc[kSOpeners + tid] = tid == 0 ? run0 : tid == 1 ? run1 : tid == 2 ? run2 : run3;
  }
  consumers_sync();
}

// One warp, after the wait on the previous kernel: the pools' page counters, and the
// first opener beyond its pool's capacity (OUT_OF_PAGES) as a call error.
__device__ __forceinline__ void step_after_wait(const AttnKernelArgs& ka, int* ent, int lane) {
  const LayerArgs& a = ka.a;
  const int n = ka.n;
  int* sc = ent + 6 * n;
  if (lane < 4) sc[kSNextPage + lane] = a.ctrl[kNextPage + lane];
  __syncwarp();
  for (int e = lane; e < n; e += 32) {
    const int tok = ent[2 * e], info = ent[2 * e + 1], c = info & 3;
    if (tok >= 0 && (info & 4) && sc[kSNextPage + c] + (info >> 3) >= a.cap[c])
      atomicMin(&sc[kSErr], e * 16 + TRR_ERR_OUT_OF_PAGES);
  }
  __syncwarp();
}

// Page and slot of entry e's token (an entry that stores KV).
__device__ __forceinline__ void step_slot(const AttnKernelArgs& ka, const int* ent, int e, int& c, int& pid,
                                          int& slot) {
  const LayerArgs& a = ka.a;
  const int tok = ent[2 * e], info = ent[2 * e + 1];
  const int* sc = ent + 6 * ka.n;
  c = info & 3;
  slot = tok % a.P;
  pid = (info & 4) ? sc[kSNextPage + c] + (info >> 3) : ent[2 * ka.n + e];  // the class's last page
}

// Entry e's K and V rows of up to 4 KV heads kv0 .. kv0 + nkv - 1, this lane's D/32
// values of each (loaded together: one round trip).
template <int D>
__device__ __forceinline__ void step_load_rows(const AttnKernelArgs& ka, int e, int kv0, int nkv, uint2 (&rk)[4],
                                               uint2 (&rv)[4], int lane) {
  const LayerArgs& a = ka.a;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    rk[k] = rv[k] = make_uint2(0, 0);
    if (k < nkv) {
      const int64_t src = (static_cast<int64_t>(e) * a.Hkv + kv0 + k) * D;
      if (D == 64) {
        rk[k].x = reinterpret_cast<const uint32_t*>(ka.k + src)[lane];
        rv[k].x = reinterpret_cast<const uint32_t*>(ka.v + src)[lane];
      } else {
        rk[k] = reinterpret_cast<const uint2*>(ka.k + src)[lane];
        rv[k] = reinterpret_cast<const uint2*>(ka.v + src)[lane];
      }
    }
  }
}

// One KV head j's K and V rows (rk, rv as step_load_rows holds them) at class c
// (Eq. 4, or the bf16 bits at width 16): written to the token's slot `slot` of page pid
// when `own`, and, when `to_ring`, to slot 0 of a page-shaped slice at shared address
// sdst (the stage consumers read).  Every lane of the warp calls it.
template <int D>
__device__ __forceinline__ void step_token_rows(const AttnKernelArgs& ka, uint2 rk, uint2 rv, int j, int c, int pid,
                                                int slot, bool own, uint32_t sdst, bool to_ring, int lane) {
  const LayerArgs& a = ka.a;
  const int P = a.P, b = bits_of_class(c), ng = D >> (__ffs(a.G) - 1);  // G: a power of two
  uint8_t* page = a.pool[c] + static_cast<int64_t>(pid) * a.page_bytes[c] + a.hdr + static_cast<int64_t>(j) * a.slice[c];
  // 8- and 16-bit code rows are swizzled in a cache of the CUDA-core consumer (swz_off,
  // relative to the slice: the page's slice, and the page-shaped slice at sdst that the
  // consumers read from the ring); a lane's 4 or 8 bytes stay inside one 16-byte chunk
  const bool sw = a.swz && b >= 8;
  auto pg = [&](int64_t o) -> uint8_t* { return page + (sw ? swz_off(o) : o); };
  auto rg = [&](int o) -> uint32_t { return sdst + static_cast<uint32_t>(sw ? swz_off(o) : o); };
  if (b == 16) {  // K [P][D] | V [P][D] bf16: this lane's D/32 values
    const int rowb = 2 * D;
    if (D == 64) {
      if (own) {
        *reinterpret_cast<uint32_t*>(pg(slot * rowb + 4 * lane)) = rk.x;
        *reinterpret_cast<uint32_t*>(pg((P + slot) * rowb + 4 * lane)) = rv.x;
      }
      if (to_ring) {
        sts32(rg(4 * lane), rk.x);
        sts32(rg(P * rowb + 4 * lane), rv.x);
      }
    } else {
      if (own) {
        *reinterpret_cast<uint2*>(pg(slot * rowb + 8 * lane)) = rk;
        *reinterpret_cast<uint2*>(pg((P + slot) * rowb + 8 * lane)) = rv;
      }
      if (to_ring) {
        sts32(rg(8 * lane), rk.x);
        sts32(rg(8 * lane) + 4, rk.y);
        sts32(rg(P * rowb + 8 * lane), rv.x);
        sts32(rg(P * rowb + 8 * lane) + 4, rv.y);
      }
    }
    return;
  }
  const int rowb = D * b / 8;
  // K, then V, through one copy of the quantiser (this code runs once per unit, so its
  // size, not its speed, decides: every instruction of it is a cold fetch)
  bool bad = false;
#pragma unroll 1
  for (int kv = 0; kv < 2; ++kv) {
    const RowCodes r = quantise_row_codes<D>(kv ? rv : rk, b, a.G, lane);
    bad |= r.bad;
    const int coff = (kv * P + slot) * rowb, soff = 2 * P * rowb + kv * P * ng * 4;
    if (own) {
      if (r.code_idx >= 0) *reinterpret_cast<uint32_t*>(pg(coff + 4 * r.code_idx)) = r.code_word;
      if (r.sz_idx >= 0) reinterpret_cast<uint32_t*>(page + soff + slot * ng * 4)[r.sz_idx] = r.sz_word;
    }
    if (to_ring) {
      if (r.code_idx >= 0) sts32(rg(kv * P * rowb + 4 * r.code_idx), r.code_word);
      if (r.sz_idx >= 0) sts32(sdst + soff + 4 * r.sz_idx, r.sz_word);
    }
  }
  if (__any_sync(0xffffffffu, bad) && lane == 0 && own) set_status(a.ctrl, TRR_ERR_BAD_VALUE);
}

// A consumer warp at the query rows of a unit that holds its query's new token (the
// query's last split): the token's K and V rows of KV head j into L1, one 128-byte line
// per lane, so that the new-token stage later finds them there.  The query-rows stage
// follows the producer's wait on the previous kernel (which wrote the rows).
template <int D>
__device__ __forceinline__ void step_prefetch_rows(const AttnKernelArgs& ka, int q, int j, int lane) {
  constexpr int kLines = D * 2 / 128;  // 128-byte lines of one row
  if (lane < 2 * kLines) {
    const uint16_t* src =
        ((lane & 1) ? ka.v : ka.k) + (static_cast<int64_t>(q) * ka.a.Hkv + j) * D + (lane >> 1) * 64;
    asm volatile("prefetch.global.L1 [%0];" ::"l"(src));
  }
}

// A consumer warp at a new-token stage: entry q's K and V rows of KV head j, quantised
// into the stage at shared address sdst (slot 0 of a page-shaped slice) and, when `own`,
// into the token's slot in the cache.  Writes of generic proxy to ring bytes that bulk
// copies later overwrite: fenced for the async proxy.
template <int D>
__device__ __forceinline__ void step_new_rows(const AttnKernelArgs& ka, const int* ent, int q, int j, bool own,
                                              uint32_t sdst, int lane) {
  int c, pid, slot;
  step_slot(ka, ent, q, c, pid, slot);
  uint2 rk[4], rv[4];
  step_load_rows<D>(ka, q, j, 1, rk, rv, lane);
  step_token_rows<D>(ka, rk[0], rv[0], j, c, pid, slot, own, sdst, true, lane);
  fence_proxy_async_smem();
  __syncwarp();
}

// The last CTA of a decode-step call: records the call's error, or commits every entry's
// metadata (page tables, page first / last positions, counts, the slot's position,
// presence, last positions, the pools' counters).  Nothing of the call's old metadata is
// read after this: every other CTA has finished.
static __device__ void step_commit(const AttnKernelArgs& ka, const int* ent) {
  const LayerArgs& a = ka.a;
  const int n = ka.n;
  const int* sc = ent + 6 * n;
  if (sc[kSErr] != INT_MAX) {
    if (threadIdx.x == 0) set_status(a.ctrl, sc[kSErr] & 15);
    return;
  }
  for (int e = threadIdx.x; e < n; e += blockDim.x) {
    const int seq = ka.seq_ids[e], pos = ka.q_positions[e], tok = ent[2 * e];
    if (tok >= 0) {
      int c, pid, slot;
      step_slot(ka, ent, e, c, pid, slot);
      const int64_t row = (static_cast<int64_t>(seq) * 4 + c) * a.MP + tok / a.P;
      if (ent[2 * e + 1] & 4) {
        a.pt[row] = pid;
        a.pfirst[row] = pos;
      }
      a.plast[row] = pos;
      a.ntok[seq * 4 + c] = tok + 1;
      a.lastpg[seq * 4 + c] = pid;
      reinterpret_cast<int32_t*>(a.pool[c] + static_cast<int64_t>(pid) * a.page_bytes[c])[slot] = pos;
      atomicOr(&a.presence[static_cast<int64_t>(seq) * a.W32 + pos / 32], 1u << (pos % 32));
    }
    a.last_pos[seq] = pos;
  }
  if (threadIdx.x < 4) a.ctrl[kNextPage + threadIdx.x] = sc[kSNextPage + threadIdx.x] + sc[kSOpeners + threadIdx.x];
}

// Everything the producer and consumers of one CTA share.
struct CtaRing {
  uint8_t* ring;
  int4* recs;
  int* sbytes;
  uint64_t* full;
  uint64_t* empty;
  volatile int* abort_flag;
  uint64_t* ent_ready;  // decode step: completes when the consumers have built the entry table
  uint32_t resc;        // shared address of the class-change factors (CUDA-core kernels)
  int R;
};

// The producer warp: takes units, plans each and pushes its stages; ends with an end
// record.
//
// With `early`, the first stages are planned and their page copies issued before the
// wait on the previous kernel (the layer's cache state is settled; the call's index
// arrays are its own): the unit's query-rows stage takes its slot first, and its record
// and copy follow the wait, so that consumers start only once the query rows (written
// by the previous kernel) are in.  Before the wait the producer takes ring space only
// where it is free, never waiting for consumers.  Nothing is written to global memory
// before the wait.
template <int D, bool STEP, bool HM>
__device__ __forceinline__ void run_producer(const AttnKernelArgs& ka, int P, int NQB, const int* pre, int* ent,
                                             const CtaRing& cr, int lane) {
  const LayerArgs& a = ka.a;
  const int n = ka.n, g = a.Hq / a.Hkv, R = cr.R;
  const int total = pre[n] * NQB;
  const int* sc = ent + 6 * n;        // decode step: the call's scalars
  uint32_t pushed = 0, released = 0;  // stages pushed / seen released by the consumers
  int rhead = 0, rused = 0;           // ring: next free offset, bytes held
  bool ok = true;
  bool waited = !(STEP && ka.early);
  // the query-rows stage waiting for the wait: its slot (-1: none), ring offset, records
  int dq_slot = -1, dq_off = 0, dq_need = 0;
  int4 dq_ra = make_int4(0, 0, 0, 0), dq_rb = dq_ra, dq_rc = dq_ra;
  const uint16_t* dq_src = nullptr;
  // decode step: the entry table the consumers build, waited for where it is first
  // needed (the producer plans its first unit meanwhile); then, after the wait on the
  // previous kernel, the pools' counters and whether a token runs out of pages (the call
  // then stores nothing, and the last CTA zeroes every row)
  bool have_ent = !STEP, have_pages = !STEP;
  auto ent_sync = [&]() {
    if (have_ent) return;
    have_ent = true;
    if (!mbar_wait(cr.ent_ready, 0, a.wait_ns)) {
      if (lane == 0) {
        *cr.abort_flag = 1;
        set_status(a.ctrl, TRR_ERR_TIMEOUT);
        atomicExch(&a.lctl[kAborted], 1);
      }
    }
  };
  // the call's error once known (a decode step with an error stores nothing and every
  // query gets its zero rows)
  auto call_failed = [&]() -> bool {
    if (!STEP) return false;
    ent_sync();
    return sc[kSErr] != INT_MAX;
  };
  // after the wait on the previous kernel: let the next kernel start, read what the
  // previous kernel wrote (decode step: the pools' counters; the combine kernel's query
  // table), then complete the deferred query-rows stage
  auto after_wait = [&]() {
    pdl_trigger();
    if (dq_slot >= 0) {
      if (lane == 0) {
        cr.recs[dq_slot * 3 + 0] = dq_ra;
        cr.recs[dq_slot * 3 + 1] = dq_rb;
        cr.recs[dq_slot * 3 + 2] = dq_rc;
        mbar_arrive_expect_tx(&cr.full[dq_slot], static_cast<uint32_t>(dq_need));
        bulk_g2s(cr.ring + dq_off, dq_src, dq_need, &cr.full[dq_slot]);
      }
      dq_slot = -1;
    }
    if (ka.defer_merge && blockIdx.x == 0) {  // for the combine kernel
      int2* qtab = reinterpret_cast<int2*>(a.cnt);
      for (int q = lane; q < n; q += 32) qtab[q] = make_int2(pre[q], pre[q + 1] - pre[q]);
    }
  };
  auto ensure_waited = [&]() {
    if (waited) return;
    pdl_wait();
    waited = true;
    after_wait();
  };
  auto pages_ready = [&]() {  // decode step: next_page and the out-of-pages check
    if (have_pages) return;
    have_pages = true;
    ensure_waited();
    ent_sync();
    step_after_wait(ka, ent, lane);
  };
  // wait for the oldest stage in flight to be released and take back its bytes
  auto release_one = [&]() -> bool {
    const uint32_t slot = released % kStages;
    if (!mbar_wait_or(&cr.empty[slot], (released / kStages) & 1, cr.abort_flag, a.wait_ns)) return false;
    rused -= static_cast<int>(lds32(smem_u32(cr.sbytes) + 4 * slot));
    ++released;
    return true;
  };
  // a slot and `need` contiguous ring bytes; -1 when a wait gave up; -2 when the space
  // is not free yet and `block` is false
  auto reserve = [&](int need, int& taken, bool block) -> int {
    for (;;) {
      if (pushed - released < static_cast<uint32_t>(kStages)) {
        if (rused == 0) rhead = 0;  // an empty ring can start anywhere
        int off = rhead, waste = 0;
        if (off + need > R) {
          waste = R - off;
          off = 0;
        }
        if (rused + waste + need <= R) {
          rhead = off + need;
          rused += waste + need;
          taken = waste + need;
          return off;
        }
      }
      if (pushed == released) return -1;
      if (!block) {  // take back released stages, without waiting for any
        const uint32_t slot = released % kStages;
        if (!mbar_test(&cr.empty[slot], (released / kStages) & 1)) return -2;
        rused -= static_cast<int>(lds32(smem_u32(cr.sbytes) + 4 * slot));
        ++released;
        continue;
      }
      if (!release_one()) return -1;
    }
  };
  // reserve before the wait where free, else wait on the previous kernel and block
  auto reserve_any = [&](int need, int& taken) -> int {
    int off = reserve(need, taken, waited);
    if (off == -2) {
      ensure_waited();
      off = reserve(need, taken, true);
    }
    return off;
  };
  // the record of the stage taking slot pushed % kStages, then its arrival with the
  // bytes its copies will bring (the copies follow, issued by lane 0)
  auto push = [&](int4 ra, int4 rb, int4 rc, int taken, int tx) -> uint32_t {
    const uint32_t slot = pushed % kStages;
    if (lane == 0) {
      cr.recs[slot * 3 + 0] = ra;
      cr.recs[slot * 3 + 1] = rb;
      cr.recs[slot * 3 + 2] = rc;
      cr.sbytes[slot] = taken;
      mbar_arrive_expect_tx(&cr.full[slot], static_cast<uint32_t>(tx));
    }
    ++pushed;
    return slot;
  };
  if (waited) after_wait();

  // A call with no more units than CTAs hands them out on demand from the call-wide
  // counter: a CTA takes its first unit as it starts and another only once its consumers
  // are done with the current one.  The CTAs that start last (on SM slots the previous
  // kernel frees as it ends) then get the last units, or none.  A larger call gives each
  // CTA its own first unit and lets the producer take the next from the counter once it
  // has pushed every stage of the current one, while the consumers still work on it: a
  // CTA whose unit turns out empty (a block of local or skip heads past its own splits)
  // or short asks again before the busy CTAs do, and takes the units they would have
  // queued.
  const bool on_demand = total <= static_cast<int>(gridDim.x);
  int u = static_cast<int>(blockIdx.x);
  if (on_demand) {
    if (lane == 0) u = atomicAdd(&a.lctl[kNextUnit], 1);
    u = __shfl_sync(0xffffffffu, u, 0);
  }
  while (u < total) {
    int u_next = 0;
    auto take_next = [&]() {
      if (lane == 0) u_next = (on_demand ? 0 : static_cast<int>(gridDim.x)) + atomicAdd(&a.lctl[kNextUnit], 1);
    };
    const int un = u / NQB, qb = u - un * NQB;
    int lo_q = 0, hi_q = n;  // the query of split un: pre[q] <= un < pre[q + 1]
    while (hi_q - lo_q > 1) {
      const int mid = (lo_q + hi_q) >> 1;
      if (pre[mid] <= un) lo_q = mid;
      else hi_q = mid;
    }
    const int q = lo_q, sp = un - pre[q];
    int ns = pre[q + 1] - pre[q];
    bool any_local;
    const int seq = ka.seq_ids[q], t = ka.q_positions[q], mode = query_mode(ka, q, any_local);
    const int w = ka.windows ? ka.windows[q] : ka.window_scalar;
    const int err = query_error(a, seq, t, mode, any_local, w);
    const int h0 = qb * ka.hpu, nh = min(ka.hpu, a.Hq - h0);
    // per-head modes: the block's own widest mode sets its key range, and its heads'
    // modes (2 bits each) travel in the query-rows record
    int bmode = mode, hpack = 0;
    const int kv0 = h0 / g, nkv = (h0 + nh - 1) / g - kv0 + 1;
    // the block's KV heads (bit k: kv0 + k) that a page must bring: every one, or with
    // per-head modes those read by a full head of the block (pages before the local
    // window) and those read by any head of the block (the other pages)
    unsigned need_full = (1u << nkv) - 1u, need_any = need_full;
    // per-head modes: the block's heads, slot s (a consumer warp) taking head hsel byte s.
    // With up to 32 query heads a query's heads are ranked by mode (full, local, skip;
    // by index within a mode) and block qb takes ranks qb * hpu .. + nh - 1, so that the
    // full heads share as few blocks as possible (a block reads the pages of its widest
    // mode); else (-1) slot s takes head h0 + s.  need_full / need_any are then masks of
    // slots, and a page brings one KV slice per slot that needs it.
    int hsel = -1;
    if (HM && !err) {
      if (a.Hq <= 32) {
        const int ml = lane < a.Hq ? ka.modes[static_cast<int64_t>(q) * a.Hq + lane] : TRR_MODE_FULL + 1;
        const int cl = ml == TRR_MODE_FULL ? 0 : ml == TRR_MODE_LOCAL ? 1 : ml == TRR_MODE_SKIP ? 2 : 3;
        const unsigned b0 = __ballot_sync(0xffffffffu, cl == 0), b1 = __ballot_sync(0xffffffffu, cl == 1);
        const unsigned b2 = __ballot_sync(0xffffffffu, cl == 2), lt = (1u << lane) - 1u;
        const int rank = cl == 0 ? __popc(b0 & lt)
                         : cl == 1 ? __popc(b0) + __popc(b1 & lt)
                         : cl == 2 ? __popc(b0) + __popc(b1) + __popc(b2 & lt) : 255;
        hsel = 0;
#pragma unroll
        for (int sl = 0; sl < kNcw; ++sl) {
          const unsigned hit = __ballot_sync(0xffffffffu, rank == h0 + sl);
          hsel |= (hit ? __ffs(hit) - 1 : 0) << (8 * sl);
        }
      }
      const int hs = hsel >= 0 ? (hsel >> (8 * (lane & 3))) & 255 : h0 + lane;  // lane < nh: slot lane's head
      const int hm = lane < nh ? ka.modes[static_cast<int64_t>(q) * a.Hq + hs] : 0;
      bmode = static_cast<int>(__reduce_max_sync(0xffffffffu, static_cast<unsigned>(hm)));
      hpack = static_cast<int>(__reduce_or_sync(0xffffffffu, static_cast<unsigned>(hm) << (2 * (lane & 15))));
      need_full = __ballot_sync(0xffffffffu, lane < nh && hm == TRR_MODE_FULL);
      need_any = __ballot_sync(0xffffffffu, lane < nh && hm != TRR_MODE_SKIP);
    }
    // the query head of slot s (per-head modes; s < nh)
    auto slot_head = [&](int sl) -> int { return hsel >= 0 ? (hsel >> (8 * sl)) & 255 : h0 + sl; };
    if (HM && !err && bmode == TRR_MODE_LOCAL) {
      // per-head modes, a block of local and skip heads in a query whose widest head is
      // full: the block's own split count, from its window; its splits past that have
      // nothing to do, and its heads merge that many partials
      ns = min(ns, splits_of(query_range(t, TRR_MODE_LOCAL, w), pre[n + 1], P, a.s_cap));
      if (sp >= ns) {
        __syncwarp();
        take_next();
        u = __shfl_sync(0xffffffffu, u_next, 0);
        continue;
      }
    }
    // decode step: this query's own token joins the last split of each head block
    const bool has_new = STEP && !err && bmode != TRR_MODE_SKIP && sp == ns - 1;
    // the unit's pages.  A decode step does not wait for its entry table here: a call
    // error makes the last CTA zero every row, so units run as if there were none and
    // only the new-token stage needs the table
    const int lo = bmode == TRR_MODE_FULL ? 0 : max(0, t - w + 1);
    int wid = -1, wmeta = 0, wfirst = 0, wlast = INT_MAX, T = 0;
    if (!err && bmode != TRR_MODE_SKIP)
      T = plan_split(a, P, seq, lo, t, sp, ns, lane, wid, wmeta, HM ? &wfirst : nullptr,
                     HM ? &wlast : nullptr);
    if (err || bmode == TRR_MODE_SKIP) {
      // zero rows (once per block); the error of the lowest query; a skip token that
      // stores KV has its rows written here
      ensure_waited();
      if (sp == 0) {
        for (int i = lane; i < nh * D / 8; i += 32) {  // slot i / (D / 8)'s row
          const int h = HM ? slot_head(i / (D / 8)) : h0 + i / (D / 8);
          reinterpret_cast<uint4*>(ka.out + (static_cast<int64_t>(q) * a.Hq + h) * D)[i % (D / 8)] =
              make_uint4(0, 0, 0, 0);
        }
      }
      if (!STEP && err && qb == 0 && lane == 0) atomicMin(&a.lctl[kFirstBadQuery], (ka.q0 + q) * 16 + err);
      if (STEP && !call_failed() && sp == 0 && ent[2 * q] >= 0) {
        pages_ready();
        int c, pid, slot;
        step_slot(ka, ent, q, c, pid, slot);
        for (int j0 = kv0; j0 < kv0 + nkv; j0 += 4) {
          const int m = min(4, kv0 + nkv - j0);
          uint2 rk[4], rv[4];
          step_load_rows<D>(ka, q, j0, m, rk, rv, lane);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (k < m) step_token_rows<D>(ka, rk[k], rv[k], j0 + k, c, pid, slot, (j0 + k) * g >= h0, 0u, false, lane);
        }
      }
    } else {
      const int lo_local = max(0, t - w + 1);
      // per-head modes: a page before the local window is read by the block's full heads
      // only; a page across the window's start brings its slot positions
      if (HM && lane < T) {
        if (wlast < lo_local) wmeta |= kEarly;
        else if (wfirst < lo_local) wmeta |= kMask;
      }
      const int4 rb = make_int4(t, sp, ns, pre[q]);
      {  // the unit's query rows
        const int need = nh * D * 2;
        int taken = 0;
        int off = reserve(need, taken, waited);
        if (off == -2) {  // before the wait with the ring full: wait, then block
          ensure_waited();
          off = reserve(need, taken, true);
        }
        if (off < 0) {
          ok = false;
          break;
        }
        const bool only = T == 0 && !has_new;
        const int meta = kQRows | kFirst | (only ? (kLast | kNoPage) : 0) | (qb << 16);
        const int4 ra = make_int4(meta, off, q, lo), rc = make_int4(hpack, max(0, t - w + 1), -1, hsel);
        const uint16_t* src = ka.q + (static_cast<int64_t>(q) * a.Hq + h0) * D;
        if (HM) {  // the slots' rows, each from its head (no early mode with head modes)
          const uint32_t slot = push(ra, rb, rc, taken, need);
          if (lane == 0)
            for (int sl = 0; sl < nh; ++sl)
              bulk_g2s(cr.ring + off + sl * D * 2, ka.q + (static_cast<int64_t>(q) * a.Hq + slot_head(sl)) * D, D * 2,
                       &cr.full[slot]);
        } else if (waited) {
          const uint32_t slot = push(ra, rb, rc, taken, need);
          if (lane == 0) bulk_g2s(cr.ring + off, src, need, &cr.full[slot]);
        } else {  // its slot now, its record and copy after the wait
          dq_slot = static_cast<int>(pushed % kStages);
          if (lane == 0) cr.sbytes[dq_slot] = taken;
          ++pushed;
          dq_off = off;
          dq_need = need;
          dq_ra = ra;
          dq_rb = rb;
          dq_rc = rc;
          dq_src = src;
        }
      }
      // every page's copy, worked out once per unit (lane j: page j), so that a push
      // is a few shuffles and the copy
      uint64_t pg_src = 0;  // the page
      int pg_geo = 0;       // slice bytes | KV slices per stage << 20
      const unsigned pg_need = wlast < lo_local ? need_full : need_any;  // the KV heads it brings
      if (lane < T) {
        const int c = wmeta & 3, slice = a.slice[c];
        const int posb = (wmeta & kMask) ? 4 * P : 0;
        pg_src = reinterpret_cast<uint64_t>(a.pool[c] + static_cast<int64_t>(wid) * a.page_bytes[c]);
        pg_geo = slice | (max(1, (R / 2 - posb) / slice) << 20);
      }
      // decode step: the query's own token, as a stage holding it at slot 0 of a
      // page-shaped slice per KV head (consumers read it as a page with one key), after
      // the unit's pages (the wait on the previous kernel that it needs then holds back
      // no page copy).  The stage comes with no bytes: each consumer warp quantises its
      // KV head's rows into it and into the token's slot in the cache, so that the
      // producer goes on issuing copies.  After a call error (known only after the wait)
      // one empty stage stands in for it.
      bool new_done = !has_new;
      auto push_new = [&](bool last) -> bool {
        ensure_waited();  // the token's K / V rows come from the previous kernel
        pages_ready();
        new_done = true;
        if (call_failed()) {
          int taken = 0;
          const int off = reserve(0, taken, true);
          if (off < 0) return false;
          push(make_int4((last ? kLast : 0) | (qb << 16), off, q, lo), rb, make_int4(0, 1 << 8, -1, 0), taken, 0);
          return true;
        }
        const int c = ent[2 * q + 1] & 3;
        const int slice = a.slice[c];
        // every KV head's slot 0 in one stage when the class's regions allow it: head j's
        // K codes, V codes, K (s, z) and V (s, z) each at j rows (j * rowb bytes) past the
        // region's start, so that a consumer reads its head as a page-shaped slice at
        // j * rowb; the reservation covers what the consumers read of the slots past the
        // fill
        const int b = bits_of_class(c), rowb = b == 16 ? 2 * D : D * b / 8, ng = D >> (__ffs(a.G) - 1);
        if (nkv <= 4 && (b == 16 || (nkv - 1) * rowb + ng * 4 <= P * ng * 4)) {
          const int span = b == 16 ? (nkv - 1 + P + 16) * rowb : (nkv - 1) * rowb + 2 * P * rowb + (P + 16) * ng * 4;
          int taken = 0;
          const int off = reserve(align16(span), taken, true);
          if (off < 0) return false;
          const int meta = c | (1 << 2) | (last ? kLast : 0) | (qb << 16);
          push(make_int4(meta, off, q, lo), rb, make_int4(0, nkv | (1 << 8), kNewRows, rowb), taken, 0);
          return true;
        }
        for (int k0 = 0; k0 < nkv; ++k0) {  // otherwise one stage per KV head
          int taken = 0;
          const int off = reserve(slice, taken, true);
          if (off < 0) return false;
          const int meta = c | (1 << 2) | (last && k0 == nkv - 1 ? kLast : 0) | (qb << 16);
          push(make_int4(meta, off, q, lo), rb, make_int4(k0, 1 | (1 << 8), kNewRows, slice), taken, 0);
        }
        return true;
      };
      for (int j = 0; j < T && ok; ++j) {
        const uint8_t* page = reinterpret_cast<const uint8_t*>(__shfl_sync(0xffffffffu, pg_src, j));
        const int geo = __shfl_sync(0xffffffffu, pg_geo, j);
        int pm = __shfl_sync(0xffffffffu, wmeta, j);
        const unsigned needed = __shfl_sync(0xffffffffu, pg_need, j);
        const int slice = geo & 0xfffff, maxk = geo >> 20;
        const unsigned all = (1u << nkv) - 1u;
        if (!HM && !(pm & kMask) && needed == all && nkv <= maxk) {
          // a run of full pages of this class, every KV head of the block: one stage
          // holding up to R/2 bytes of them (a page's slices after the other), one copy
          // per page; only the run's last page may hold fewer than P tokens
          const int pb = nkv * slice;
          int run = 1;
          while (j + run < T && (run + 1) * pb <= R / 2) {
            const int pm2 = __shfl_sync(0xffffffffu, wmeta, j + run);
            if ((pm2 & (3 | kMask)) != (pm & 3) || ((pm >> 2) & 127) != P) break;
            pm = pm2;
            ++run;
          }
          int taken = 0;
          const int off = reserve_any(run * pb, taken);
          if (off < 0) {
            ok = false;
            break;
          }
          const bool last = j + run == T && new_done;
          const int meta = pm | (last ? kLast : 0) | (qb << 16);
          const uint32_t slot =
              push(make_int4(meta, off, q, lo), rb, make_int4(0, nkv | (run << 8), -1, slice), taken, run * pb);
          for (int r = 0; r < run; ++r) {
            const uint8_t* pg = reinterpret_cast<const uint8_t*>(__shfl_sync(0xffffffffu, pg_src, j + r));
            if (lane == 0) bulk_g2s(cr.ring + off + r * pb, pg + a.hdr + static_cast<int64_t>(kv0) * slice, pb, &cr.full[slot]);
          }
          j += run - 1;
          continue;
        }
        if (HM) {  // per-head modes: the needed slots' slices, at most maxk a stage
          unsigned rest = needed;
          while (rest && ok) {
            unsigned chunk = 0;
            int nk = 0;
            while (rest && nk < maxk) {
              chunk |= rest & (0u - rest);
              rest &= rest - 1u;
              ++nk;
            }
            const int posb = (pm & kMask) ? 4 * P : 0;
            const int need = nk * slice + posb;
            int taken = 0;
            const int off = reserve_any(need, taken);
            if (off < 0) {
              ok = false;
              break;
            }
            const bool last = j == T - 1 && rest == 0 && new_done;
            const int meta = pm | (last ? kLast : 0) | (qb << 16);
            const uint32_t slot = push(make_int4(meta, off, q, lo), rb,
                                       make_int4(static_cast<int>(chunk), nk | (1 << 8), posb ? off + nk * slice : -1, slice),
                                       taken, need);
            if (lane == 0) {
              int pos = 0;
              for (unsigned m = chunk; m; m &= m - 1u, ++pos) {
                const int kvh = slot_head(__ffs(m) - 1) / g;
                bulk_g2s(cr.ring + off + pos * slice, page + a.hdr + static_cast<int64_t>(kvh) * slice, slice,
                         &cr.full[slot]);
              }
              if (posb) bulk_g2s(cr.ring + off + nk * slice, page, posb, &cr.full[slot]);
            }
          }
          continue;
        }
        // one stage per run of consecutive needed KV heads, at most maxk slices each
        for (int k0 = __ffs(needed) - 1; k0 >= 0 && k0 < nkv;) {
          int nk = 1;
          while (nk < maxk && k0 + nk < nkv && ((needed >> (k0 + nk)) & 1u)) ++nk;
          const int posb = (pm & kMask) ? 4 * P : 0;
          const int need = nk * slice + posb;
          int taken = 0;
          const int off = reserve_any(need, taken);
          if (off < 0) {
            ok = false;
            break;
          }
          const unsigned later = needed >> (k0 + nk);  // needed KV heads after this stage
          const bool last = j == T - 1 && later == 0 && new_done;
          const int meta = pm | (last ? kLast : 0) | (qb << 16);
          const uint32_t slot = push(make_int4(meta, off, q, lo), rb,
                                     make_int4(k0, nk | (1 << 8), posb ? off + nk * slice : -1, slice), taken, need);
          if (lane == 0) {
            bulk_g2s(cr.ring + off, page + a.hdr + static_cast<int64_t>(kv0 + k0) * slice, nk * slice, &cr.full[slot]);
            if (posb) bulk_g2s(cr.ring + off + nk * slice, page, posb, &cr.full[slot]);
          }
          k0 = later ? k0 + nk + __ffs(later) - 1 : nkv;
        }
      }
      if (ok && !new_done && !push_new(true)) ok = false;
      if (!ok) break;
      ensure_waited();  // the next unit's query rows come from the previous kernel
    }
    __syncwarp();
    if (on_demand) {  // the consumers first finish this unit
      while (ok && released < pushed) ok = release_one();
      if (!ok) break;
    }
    take_next();
    u = __shfl_sync(0xffffffffu, u_next, 0);
  }
  if (ok) {
    ensure_waited();
    pages_ready();  // the last CTA commits from them
    int taken = 0;
    if (reserve(0, taken, true) < 0) ok = false;
    else push(make_int4(kEnd, 0, 0, 0), make_int4(0, 0, 0, 0), make_int4(0, 0, -1, 0), taken, 0);
  }
  if (!ok) {  // a wait gave up: stop the consumers, then let every copy in flight land
    if (!waited) {
      pdl_wait();
      waited = true;
      pdl_trigger();
    }
    if (lane == 0) {
      *cr.abort_flag = 1;
      set_status(a.ctrl, TRR_ERR_TIMEOUT);
      atomicExch(&a.lctl[kAborted], 1);
    }
    // copies in flight always land (they only read memory): wait for them with the
    // default bound whatever the configured one
    for (uint32_t s = released; s < pushed; ++s)
      if (static_cast<int>(s % kStages) != dq_slot) mbar_wait(&cr.full[s % kStages], (s / kStages) & 1);
  }
}

// Merges `count` partial rows at p0, p0 + stride, ...: the common maximum Mx, the
// weighted sum of L and the weighted rows (lane holds dims lane * DPL ..).
template <int D>
__device__ __forceinline__ void merge_partials(const float* p0, int64_t stride, int count, int lane, float& Mx,
                                               float& Ls, float (&acc_o)[D / 32]) {
  // Chunks of CH partials: each chunk's (max, sum) words and rows are loaded together
  // (one round trip to L2 for up to CH splits), then folded into the running result;
  // CH keeps the rows within the registers the consumers have free at this point.
  constexpr int DPL = D / 32, CH = D == 64 ? 8 : 4;
  Mx = kNegInf;
  float lsum = 0.f;  // lane s: the weighted sums of the partials it reads the words of
#pragma unroll
  for (int j = 0; j < DPL; ++j) acc_o[j] = 0.f;
  for (int s0 = 0; s0 < count; s0 += CH) {
    const int cnt = min(CH, count - s0);
    float2 ml = make_float2(kNegInf, 0.f);
    if (lane < cnt) ml = __ldcg(reinterpret_cast<const float2*>(p0 + (s0 + lane) * stride + D));
    float rows[CH][DPL];
#pragma unroll
    for (int s = 0; s < CH; ++s) {
#pragma unroll
      for (int j = 0; j < DPL; ++j) rows[s][j] = s < cnt ? __ldcg(p0 + (s0 + s) * stride + lane * DPL + j) : 0.f;
    }
    float cm = ml.x;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, o));
    const float nm = fmaxf(Mx, cm);
    if (nm != kNegInf) {
      const float f = Mx == kNegInf ? 0.f : fast_exp2(Mx - nm);  // the earlier chunks' scale
#pragma unroll
      for (int j = 0; j < DPL; ++j) acc_o[j] *= f;
      lsum *= f;
      const float wl = ml.x == kNegInf ? 0.f : fast_exp2(ml.x - nm);  // lane s: weight of row s0 + s
      lsum = fmaf(wl, ml.y, lsum);
#pragma unroll
      for (int s = 0; s < CH; ++s) {
        const float wgt = __shfl_sync(0xffffffffu, wl, s);
#pragma unroll
        for (int j = 0; j < DPL; ++j) acc_o[j] = fmaf(wgt, rows[s][j], acc_o[j]);
      }
      Mx = nm;
    }
  }
  Ls = lsum;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, o);
}

// Counts this warp's arrival on *counter (release of its partial stores, acquire of
// the others'); true for the last of `expected` arrivals, which resets the counter.
__device__ __forceinline__ bool arrive_last(int* counter, int expected, int lane) {
  __syncwarp();
  int arrivals = 0;
  if (lane == 0) arrivals = atom_add_acq_rel(counter, 1);
  __syncwarp();
  arrivals = __shfl_sync(0xffffffffu, arrivals, 0);
  if (arrivals != expected - 1) return false;
  if (lane == 0) *counter = 0;  // ready for the next call
  return true;
}

// A (query, head) row at its end: lane holds DPL consecutive dims from dim0 of the
// unnormalised sum acc = sum_j p_j v_j (weights relative to max M, log2 domain) and the
// row's weight sum L.  One split: the bf16 row.  Otherwise the split's fp32 partial,
// merged in two levels: the last split of each group of kMergeGroup to arrive folds the
// group into the group's first partial, and the last group to arrive merges the groups
// into the row (one level when nsplit <= kMergeGroup).
template <int D>
__device__ __forceinline__ void store_or_merge(const AttnKernelArgs& ka, const float* v, int dim0, float M, float L,
                                               int sp, int qi, int qh, int nsplit, int base, int lane) {
  constexpr int DPL = D / 32;
  const LayerArgs& a = ka.a;
  const int64_t orow = (static_cast<int64_t>(qi) * a.Hq + qh) * D;
  if (nsplit == 1) {
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int j = 0; j < DPL; j += 2)
      *reinterpret_cast<__nv_bfloat162*>(ka.out + orow + dim0 + j) = __floats2bfloat162_rn(v[j] * inv, v[j + 1] * inv);
    return;
  }
  const int64_t sstride = static_cast<int64_t>(a.Hq) * (D + 4);
  float* p0 = a.part + (static_cast<int64_t>(base) * a.Hq + qh) * (D + 4);  // split 0's partial
  float* pp = p0 + sp * sstride;
#pragma unroll
  for (int j = 0; j < DPL; j += 2) *reinterpret_cast<float2*>(pp + dim0 + j) = make_float2(v[j], v[j + 1]);
  if (lane == 0) *reinterpret_cast<float2*>(pp + D) = make_float2(M, L);
  if (ka.defer_merge) return;  // the combine kernel merges this query's splits
  int* counters = a.cnt + (static_cast<int64_t>(qi) * a.Hq + qh) * a.cnt_stride;
  float Mx, Ls, acc_o[DPL];
  int ngroups = nsplit, gstride = 1;
  if (nsplit > kMergeGroup) {
    const int gr = sp / kMergeGroup, g0 = gr * kMergeGroup, gn = min(kMergeGroup, nsplit - g0);
    if (!arrive_last(counters + 1 + gr, gn, lane)) return;
    float* pg = p0 + g0 * sstride;
    merge_partials<D>(pg, sstride, gn, lane, Mx, Ls, acc_o);
    __syncwarp();  // every lane has read the group's rows before the first is overwritten
#pragma unroll
    for (int j = 0; j < DPL; ++j) __stcg(pg + lane * DPL + j, acc_o[j]);
    if (lane == 0) __stcg(reinterpret_cast<float2*>(pg + D), make_float2(Mx, Ls));
    ngroups = (nsplit + kMergeGroup - 1) / kMergeGroup;
    gstride = kMergeGroup;
  }
  if (!arrive_last(counters, ngroups, lane)) return;
  merge_partials<D>(p0, sstride * gstride, ngroups, lane, Mx, Ls, acc_o);
  const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
  for (int j = 0; j < DPL; j += 2)
    *reinterpret_cast<__nv_bfloat162*>(ka.out + orow + lane * DPL + j) =
        __floats2bfloat162_rn(acc_o[j] * inv, acc_o[j + 1] * inv);
}

// ------------------------------------------------- CUDA-core consumer (MHA) --
// Warp cw computes query head (block * kNcw + cw): lane pair (key, half) of a 64-wide
// head (four lanes for 128) dequantises in registers and keeps its own online softmax.

// The end of a unit for a CUDA-core consumer: merge the lanes' states, then store.
template <int D, int E>
__device__ __forceinline__ void finish_unit(const AttnKernelArgs& ka, LaneState<E>& st, int cur_cls, int sp, int qi,
                                            int qh, int nsplit, int base, uint32_t tbl, int lane) {
  constexpr int LPK = D / E;   // lanes per key
  constexpr int DPL = D / 32;  // dimensions per lane after the merge
  const int part = lane % LPK, kl = lane / LPK;
  // rescale to the common maximum, then reduce-scatter over the key lanes: each
  // halving step keeps half of the 32 dims and sends the other half to the partner
  acc_to_neutral(st.acc, cur_cls, tbl);
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
    for (int j = 0; j < E; j += 2) {
      const float2 r = __ffma2_rn(make_float2(st.acc[j], st.acc[j + 1]), s49, zf);
      st.acc[j] = r.x;
      st.acc[j + 1] = r.y;
    }
  }
#pragma unroll
  for (int width = E / 2, o = 16; o >= LPK; width >>= 1, o >>= 1) {
    const bool upper = lane & o;
#pragma unroll
    for (int i = 0; i < E / 2; ++i) {
      if (i < width) {
        const float keep = upper ? st.acc[width + i] : st.acc[i];
        const float give = upper ? st.acc[i] : st.acc[width + i];
        st.acc[i] = keep + __shfl_xor_sync(0xffffffffu, give, o);
      }
    }
  }
  // lane (kl, part) now holds dims part*E + DPL*kl .. + DPL-1 in acc[0 .. DPL-1]
  store_or_merge<D>(ka, st.acc, part * E + DPL * kl, M, L, sp, qi, qh, nsplit, base, lane);
}

template <int D, int P, int E, bool HM, bool STEP>
__device__ __forceinline__ void run_consumer_cc(const AttnKernelArgs& ka, const CtaRing& cr, const int* ent, int cw,
                                                int lane) {
  constexpr int LPK = D / E;     // lanes per key
  constexpr int KPI = 32 / LPK;  // keys per warp iteration
  const LayerArgs& a = ka.a;
  const int g = a.Hq / a.Hkv;
  const int part = lane % LPK;
  LaneState<E> st;
  float qp[E];
  float sumq = 0.f;
  int cur_cls = 3;
  st.m = kNegInf;
  st.l = 0.f;
  st.zacc = 0.f;
#pragma unroll
  for (int j = 0; j < E; ++j) st.acc[j] = 0.f;
  // the current unit
  int u_q = 0, u_h = 0, u_kvi = 0, u_lo = 0, u_hi = 0, u_sp = 0, u_ns = 1, u_base = 0;
  bool u_local = false;  // per-head modes: this warp's head is local (it skips early pages)
  bool active = false;
  for (uint32_t s = 0;; ++s) {
    const uint32_t slot = s % kStages;
    const bool arrived = mbar_wait_or(&cr.full[slot], (s / kStages) & 1, cr.abort_flag, a.wait_ns);
    if (!__all_sync(0xffffffffu, arrived)) {  // give up together, never half a warp
      if (lane == 0) {
        *cr.abort_flag = 1;
        set_status(a.ctrl, TRR_ERR_TIMEOUT);
        atomicExch(&a.lctl[kAborted], 1);
      }
      break;
    }
    const uint32_t rec = smem_u32(cr.recs) + slot * 48;
    const int4 ra = lds128i(rec);
    const int meta = ra.x;
    if (meta & kEnd) break;
    if (meta & kQRows) {
      const int4 rb = lds128i(rec + 16);
      const int qb = (meta >> 16) & 0x7fff;
      u_h = qb * kNcw + cw;
      active = u_h < a.Hq;
      if (HM && active) {  // the head of this warp's slot (ranked by mode; or h0 + slot)
        const int hsel = lds128i(rec + 32).w;
        if (hsel >= 0) u_h = (hsel >> (8 * cw)) & 255;
      }
      u_kvi = u_h / g - (qb * kNcw) / g;
      u_q = ra.z;
      u_lo = ra.w;
      u_hi = rb.x;
      u_sp = rb.y;
      u_ns = rb.z;
      u_base = rb.w;
      u_local = false;
      if (STEP && active && u_sp == u_ns - 1) step_prefetch_rows<D>(ka, u_q, u_h / g, lane);
      if (HM && active) {  // this head's own mode: {head modes, local lo}
        const int4 rq = lds128i(rec + 32);
        const int hm = (rq.x >> (2 * cw)) & 3;
        if (hm == TRR_MODE_SKIP) {  // a zero row (written once, by split 0), no merge
          if (u_sp == 0 && lane < D / 8)
            reinterpret_cast<uint4*>(ka.out + (static_cast<int64_t>(u_q) * a.Hq + u_h) * D)[lane] =
                make_uint4(0, 0, 0, 0);
          active = false;
        } else if (hm == TRR_MODE_LOCAL) {
          u_lo = rq.y;
          u_local = true;
        }
      }
      cur_cls = 3;  // the neutral scale is class 16's
      st.m = kNegInf;
      st.l = 0.f;
      st.zacc = 0.f;
#pragma unroll
      for (int j = 0; j < E; ++j) st.acc[j] = 0.f;
      if (active && !(meta & kNoPage)) {
        const uint32_t qa = smem_u32(cr.ring + ra.y + cw * D * 2 + part * E * 2);
        const float2 qs2 = make_float2(ka.qscale, ka.qscale);
        float2 sq2 = make_float2(0.f, 0.f);
#pragma unroll
        for (int qq = 0; qq < E / 8; ++qq) {
          const uint4 uq = lds128(qa + 16 * qq);
          const uint32_t wv[4] = {uq.x, uq.y, uq.z, uq.w};
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const float2 r = __fmul2_rn(make_float2(bf_lo(wv[h]), bf_hi(wv[h])), qs2);
            qp[8 * qq + 2 * h] = r.x;
            qp[8 * qq + 2 * h + 1] = r.y;
            sq2 = __fadd2_rn(sq2, r);
          }
        }
        sumq = sq2.x + sq2.y;
      }
    } else if (active) {
      const int4 rc = lds128i(rec + 32);
      const int nks = rc.y & 255, npg = rc.y >> 8;  // KV slices per page, pages of the stage
      // per-head modes: the stage brings one slice per slot of its mask (rc.x), in slot
      // order; otherwise KV slices rc.x .. rc.x + nks - 1 of the block
      const bool mine = HM ? ((static_cast<unsigned>(rc.x) >> cw) & 1u) != 0 : (u_kvi >= rc.x && u_kvi < rc.x + nks);
      if (mine && !(HM && u_local && (meta & kEarly))) {
        const int cls = meta & 3, fill = (meta >> 2) & 127;  // the last page's fill; the others are full
        if (STEP && rc.z == kNewRows) {  // the query's own token: this warp's KV head (warps that
                                         // share a KV head write the same bytes); the keys past
                                         // the fill that consume_page reads are never used
          const int j = u_h / g;
          step_new_rows<D>(ka, ent, u_q, j, j * g >= u_h - cw, smem_u32(cr.ring + ra.y + (u_kvi - rc.x) * rc.w), lane);
        }
        if (cls != cur_cls) {
          rescale_dyn(qp, st.acc, cur_cls, cls, cr.resc);
          cur_cls = cls;
        }
        const bool masked = meta & kMask;
        for (int pg = 0; pg < npg; ++pg) {
          const int idx = HM ? __popc(static_cast<unsigned>(rc.x) & ((1u << cw) - 1u)) : u_kvi - rc.x;
          const uint32_t s0 = smem_u32(cr.ring + ra.y + (pg * nks + idx) * rc.w);
          const int f = pg == npg - 1 ? fill : P;
          const uint32_t sp = masked ? smem_u32(cr.ring + rc.z) : s0;
          uint64_t pm = ~0ull;  // per-head modes: this KV head's presence mask, which ends
                                // its slice
          if (HM) {
            const uint2 m2 = lds64(s0 + rc.w - a.maskb);
            pm = (static_cast<uint64_t>(m2.y) << 32) | m2.x;
          }
          switch (cls) {
            case 0: consume_page<D, 2, P / KPI, E, HM>(s0, sp, masked, pm, a.G, f, u_lo, u_hi, qp, sumq, st, lane); break;
            case 1: consume_page<D, 4, P / KPI, E, HM>(s0, sp, masked, pm, a.G, f, u_lo, u_hi, qp, sumq, st, lane); break;
            case 2: consume_page<D, 8, P / KPI, E, HM>(s0, sp, masked, pm, a.G, f, u_lo, u_hi, qp, sumq, st, lane); break;
            default: consume_page<D, 16, P / KPI, E, HM>(s0, sp, masked, pm, a.G, f, u_lo, u_hi, qp, sumq, st, lane); break;
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&cr.empty[slot]);  // the stage's bytes are read
    if ((meta & kLast) && active)
      finish_unit<D, E>(ka, st, cur_cls, u_sp, u_q, u_h, u_ns, u_base, cr.resc, lane);
  }
}

// ------------------------------------------------ tensor-core consumer (GQA) --
//
// Warp cw computes the g query heads of KV head (block * kNcw + cw) with mma.sync
// m16n8k16 (f16 or bf16 operands, f32 accumulation).  Thread (gid, tig) = (lane / 4,
// lane % 4) as in the PTX fragment layouts.
//
// q.k: D_s[key][col] = sum_k A[key][k] B[k][col] with A the K codes of 16 keys and B
// the query rows, column col = (head r, quantiser group gi) = (col / NG, col % NG)
// holding head r's query on group gi's dimensions (zero elsewhere), so every column
// gets its own group sum and s, z apply per group.  A code is masked in place and
// read as an f16 subnormal c * 2^(pos - 24) (pos = its bit offset in the 16-bit half);
// the query is pre-scaled by 2^(smax - pos) in f16 so that every product carries the
// same factor 2^(smax - 24).  Width 16 uses bf16 operands (the query is bf16 already).
//
// P.V: O^T[dim][col] = sum_k V^T[dim][key] W[key][col] with W = p * s (f16; bf16 hi
// and lo parts for width 16, whose values are raw bf16).  Pairs along keys for the A
// operand come from byte permutes of two keys' code words.  Each accumulator row keeps
// its class's factor 2^(pos - 24) until the class changes.

__device__ __forceinline__ void mma_f16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                        uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
template <int B>
__device__ __forceinline__ void mma_cls(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                        uint32_t b0, uint32_t b1) {
  if (B == 16) mma_bf16(c, a0, a1, a2, a3, b0, b1);
  else mma_f16(c, a0, a1, a2, a3, b0, b1);
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// K side: pair i of a thread's D/4 dims of one key, as an A-operand word.
template <int B>
__device__ __forceinline__ uint32_t k_pair(const uint32_t* kw, int i) {
  if (B == 16) return kw[i];
  if (B == 8) return __byte_perm(kw[i >> 1], 0u, (i & 1) ? 0x4342 : 0x4140);
  if (B == 4) {
    const int k = i & 3;
    const uint32_t w = k < 2 ? kw[i >> 2] : (kw[i >> 2] >> 8);
    return w & ((k & 1) ? 0x00F000F0u : 0x000F000Fu);
  }
  const int k = i & 7;
  const uint32_t w = k < 5 ? kw[i >> 3] : (kw[i >> 3] >> 10);
  return w & (0x00030003u << (2 * (k < 5 ? k : k - 5)));
}
// the two dims (relative to the thread's first) of K pair i and their bit offset
template <int B> __host__ __device__ constexpr int kp_lo(int i) {
  return B >= 8 ? 2 * i : B == 4 ? 8 * (i / 4) + i % 4 : 16 * (i / 8) + i % 8;
}
template <int B> __host__ __device__ constexpr int kp_hi(int i) {
  return B >= 8 ? 2 * i + 1 : B == 4 ? 8 * (i / 4) + i % 4 + 4 : 16 * (i / 8) + 8 + i % 8;
}
template <int B> __host__ __device__ constexpr int kp_pos(int i) {
  return B >= 8 ? 0 : B == 4 ? 4 * (i % 2) : 2 * ((i % 8) < 5 ? i % 8 : i % 8 - 5);
}
template <int B> __host__ __device__ constexpr int smax_of() { return B == 2 ? 8 : B == 4 ? 4 : 0; }

// V side: dim j of the thread's D/8 dims for keys (a, b) as an A-operand word (key a
// in the low half).
template <int B>
__device__ __forceinline__ uint32_t v_pair(const uint32_t* wa, const uint32_t* wb, int j) {
  if (B == 16) return __byte_perm(wa[j >> 1], wb[j >> 1], (j & 1) ? 0x7632 : 0x5410);
  if (B == 8) {
    const int k = j & 3;
    const uint32_t x = __byte_perm(wa[j >> 2], wb[j >> 2], k < 2 ? 0x5140 : 0x7362);
    return __byte_perm(x, 0u, (k & 1) ? 0x4342 : 0x4140);
  }
  if (B == 4) {
    const int k = j & 7;
    uint32_t x = __byte_perm(wa[j >> 3], wb[j >> 3], k < 4 ? 0x5410 : 0x7632);
    if ((k & 3) >= 2) x >>= 8;
    return x & ((k & 1) ? 0x00F000F0u : 0x000F000Fu);
  }
  const int k = j & 15, kk = k & 7;
  uint32_t x = __byte_perm(wa[j >> 4], wb[j >> 4], k < 8 ? 0x5410 : 0x7632);
  if (kk >= 5) x >>= 10;
  return x & (0x00030003u << (2 * (kk < 5 ? kk : kk - 5)));
}
// log2 of the factor a V accumulator row carries in class index c (dim j of the
// thread's D/8): 2^(pos - 24) for codes, 1 for bf16
__host__ __device__ constexpr int vfac_log2(int c, int j) {
  return c == 3 ? 0 : c == 2 ? -24 : c == 1 ? 4 * (j & 1) - 24 : 2 * ((j & 7) < 5 ? (j & 7) : (j & 7) - 5) - 24;
}

// Loads `nw` 32-bit words from shared address a (16-byte loads where aligned).
template <int NW>
__device__ __forceinline__ void lds_words(uint32_t a, uint32_t* w) {
  if (NW % 4 == 0) {
#pragma unroll
    for (int k = 0; k < NW; k += 4) {
      const uint4 u = lds128(a + 4 * k);
      w[k] = u.x; w[k + 1] = u.y; w[k + 2] = u.z; w[k + 3] = u.w;
    }
  } else if (NW == 2) {
    const uint2 u = lds64(a);
    w[0] = u.x; w[1] = u.y;
  } else {
    w[0] = lds32(a);
  }
}

template <int D, int NG>
struct MmaState {
  static constexpr int NP = D / 8;   // K pairs per thread and key
  static constexpr int MT = D / 16;  // m-tiles of P.V
  uint32_t qaddr;     // shared address of word 0 of the bf16 query of the thread's B column
                      // on its D/4 dims, kept in the warp's scratch (word i at + 128 i)
  uint32_t kb[NP];    // the q.k B operand in the current class
  float qsum[2];      // qscale * sum of the query over (head, group) of the thread's two columns
  float m[2], l[2], zacc[2];
  float acc[MT][4];
  float escale;       // 2^-E: the query pre-scale keeping f16 values in range
  int E;
};

template <int D, int NG, int B>
__device__ __forceinline__ void mma_build_kb(MmaState<D, NG>& ms) {
  constexpr int NP = D / 8;
  uint32_t qraw[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) qraw[i] = lds32(ms.qaddr + 128 * i);
  if (B == 16) {
#pragma unroll
    for (int i = 0; i < NP; ++i) ms.kb[i] = qraw[i];
  } else {
#pragma unroll
    for (int i = 0; i < NP; ++i) {
      const int lo = kp_lo<B>(i), hi = kp_hi<B>(i);
      const float f = pow2f(smax_of<B>() - kp_pos<B>(i)) * ms.escale;
      const float ql = (lo & 1) ? bf_hi(qraw[lo >> 1]) : bf_lo(qraw[lo >> 1]);
      const float qh = (hi & 1) ? bf_hi(qraw[hi >> 1]) : bf_lo(qraw[hi >> 1]);
      ms.kb[i] = pack_f16x2(ql * f, qh * f);
    }
  }
}

// class index from -> to: new B operand, accumulator rows to the new class's factors
template <int D, int NG>
__device__ __forceinline__ void mma_switch(MmaState<D, NG>& ms, int from, int to) {
  switch (to) {
    case 0: mma_build_kb<D, NG, 2>(ms); break;
    case 1: mma_build_kb<D, NG, 4>(ms); break;
    case 2: mma_build_kb<D, NG, 8>(ms); break;
    default: mma_build_kb<D, NG, 16>(ms); break;
  }
#pragma unroll
  for (int t = 0; t < D / 16; ++t) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int j = 2 * t + r;
      const float f = __int_as_float((127 + vfac_log2(to, j) - vfac_log2(from, j)) << 23);
      ms.acc[t][2 * r] *= f;
      ms.acc[t][2 * r + 1] *= f;
    }
  }
}

// One page of class B: keys in chunks of 16.
template <int D, int NG, int B>
__device__ __forceinline__ void mma_page(MmaState<D, NG>& ms, uint32_t s0, uint32_t spos, bool masked, int P, int fill,
                                         int lo, int hi, float qscale, const bool (&col_ok)[2],
                                         const int (&col_gi)[2], int lane) {
  constexpr int KS = D / 16, MT = D / 16;
  constexpr int rowb = B == 16 ? 2 * D : D * B / 8;  // bytes of one key's K (or V) row
  constexpr int KW = D * B / 128;                    // K words per thread and key (D/4 dims)
  constexpr int VB = D * B / 64;                     // V bytes per thread and key (D/8 dims)
  constexpr int VW = VB >= 4 ? VB / 4 : 1;           // V words loaded per key
  const int gid = lane >> 2, tig = lane & 3;
  const uint32_t kbase = s0, vbase = s0 + P * rowb;
  const uint32_t kszb = s0 + 2 * P * rowb, vszb = kszb + P * NG * 4;
  const float kfac = __int_as_float((127 + 24 - smax_of<B>() + ms.E) << 23) * qscale;
  const uint32_t wsel = (gid & 1) ? 0x7632u : 0x5410u;  // the W half of this thread's B column
#pragma unroll 1
  for (int c0 = 0; c0 < fill; c0 += 16) {
    // ------------------------------------------------ scores of keys c0+gid, c0+gid+8
    const int k1 = c0 + gid, k2 = k1 + 8;
    float ca[4] = {0.f, 0.f, 0.f, 0.f}, cb[4] = {0.f, 0.f, 0.f, 0.f};
    // the keys' words in two halves (k-steps 0 .. KS/2-1, then the rest), so that only
    // half a row per key is live at a time
    constexpr int KH = KW >= 2 ? 2 : 1, KWH = KW / KH, KSH = KS / KH;
#pragma unroll
    for (int hf = 0; hf < KH; ++hf) {
      uint32_t kw1[KWH], kw2[KWH];
      lds_words<KWH>(kbase + k1 * rowb + tig * (KW * 4) + hf * KWH * 4, kw1);
      lds_words<KWH>(kbase + k2 * rowb + tig * (KW * 4) + hf * KWH * 4, kw2);
#pragma unroll
      for (int s = hf * KSH; s < (hf + 1) * KSH; ++s) {
        const int i0 = 2 * s - hf * 2 * KSH;  // pair index inside the half
        if (s & 1)
          mma_cls<B>(cb, k_pair<B>(kw1, i0), k_pair<B>(kw2, i0), k_pair<B>(kw1, i0 + 1), k_pair<B>(kw2, i0 + 1),
                     ms.kb[2 * s], ms.kb[2 * s + 1]);
        else
          mma_cls<B>(ca, k_pair<B>(kw1, i0), k_pair<B>(kw2, i0), k_pair<B>(kw1, i0 + 1), k_pair<B>(kw2, i0 + 1),
                     ms.kb[2 * s], ms.kb[2 * s + 1]);
      }
    }
    bool v1 = k1 < fill, v2 = k2 < fill;
    if (masked) {
      const int p1 = static_cast<int>(lds32(spos + 4 * k1)), p2 = static_cast<int>(lds32(spos + 4 * k2));
      v1 = v1 && p1 >= lo && p1 <= hi;
      v2 = v2 && p2 >= lo && p2 <= hi;
    }
    // column partial scores cp[key][j] (log2 units)
    float cp[2][2];
    float2 vsz[2][2];  // V (s, z) of the thread's two keys for its two columns' groups
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const int key = kk ? k2 : k1;
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const float cv = ca[2 * kk + j] + cb[2 * kk + j];
        if (B == 16) {
          cp[kk][j] = cv * qscale;
        } else {
          const uint32_t szw = lds32(kszb + (key * NG + col_gi[j]) * 4);
          const float2 sz = __half22float2(*reinterpret_cast<const __half2*>(&szw));
          cp[kk][j] = fmaf(sz.x * kfac, cv, sz.y * ms.qsum[j]);
        }
      }
      if (B != 16) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const uint32_t szw = lds32(vszb + (key * NG + col_gi[j]) * 4);
          vsz[kk][j] = __half22float2(*reinterpret_cast<const __half2*>(&szw));
        }
      }
    }
    if (B != 16) {  // a slot past the fill or outside the range may hold any bytes
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        if (!v1) vsz[0][j] = make_float2(0.f, 0.f);
        if (!v2) vsz[1][j] = make_float2(0.f, 0.f);
      }
    }
    // head scores per column slot
    float sc[2][2];
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      if (NG == 1) {
        sc[kk][0] = cp[kk][0];
        sc[kk][1] = cp[kk][1];
      } else {
        float h = cp[kk][0] + cp[kk][1];
        if (NG == 4) h += __shfl_xor_sync(0xffffffffu, h, 1);
        sc[kk][0] = sc[kk][1] = h;
      }
      const bool vk = kk ? v2 : v1;
#pragma unroll
      for (int j = 0; j < 2; ++j)
        if (!(vk && col_ok[j])) sc[kk][j] = kNegInf;
    }
    // online softmax per slot (the running max is shared by the key lanes: p <= 1)
    float p[2][2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      if (NG > 1 && j == 1) {
        p[0][1] = p[0][0];
        p[1][1] = p[1][0];
        continue;
      }
      float mx = fmaxf(sc[0][j], sc[1][j]);
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      if (mx > ms.m[j]) {
        const float alpha = fast_exp2(ms.m[j] - mx);
        ms.m[j] = mx;
        const int j1 = NG > 1 ? 1 : j;  // both slots hold one head when NG > 1
#pragma unroll
        for (int jj = j; jj <= j1; ++jj) {
          ms.l[jj] *= alpha;
          ms.zacc[jj] *= alpha;
#pragma unroll
          for (int t = 0; t < MT; ++t) {
            ms.acc[t][jj] *= alpha;
            ms.acc[t][jj + 2] *= alpha;
          }
        }
        if (NG > 1) ms.m[1] = mx;
      }
      p[0][j] = fast_exp2(sc[0][j] - ms.m[j]);
      p[1][j] = fast_exp2(sc[1][j] - ms.m[j]);
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      ms.l[j] += p[0][j] + p[1][j];
      if (B != 16) ms.zacc[j] = fmaf(p[0][j], vsz[0][j].y, fmaf(p[1][j], vsz[1][j].y, ms.zacc[j]));
    }
    // ------------------------------------------------ P.V
    // W of the thread's keys (gid, gid + 8) x columns (2 tig, 2 tig + 1), then the
    // B operand of column gid, keys (2 tig, 2 tig + 1) and (2 tig + 8, 2 tig + 9)
    const int src0 = 8 * tig + (gid >> 1), src1 = src0 + 4;
    uint32_t b0, b1, bl0 = 0, bl1 = 0;
    if (B == 16) {
      const uint32_t h1 = pack_bf16x2(p[0][0], p[0][1]), h2 = pack_bf16x2(p[1][0], p[1][1]);
      const uint32_t l1 = pack_bf16x2(p[0][0] - bf_lo(h1), p[0][1] - bf_hi(h1));
      const uint32_t l2 = pack_bf16x2(p[1][0] - bf_lo(h2), p[1][1] - bf_hi(h2));
      b0 = __byte_perm(__shfl_sync(0xffffffffu, h1, src0), __shfl_sync(0xffffffffu, h1, src1), wsel);
      b1 = __byte_perm(__shfl_sync(0xffffffffu, h2, src0), __shfl_sync(0xffffffffu, h2, src1), wsel);
      bl0 = __byte_perm(__shfl_sync(0xffffffffu, l1, src0), __shfl_sync(0xffffffffu, l1, src1), wsel);
      bl1 = __byte_perm(__shfl_sync(0xffffffffu, l2, src0), __shfl_sync(0xffffffffu, l2, src1), wsel);
    } else {
      const uint32_t x1 = pack_f16x2(p[0][0] * vsz[0][0].x, p[0][1] * vsz[0][1].x);
      const uint32_t x2 = pack_f16x2(p[1][0] * vsz[1][0].x, p[1][1] * vsz[1][1].x);
      b0 = __byte_perm(__shfl_sync(0xffffffffu, x1, src0), __shfl_sync(0xffffffffu, x1, src1), wsel);
      b1 = __byte_perm(__shfl_sync(0xffffffffu, x2, src0), __shfl_sync(0xffffffffu, x2, src1), wsel);
    }
    // V codes of keys (2 tig, 2 tig + 1) and (2 tig + 8, 2 tig + 9) on dims gid * D/8 ..
    const int ka0 = c0 + 2 * tig;
    const uint32_t voff = vbase + (VB >= 4 ? gid * VB : (gid * VB) & ~3);
    uint32_t m0 = 0xffffffffu, m1 = 0xffffffffu;  // bf16 values of keys out of range read as 0
    if (B == 16) {
      const uint32_t bal1 = __ballot_sync(0xffffffffu, v1), bal2 = __ballot_sync(0xffffffffu, v2);
      m0 = ((bal1 >> (8 * tig)) & 1 ? 0x0000ffffu : 0u) | ((bal1 >> (8 * tig + 4)) & 1 ? 0xffff0000u : 0u);
      m1 = ((bal2 >> (8 * tig)) & 1 ? 0x0000ffffu : 0u) | ((bal2 >> (8 * tig + 4)) & 1 ? 0xffff0000u : 0u);
    }
    // the words in two halves (m-tiles 0 .. MT/2-1, then the rest)
    constexpr int VH = VW >= 2 ? 2 : 1, VWH = VW / VH, MTH = MT / VH;
#pragma unroll
    for (int hf = 0; hf < VH; ++hf) {
      uint32_t wa0[VWH], wb0[VWH], wa1[VWH], wb1[VWH];
      const uint32_t vo = voff + hf * VWH * 4;
      lds_words<VWH>(vo + ka0 * rowb, wa0);
      lds_words<VWH>(vo + (ka0 + 1) * rowb, wb0);
      lds_words<VWH>(vo + (ka0 + 8) * rowb, wa1);
      lds_words<VWH>(vo + (ka0 + 9) * rowb, wb1);
      if (VB < 4) {  // two bytes per key: this thread's half of the word
        const int sh = ((gid * VB) & 3) * 8;
        wa0[0] >>= sh; wb0[0] >>= sh; wa1[0] >>= sh; wb1[0] >>= sh;
      }
#pragma unroll
      for (int t = hf * MTH; t < (hf + 1) * MTH; ++t) {
        const int j0 = 2 * t - hf * 2 * MTH;  // dim pair inside the half
        const uint32_t a0 = v_pair<B>(wa0, wb0, j0) & m0, a1 = v_pair<B>(wa0, wb0, j0 + 1) & m0;
        const uint32_t a2 = v_pair<B>(wa1, wb1, j0) & m1, a3 = v_pair<B>(wa1, wb1, j0 + 1) & m1;
        mma_cls<B>(ms.acc[t], a0, a1, a2, a3, b0, b1);
        if (B == 16) mma_bf16(ms.acc[t], a0, a1, a2, a3, bl0, bl1);
      }
    }
  }
}

// The end of a unit for a tensor-core consumer: per head, the row into the warp's
// scratch, then stored or merged like a CUDA-core row.
template <int D, int NG>
__device__ __forceinline__ void mma_finish(const AttnKernelArgs& ka, MmaState<D, NG>& ms, int cur_cls, int kv, int qi,
                                           int sp, int ns, int base, const bool (&col_ok)[2], const int (&col_r)[2],
                                           const int (&col_gi)[2], float* scr, int lane) {
  constexpr int G = D / NG, DPL = D / 32, MT = D / 16, DV = D / 8;
  const LayerArgs& a = ka.a;
  const int g = a.Hq / a.Hkv;
  const int gid = lane >> 2;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      ms.l[j] += __shfl_xor_sync(0xffffffffu, ms.l[j], o);
      ms.zacc[j] += __shfl_xor_sync(0xffffffffu, ms.zacc[j], o);
    }
  }
#pragma unroll
  for (int t = 0; t < MT; ++t) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int jd = 2 * t + r, dim = gid * DV + jd;
      const float inv = __int_as_float((127 - vfac_log2(cur_cls, jd)) << 23);
#pragma unroll
      for (int j = 0; j < 2; ++j)
        if (col_ok[j] && dim / G == col_gi[j]) scr[col_r[j] * (D + 4) + dim] = fmaf(ms.acc[t][2 * r + j], inv, ms.zacc[j]);
    }
  }
  if (gid == 0) {
#pragma unroll
    for (int j = 0; j < 2; ++j)
      if (col_ok[j] && col_gi[j] == 0) {
        scr[col_r[j] * (D + 4) + D] = ms.m[j];
        scr[col_r[j] * (D + 4) + D + 1] = ms.l[j];
      }
  }
  __syncwarp();
  for (int r = 0; r < g; ++r) {
    const float* row = scr + r * (D + 4);
    float v[DPL];
#pragma unroll
    for (int j = 0; j < DPL; ++j) v[j] = row[lane * DPL + j];
    const int qh = kv * g + r;
    store_or_merge<D>(ka, v, lane * DPL, row[D], row[D + 1], sp, qi, qh, ns, base, lane);
  }
  __syncwarp();
}

template <int D, int NG, bool STEP>
__device__ __forceinline__ void run_consumer_mma(const AttnKernelArgs& ka, const CtaRing& cr, const int* ent, int P, int cw,
                                                 int lane, float* scr) {
  constexpr int NP = D / 8, MT = D / 16, G = D / NG;
  const LayerArgs& a = ka.a;
  const int g = a.Hq / a.Hkv;
  const int gid = lane >> 2, tig = lane & 3;
  // the B column of q.k this thread holds, and its two accumulator columns
  const int brow_r = gid / NG, brow_gi = gid % NG;
  const bool b_ok = brow_r < g && (tig * (D / 4)) / G == brow_gi;
  bool col_ok[2];
  int col_r[2], col_gi[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int c = 2 * tig + j;
    col_r[j] = c / NG;
    col_gi[j] = c % NG;
    col_ok[j] = col_r[j] < g;
  }
  MmaState<D, NG> ms;
  ms.qaddr = smem_u32(scr) + 4 * lane;
  int cur_cls = 3;
  int u_q = 0, u_kv = 0, u_lo = 0, u_hi = 0, u_sp = 0, u_ns = 1, u_base = 0;
  bool active = false;
  for (uint32_t s = 0;; ++s) {
    const uint32_t slot = s % kStages;
    const bool arrived = mbar_wait_or(&cr.full[slot], (s / kStages) & 1, cr.abort_flag, a.wait_ns);
    if (!__all_sync(0xffffffffu, arrived)) {  // give up together, never half a warp
      if (lane == 0) {
        *cr.abort_flag = 1;
        set_status(a.ctrl, TRR_ERR_TIMEOUT);
        atomicExch(&a.lctl[kAborted], 1);
      }
      break;
    }
    const uint32_t rec = smem_u32(cr.recs) + slot * 48;
    const int4 ra = lds128i(rec);
    const int meta = ra.x;
    if (meta & kEnd) break;
    if (meta & kQRows) {
      const int4 rb = lds128i(rec + 16);
      const int qb = (meta >> 16) & 0x7fff;
      u_kv = qb * kNcw + cw;
      active = u_kv < a.Hkv;
      u_q = ra.z;
      u_lo = ra.w;
      u_hi = rb.x;
      u_sp = rb.y;
      u_ns = rb.z;
      u_base = rb.w;
      if (STEP && active && u_sp == u_ns - 1) step_prefetch_rows<D>(ka, u_q, u_kv, lane);
      cur_cls = 3;
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        ms.m[j] = -1e30f;
        ms.l[j] = 0.f;
        ms.zacc[j] = 0.f;
        ms.qsum[j] = 0.f;
      }
#pragma unroll
      for (int t = 0; t < MT; ++t) ms.acc[t][0] = ms.acc[t][1] = ms.acc[t][2] = ms.acc[t][3] = 0.f;
      if (active && !(meta & kNoPage)) {
        // head brow_r's query on the thread's D/4 dims, zero outside its group, kept in
        // the warp's scratch (it is needed again only when the width class changes)
        const uint32_t qa = smem_u32(cr.ring + ra.y + ((cw * g + min(brow_r, g - 1)) * D + tig * (D / 4)) * 2);
        uint32_t qraw[NP];
        lds_words<NP>(qa, qraw);
        float qmax = 0.f, qs = 0.f;
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          if (!b_ok) qraw[i] = 0u;
          const float x0 = bf_lo(qraw[i]), x1 = bf_hi(qraw[i]);
          qmax = fmaxf(qmax, fmaxf(fabsf(x0), fabsf(x1)));
          qs += x0 + x1;
          sts32(ms.qaddr + 128 * i, qraw[i]);
        }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) qmax = fmaxf(qmax, __shfl_xor_sync(0xffffffffu, qmax, o));
        qs += __shfl_xor_sync(0xffffffffu, qs, 1);
        qs += __shfl_xor_sync(0xffffffffu, qs, 2);
        // qs: this B column's (head, group) sum; the accumulator columns 2 tig, 2 tig + 1
        // are the B columns of lanes 4 (2 tig) and 4 (2 tig + 1)
        ms.qsum[0] = __shfl_sync(0xffffffffu, qs, 8 * tig) * ka.qscale;
        ms.qsum[1] = __shfl_sync(0xffffffffu, qs, 8 * tig + 4) * ka.qscale;
        const int ex = static_cast<int>((__float_as_uint(qmax) >> 23) & 0xff) - 127;
        ms.E = min(100, max(0, ex - 6));
        ms.escale = __int_as_float((127 - ms.E) << 23);
        __syncwarp();
        mma_build_kb<D, NG, 16>(ms);
      }
    } else if (active) {
      const int4 rc = lds128i(rec + 32);
      const int nks = rc.y & 255, npg = rc.y >> 8;  // KV slices per page, pages of the stage
      if (cw >= rc.x && cw < rc.x + nks) {
        const int cls = meta & 3, fill = (meta >> 2) & 127;  // the last page's fill; the others are full
        if (STEP && rc.z == kNewRows)  // the query's own token, this warp's KV head
          step_new_rows<D>(ka, ent, u_q, u_kv, true, smem_u32(cr.ring + ra.y + (cw - rc.x) * rc.w), lane);
        if (cls != cur_cls) {
          mma_switch<D, NG>(ms, cur_cls, cls);
          cur_cls = cls;
        }
        const bool masked = meta & kMask;
        for (int pg = 0; pg < npg; ++pg) {
          const uint32_t s0 = smem_u32(cr.ring + ra.y + (pg * nks + cw - rc.x) * rc.w);
          const int f = pg == npg - 1 ? fill : P;
          const uint32_t sp = masked ? smem_u32(cr.ring + rc.z) : s0;
          switch (cls) {
            case 0: mma_page<D, NG, 2>(ms, s0, sp, masked, P, f, u_lo, u_hi, ka.qscale, col_ok, col_gi, lane); break;
            case 1: mma_page<D, NG, 4>(ms, s0, sp, masked, P, f, u_lo, u_hi, ka.qscale, col_ok, col_gi, lane); break;
            case 2: mma_page<D, NG, 8>(ms, s0, sp, masked, P, f, u_lo, u_hi, ka.qscale, col_ok, col_gi, lane); break;
            default: mma_page<D, NG, 16>(ms, s0, sp, masked, P, f, u_lo, u_hi, ka.qscale, col_ok, col_gi, lane); break;
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&cr.empty[slot]);  // the stage's bytes are read
    if ((meta & kLast) && active)
      mma_finish<D, NG>(ka, ms, cur_cls, u_kv, u_q, u_sp, u_ns, u_base, col_ok, col_r, col_gi, scr, lane);
  }
}

// ---------------------------------------------------------------- kernels --

// The prologue every attention kernel shares: barriers, the dependency on the previous
// kernel, the call's work units.
template <bool STEP>
__device__ __forceinline__ CtaRing attn_prologue(const AttnKernelArgs& ka, uint8_t* smem, int P, int NQB, int*& pre,
                                                int*& ent) {
  const AttnSmem lay(ka.ring_bytes, ka.n, ka.scr_floats, STEP);
  CtaRing cr;
  cr.ring = smem + lay.ring;
  cr.recs = reinterpret_cast<int4*>(smem + lay.recs);
  cr.sbytes = reinterpret_cast<int*>(smem + lay.sbytes);
  cr.full = reinterpret_cast<uint64_t*>(smem + lay.full);
  cr.empty = reinterpret_cast<uint64_t*>(smem + lay.empty);
  cr.abort_flag = reinterpret_cast<volatile int*>(smem + lay.flag);
  cr.ent_ready = reinterpret_cast<uint64_t*>(smem + lay.flag + 8);
  cr.resc = smem_u32(smem + lay.resc);
  cr.R = ka.ring_bytes;
  pre = reinterpret_cast<int*>(smem + lay.pre);
  if (ka.scr_floats == 0) {  // the CUDA-core consumers' class-change factors (the unit plan's
                             // barriers order these writes before any read)
    float* t = reinterpret_cast<float*>(smem + lay.resc);
    for (int k = threadIdx.x; k < kRescaleFloats; k += blockDim.x) t[k] = rescale_entry(k);
  }
  if (threadIdx.x == 0) {
#pragma unroll 1
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&cr.full[i], 1);
      mbar_init(&cr.empty[i], kNcw);
    }
    mbar_init(cr.ent_ready, kNcw);
    *cr.abort_flag = 0;
    fence_barrier_init();
  }
  // The unit plan reads only the call's own index arrays (sequence ids, positions,
  // modes, windows, bit-widths), which no kernel of this library writes, so it overlaps
  // the previous kernel of the stream.  The layer's cache state (metadata, pages, its
  // control words) is read before the wait only when `early` says that no kernel still
  // running can write it; everything else the previous kernel may write (query, K and V
  // rows, the pools' counters, scratch) is read after the producer's wait.
  plan_units(ka, P, NQB, pre, reinterpret_cast<long long*>(smem + lay.red));
  ent = reinterpret_cast<int*>(smem + lay.ent);
  if (!(STEP && ka.early)) pdl_wait();
  if (STEP && threadIdx.x >= 32) {  // the consumers build the entry table
    plan_entries(ka, ent);
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(cr.ent_ready);
  }
  return cr;
}

// The epilogue: the last CTA to finish records the error of the lowest failing query,
// readies the layer's counters for the next call and, for a decode step, commits the
// appended tokens' metadata.
template <bool STEP>
__device__ __forceinline__ void attn_epilogue(const AttnKernelArgs& ka, const int* ent) {
  const LayerArgs& a = ka.a;
  __shared__ int s_last, s_aborted;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&a.lctl[kDoneCtas], 1) == static_cast<int>(gridDim.x) - 1;
    if (s_last) {
      __threadfence();
      const int bad = atomicExch(&a.lctl[kFirstBadQuery], INT_MAX);
      if (bad != INT_MAX) set_status(a.ctrl, bad & 15);
      s_aborted = atomicExch(&a.lctl[kAborted], 0);
      atomicExch(&a.lctl[kNextUnit], 0);
      atomicExch(&a.lctl[kDoneCtas], 0);
    }
  }
  if (!STEP) return;
  __syncthreads();
  if (!s_last) return;
  const int* sc = ent + 6 * ka.n;
  if (sc[kSErr] != INT_MAX) {
    // a call error (some known only after the wait, when rows were already being
    // computed): every row zero, nothing for the combine kernel to merge
    uint4* o = reinterpret_cast<uint4*>(ka.out);
    const int64_t n16 = static_cast<int64_t>(ka.n) * a.Hq * a.d / 8;
    for (int64_t i = threadIdx.x; i < n16; i += blockDim.x) o[i] = make_uint4(0, 0, 0, 0);
    if (ka.defer_merge) {
      int2* qtab = reinterpret_cast<int2*>(a.cnt);
      for (int q = threadIdx.x; q < ka.n; q += blockDim.x) qtab[q] = make_int2(0, 1);
    }
  }
  if (!s_aborted) step_commit(ka, ent);  // a call that gave up a wait stores nothing
}

// CUDA-core path: units of kNcw query heads, one per consumer warp; HM: per-head modes
// (presence masks read with every page).
template <int D, int P, bool HM, bool STEP>
__global__ void __launch_bounds__(32 * (kNcw + 1), cc_ctas_per_sm(D))
    attn_kernel(const __grid_constant__ AttnKernelArgs ka) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int NQB = (ka.a.Hq + ka.hpu - 1) / ka.hpu;
  int *pre, *ent;
  const CtaRing cr = attn_prologue<STEP>(ka, smem, P, NQB, pre, ent);
  if (warp == 0) run_producer<D, STEP, HM>(ka, P, NQB, pre, ent, cr, lane);
  else run_consumer_cc<D, P, cc_elems(D), HM, STEP>(ka, cr, ent, warp - 1, lane);
  attn_epilogue<STEP>(ka, ent);
}

// Tensor-core path: units of kNcw KV heads with all their query heads.
template <int D, int NG, bool STEP>
__global__ void __launch_bounds__(32 * (kNcw + 1), kMmaCtasPerSm) attn_mma_kernel(const __grid_constant__ AttnKernelArgs ka) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int NQB = (ka.a.Hq + ka.hpu - 1) / ka.hpu;
  const int P = ka.a.P;
  int *pre, *ent;
  const CtaRing cr = attn_prologue<STEP>(ka, smem, P, NQB, pre, ent);
  if (warp == 0) {
    run_producer<D, STEP, false>(ka, P, NQB, pre, ent, cr, lane);
  } else {
    const AttnSmem lay(ka.ring_bytes, ka.n, ka.scr_floats, STEP);
    float* scr = reinterpret_cast<float*>(smem + lay.scr) + (warp - 1) * ka.scr_floats;
    run_consumer_mma<D, NG, STEP>(ka, cr, ent, P, warp - 1, lane, scr);
  }
  attn_epilogue<STEP>(ka, ent);
}

// ------------------------------------------------------------------ combine --
// Merges the split partials of every (query, head) of a tensor-core launch whose query
// has more than one split: one CTA of kCombineWarps warps per (query, head); warp w folds splits
// w, w + kCombineWarps, ... over its own maximum, then warp 0 folds the warps and
// writes the bf16 row.  Chained after the attention kernel (programmatic dependent
// launch): it reads nothing before that kernel has finished.
constexpr int kCombineWarps = 4;

struct CombineArgs {
  const float* part;  // [units][Hq][D + 4] partials of the launch
  const int2* qtab;   // [n] first partial and splits of each query (written by CTA 0 of the
                      // attention kernel, in the arrival-counter region it does not use)
  uint16_t* out;      // [n][Hq][D] bf16 rows of the launch
  int Hq;
};

template <int D>
__global__ void __launch_bounds__(32 * kCombineWarps) attn_combine_kernel(const __grid_constant__ CombineArgs ca) {
  constexpr int DPL = D / 32;
  __shared__ float sacc[kCombineWarps][D];
  __shared__ float sml[kCombineWarps][2];
  pdl_wait();
  pdl_trigger();
  const int qi = blockIdx.x / ca.Hq, qh = blockIdx.x - qi * ca.Hq;
  const int2 e = ca.qtab[qi];
  if (e.y <= 1) return;  // one split: written by the attention kernel
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t stride = static_cast<int64_t>(ca.Hq) * (D + 4);
  const float* p0 = ca.part + (static_cast<int64_t>(e.x) * ca.Hq + qh) * (D + 4) + warp * stride;
  const int64_t wstride = stride * kCombineWarps;  // between this warp's splits
  const int cnt = (e.y - warp + kCombineWarps - 1) / kCombineWarps;
  float Mx = kNegInf;
  for (int s = lane; s < cnt; s += 32) Mx = fmaxf(Mx, __ldcg(p0 + s * wstride + D));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) Mx = fmaxf(Mx, __shfl_xor_sync(0xffffffffu, Mx, o));
  float Ls = 0.f, acc[DPL];
#pragma unroll
  for (int j = 0; j < DPL; ++j) acc[j] = 0.f;
  for (int s0 = 0; s0 < cnt; s0 += 32) {
    float wl = 0.f;  // lane s: weight of split s0 + s of this warp
    if (s0 + lane < cnt) {
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(p0 + (s0 + lane) * wstride + D));
      wl = (ml.x == kNegInf) ? 0.f : fast_exp2(ml.x - Mx);
      Ls = fmaf(wl, ml.y, Ls);
    }
    const int m = min(32, cnt - s0);
#pragma unroll 8
    for (int s = 0; s < m; ++s) {
      const float wgt = __shfl_sync(0xffffffffu, wl, s);
      const float* ps = p0 + (s0 + s) * wstride + lane * DPL;
#pragma unroll
      for (int j = 0; j < DPL; ++j) acc[j] = fmaf(wgt, __ldcg(ps + j), acc[j]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, o);
#pragma unroll
  for (int j = 0; j < DPL; ++j) sacc[warp][lane * DPL + j] = acc[j];
  if (lane == 0) {
    sml[warp][0] = Mx;
    sml[warp][1] = Ls;
  }
  __syncthreads();
  if (warp != 0) return;
  float M = kNegInf;
#pragma unroll
  for (int w = 0; w < kCombineWarps; ++w) M = fmaxf(M, sml[w][0]);
  float L = 0.f, o[DPL];
#pragma unroll
  for (int j = 0; j < DPL; ++j) o[j] = 0.f;
#pragma unroll
  for (int w = 0; w < kCombineWarps; ++w) {
    const float f = sml[w][0] == kNegInf ? 0.f : fast_exp2(sml[w][0] - M);
    L = fmaf(f, sml[w][1], L);
#pragma unroll
    for (int j = 0; j < DPL; ++j) o[j] = fmaf(f, sacc[w][lane * DPL + j], o[j]);
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  uint16_t* orow = ca.out + (static_cast<int64_t>(qi) * ca.Hq + qh) * D + lane * DPL;
#pragma unroll
  for (int j = 0; j < DPL; j += 2)
    *reinterpret_cast<__nv_bfloat162*>(orow + j) = __floats2bfloat162_rn(o[j] * inv, o[j + 1] * inv);
}

// ------------------------------------------------------------- launchers --
// One translation unit per kernel family (compiled side by side): each launches its
// instances with programmatic dependent launch and sets their shared-memory limit.
//   attn_cc:          CUDA-core kernels of trr_decode_attn (one mode per query)
//   attn_head_modes:  CUDA-core kernels of caches with per-head modes
//   attn_mma:         tensor-core kernels of trr_decode_attn and the combine kernel
//   attn_step_cc / attn_step_mma: the decode-step kernels (trr_decode_step)
cudaError_t launch_attn_cc(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const AttnKernelArgs& k);
cudaError_t launch_attn_head_modes(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                   const AttnKernelArgs& k);
cudaError_t launch_attn_mma(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const AttnKernelArgs& k);
cudaError_t launch_attn_step_cc(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                const AttnKernelArgs& k);
cudaError_t launch_attn_step_mma(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                 const AttnKernelArgs& k);
cudaError_t launch_attn_combine(int d, dim3 grid, dim3 block, cudaStream_t s, const CombineArgs& ca);
cudaError_t configure_attn_cc();
cudaError_t configure_attn_head_modes();
cudaError_t configure_attn_mma();
cudaError_t configure_attn_step_cc();
cudaError_t configure_attn_step_mma();

}  // namespace trr
