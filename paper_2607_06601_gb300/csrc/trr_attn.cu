// trr_attn.cu - trr_decode_attn: mode-routed split-K decode attention over the
// mixed-precision paged cache (Sec. 3.2(A), Eq. 2; Sec. 3.8; Sec. 7).
//
// Two kernels per call:
//   attn_plan_kernel  one warp per query.  Key range by mode (full: [0, t]; local:
//                     [t-w+1, t]; skip: none), the pages of each width class that
//                     intersect it (found from each page's first/last position), and
//                     the number of split-K work items from the bytes in range.  Skip
//                     queries and empty ranges get their zero rows here.
//   attn_kernel       persistent, one CTA per SM, every warp an independent worker.
//                     A warp takes one (query, head, split) item at a time, streams its
//                     pages through a private ring of shared-memory slots filled by 1-D
//                     bulk copies (cp.async.bulk + mbarrier), dequantises in registers
//                     (k = z + c*s folded as s*sum(q*c) + z*sum(q)), runs an online
//                     softmax per lane, merges lanes with shuffles, and either writes
//                     the bf16 row (one split) or a partial; the last split to finish
//                     merges the partials (no waiting: an atomic arrival counter).
#include <algorithm>
#include <climits>

#include "trr_internal.cuh"

namespace trr {

#define kNegInf (-__int_as_float(0x7f800000))

__global__ void __launch_bounds__(256) attn_plan_kernel(LayerArgs a, int n, const int32_t* __restrict__ seq_ids,
                                                        const int32_t* __restrict__ q_positions,
                                                        const uint8_t* __restrict__ modes,
                                                        const int32_t* __restrict__ windows, int window_scalar,
                                                        uint16_t* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int qi = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (blockIdx.x == 0 && threadIdx.x == 0) a.ctrl[kWorkCounter] = 0;
  if (qi >= n) return;
  const int seq = seq_ids[qi], t = q_positions[qi], mode = modes[qi];
  const int w = windows ? windows[qi] : window_scalar;
  int err = 0;
  if (seq < 0 || seq >= a.S || mode > TRR_MODE_FULL) err = TRR_ERR_INVALID_ARG;
  else if (t < 0 || t >= a.maxctx) err = TRR_ERR_BAD_POSITION;
  else if (mode == TRR_MODE_LOCAL && w < 1) err = TRR_ERR_INVALID_ARG;

  QueryPlan qp;
  qp.seq = seq;
  qp.err = err;
  qp.nsplit = 0;
  qp.lo = 0;
  qp.hi = t;
  qp.pad0 = qp.pad1 = qp.pad2 = 0;
  int64_t bytes = 0;
  int total_pages = 0;
  for (int c = 0; c < kClasses; ++c) {
    qp.first[c] = 0;
    qp.npages[c] = 0;
    qp.ntok[c] = 0;
  }
  if (!err && mode != TRR_MODE_SKIP) {
    const int lo = mode == TRR_MODE_FULL ? 0 : max(0, t - w + 1);
    qp.lo = lo;
    for (int c = 0; c < kClasses; ++c) {
      const int nt = a.ntok[seq * 4 + c];
      const int np = (nt + a.P - 1) / a.P;
      const int64_t row = static_cast<int64_t>(seq * 4 + c) * a.MP;
      int below = 0, upto = 0;  // pages ending before lo; pages starting at or before t
      for (int base = 0; base < np; base += 32) {
        const int kk = base + lane;
        const bool in = kk < np;
        const int pl = in ? a.plast[row + kk] : INT_MAX;
        const int pf = in ? a.pfirst[row + kk] : INT_MAX;
        below += __popc(__ballot_sync(0xffffffffu, in && pl < lo));
        upto += __popc(__ballot_sync(0xffffffffu, in && pf <= t));
      }
      qp.ntok[c] = nt;
      qp.first[c] = below;
      qp.npages[c] = max(0, upto - below);
      bytes += static_cast<int64_t>(qp.npages[c]) * a.slice[c];
      total_pages += qp.npages[c];
    }
    if (bytes > 0) {
      int64_t ns = (bytes + a.split_bytes - 1) / a.split_bytes;
      ns = min(ns, static_cast<int64_t>(a.s_cap));
      qp.nsplit = static_cast<int>(min(ns, static_cast<int64_t>(total_pages)));
    }
  }
  if (lane == 0) a.qplan[qi] = qp;
  if (qp.nsplit == 0) {  // skip, invalid or nothing stored in range: a zero row
    uint4* o = reinterpret_cast<uint4*>(out + static_cast<int64_t>(qi) * a.Hq * a.d);
    const int n16 = a.Hq * a.d / 8;
    for (int i = lane; i < n16; i += 32) o[i] = make_uint4(0, 0, 0, 0);
  }
  if (err && lane == 0) atomicMin(&a.ctrl[kFirstBadQuery], qi);
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// State of one lane: an online softmax over its keys (log2 domain) and the weighted
// sum of V over its 32 dimensions.  zacc collects p*z, the zero-point part of V.
struct LaneState {
  float m, l, zacc;
  float acc[32];
};

// Lazy rescaling: the running maximum moves only when a score exceeds it by more than
// kTau (log2 units), so p = 2^(score - m) stays below 2^kTau.
constexpr float kTau = 8.f;

__device__ __forceinline__ void softmax_step(LaneState& st, float score, float& p) {
  if (score > st.m + kTau) {
    const float alpha = exp2f(st.m - score);  // 0 when m = -inf
#pragma unroll
    for (int j = 0; j < 32; ++j) st.acc[j] *= alpha;
    st.l *= alpha;
    st.zacc *= alpha;
    st.m = score;
  }
  p = exp2f(score - st.m);
  st.l += p;
}

// One page of width class B in shared memory.  Lane -> (key kl, 32-dim part).
template <int D, int B>
__device__ __forceinline__ void consume_page(const uint8_t* sl, const int* spos, int P, int G, int fill,
                                             int lo, int hi, const float (&qf)[32], float sumq,
                                             LaneState& st, int lane) {
  constexpr int LPK = D / 32;   // lanes per key
  constexpr int KPI = 32 / LPK; // keys per pass
  const int part = lane % LPK, kl = lane / LPK;
  const int ng = D / G;
  const int grp = part * 32 / G;
  for (int it = 0; it < P / KPI; ++it) {
    const int key = it * KPI + kl;
    const int pos = spos[key];
    const bool valid = key < fill && pos >= lo && pos <= hi;
    float dot = 0.f;
    if (B == 16) {
      const uint4* kp = reinterpret_cast<const uint4*>(sl + (static_cast<int64_t>(key) * D + part * 32) * 2);
      float d0 = 0.f, d1 = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 u = kp[q];
        d0 = fmaf(qf[8 * q + 0], bf_lo(u.x), d0);
        d1 = fmaf(qf[8 * q + 1], bf_hi(u.x), d1);
        d0 = fmaf(qf[8 * q + 2], bf_lo(u.y), d0);
        d1 = fmaf(qf[8 * q + 3], bf_hi(u.y), d1);
        d0 = fmaf(qf[8 * q + 4], bf_lo(u.z), d0);
        d1 = fmaf(qf[8 * q + 5], bf_hi(u.z), d1);
        d0 = fmaf(qf[8 * q + 6], bf_lo(u.w), d0);
        d1 = fmaf(qf[8 * q + 7], bf_hi(u.w), d1);
      }
      dot = d0 + d1;
    } else {
      constexpr int rowb = D * B / 8;
      constexpr int WORDS = B;  // 32 codes of B bits
      constexpr int PER = 32 / B;
      const uint32_t* kc = reinterpret_cast<const uint32_t*>(sl + key * rowb + part * 4 * B);
      uint32_t wv[WORDS];
#pragma unroll
      for (int w = 0; w < WORDS; ++w) wv[w] = kc[w];
      const uint32_t szw = *reinterpret_cast<const uint32_t*>(sl + 2 * P * rowb + (key * ng + grp) * 4);
      const float s = __half2float(__ushort_as_half(static_cast<unsigned short>(szw & 0xFFFF)));
      const float z = __half2float(__ushort_as_half(static_cast<unsigned short>(szw >> 16)));
      float d0 = 0.f, d1 = 0.f;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float cf = static_cast<float>((wv[j / PER] >> ((j % PER) * B)) & ((1u << B) - 1));
        if (j & 1) d1 = fmaf(qf[j], cf, d1);
        else d0 = fmaf(qf[j], cf, d0);
      }
      dot = fmaf(s, d0 + d1, z * sumq);
    }
#pragma unroll
    for (int o = 1; o < LPK; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    if (valid) {
      float p;
      softmax_step(st, dot, p);
      if (B == 16) {
        const uint4* vp =
            reinterpret_cast<const uint4*>(sl + (static_cast<int64_t>(P) * D + key * D + part * 32) * 2);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 u = vp[q];
          st.acc[8 * q + 0] = fmaf(p, bf_lo(u.x), st.acc[8 * q + 0]);
          st.acc[8 * q + 1] = fmaf(p, bf_hi(u.x), st.acc[8 * q + 1]);
          st.acc[8 * q + 2] = fmaf(p, bf_lo(u.y), st.acc[8 * q + 2]);
          st.acc[8 * q + 3] = fmaf(p, bf_hi(u.y), st.acc[8 * q + 3]);
          st.acc[8 * q + 4] = fmaf(p, bf_lo(u.z), st.acc[8 * q + 4]);
          st.acc[8 * q + 5] = fmaf(p, bf_hi(u.z), st.acc[8 * q + 5]);
          st.acc[8 * q + 6] = fmaf(p, bf_lo(u.w), st.acc[8 * q + 6]);
          st.acc[8 * q + 7] = fmaf(p, bf_hi(u.w), st.acc[8 * q + 7]);
        }
      } else {
        constexpr int rowb = D * B / 8;
        constexpr int PER = 32 / B;
        const uint32_t* vc = reinterpret_cast<const uint32_t*>(sl + P * rowb + key * rowb + part * 4 * B);
        uint32_t wv[B];
#pragma unroll
        for (int w = 0; w < B; ++w) wv[w] = vc[w];
        const uint32_t szw =
            *reinterpret_cast<const uint32_t*>(sl + 2 * P * rowb + P * ng * 4 + (key * ng + grp) * 4);
        const float s = __half2float(__ushort_as_half(static_cast<unsigned short>(szw & 0xFFFF)));
        const float z = __half2float(__ushort_as_half(static_cast<unsigned short>(szw >> 16)));
        const float ps = p * s;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float cf = static_cast<float>((wv[j / PER] >> ((j % PER) * B)) & ((1u << B) - 1));
          st.acc[j] = fmaf(ps, cf, st.acc[j]);
        }
        st.zacc = fmaf(p, z, st.zacc);
      }
    }
  }
}

struct AttnKernelArgs {
  LayerArgs a;
  int n;
  const uint16_t* q;
  uint16_t* out;
  float qscale;      // softmax scale * log2(e)
  int ns;            // ring slots per warp
  int slot_bytes;    // bytes of one slot (the largest slice)
  int base_bytes;    // shared bytes of the item-base table
};

template <int D>
__global__ void __launch_bounds__(256, 1) attn_kernel(const AttnKernelArgs ka) {
  constexpr int LPK = D / 32;
  const LayerArgs& a = ka.a;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int n = ka.n;
  int* s_base = reinterpret_cast<int*>(smem);  // [n + 1] first item of each query
  uint8_t* slots = smem + ka.base_bytes + static_cast<int64_t>(warp) * ka.ns * ka.slot_bytes;
  int* wpos = reinterpret_cast<int*>(smem + ka.base_bytes + static_cast<int64_t>(nwarps) * ka.ns * ka.slot_bytes) +
              warp * ka.ns * a.P;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + ka.base_bytes +
                                               static_cast<int64_t>(nwarps) * ka.ns * (ka.slot_bytes + 4 * a.P)) +
                   warp * ka.ns;

  // item bases: exclusive scan of nsplit * units over the queries
  {
    __shared__ int s_warp_sum[32];
    const int per = (n + blockDim.x - 1) / blockDim.x;
    const int i0 = threadIdx.x * per;
    int sum = 0;
    for (int i = i0; i < min(n, i0 + per); ++i) sum += a.qplan[i].nsplit * a.units;
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_warp_sum[warp] = incl;
    __syncthreads();
    int woff = 0;
    for (int w = 0; w < warp; ++w) woff += s_warp_sum[w];
    int run = woff + incl - sum;
    for (int i = i0; i < min(n, i0 + per); ++i) {
      s_base[i] = run;
      run += a.qplan[i].nsplit * a.units;
    }
    if (threadIdx.x == blockDim.x - 1) s_base[n] = woff + incl;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {  // status of the lowest invalid query
    const int bad = a.ctrl[kFirstBadQuery];
    if (bad != INT_MAX) {
      set_status(a.ctrl, a.qplan[bad].err);
      a.ctrl[kFirstBadQuery] = INT_MAX;
    }
  }
  if (lane == 0) {
    for (int i = 0; i < ka.ns; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
  }
  __syncthreads();
  const int total = s_base[n];
  const int group = a.Hq / a.Hkv;
  uint32_t gcount = 0;  // pages this warp has consumed so far (slot ring position)

  for (;;) {
    int item = 0;
    if (lane == 0) item = atomicAdd(&a.ctrl[kWorkCounter], 1);
    item = __shfl_sync(0xffffffffu, item, 0);
    if (item >= total) break;
    int qlo = 0, qhi = n - 1;  // the query whose items contain `item`
    while (qlo < qhi) {
      const int mid = (qlo + qhi + 1) >> 1;
      if (s_base[mid] <= item) qlo = mid;
      else qhi = mid - 1;
    }
    const int qi = qlo;
    const QueryPlan& qp = a.qplan[qi];
    const int nsplit = qp.nsplit, seq = qp.seq, lo = qp.lo, hi = qp.hi;
    const int local = item - s_base[qi];
    const int unit = local / nsplit, split = local % nsplit;
    const int qh = unit, kvh = qh / group;
    int cb[kClasses], cum[kClasses + 1], ntk[kClasses];
    cum[0] = 0;
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      const int np = qp.npages[c];
      cb[c] = qp.first[c] + static_cast<int>(static_cast<int64_t>(split) * np / nsplit);
      const int ce = qp.first[c] + static_cast<int>(static_cast<int64_t>(split + 1) * np / nsplit);
      cum[c + 1] = cum[c] + (ce - cb[c]);
      ntk[c] = qp.ntok[c];
    }
    const int T = cum[kClasses];
    const int64_t ptrow = static_cast<int64_t>(seq) * 4 * a.MP;

    // query: this lane's 32 dimensions, scaled into the log2 domain
    const int part = lane % LPK;
    float qf[32];
    float sumq = 0.f;
    {
      const uint4* qp4 = reinterpret_cast<const uint4*>(ka.q + (static_cast<int64_t>(qi) * a.Hq + qh) * D + part * 32);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 u = qp4[q];
        qf[8 * q + 0] = bf_lo(u.x) * ka.qscale;
        qf[8 * q + 1] = bf_hi(u.x) * ka.qscale;
        qf[8 * q + 2] = bf_lo(u.y) * ka.qscale;
        qf[8 * q + 3] = bf_hi(u.y) * ka.qscale;
        qf[8 * q + 4] = bf_lo(u.z) * ka.qscale;
        qf[8 * q + 5] = bf_hi(u.z) * ka.qscale;
        qf[8 * q + 6] = bf_lo(u.w) * ka.qscale;
        qf[8 * q + 7] = bf_hi(u.w) * ka.qscale;
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) sumq += qf[j];
    }
    LaneState st;
    st.m = kNegInf;
    st.l = 0.f;
    st.zacc = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j) st.acc[j] = 0.f;

    // page ids of flat pages [wbase, wbase + 32), one per lane
    auto class_of_flat = [&](int f) { return (f >= cum[1]) + (f >= cum[2]) + (f >= cum[3]); };
    int wbase = 0, wid = -1;
    auto load_window = [&](int base) {
      const int f = base + lane;
      wid = -1;
      if (f < T) {
        const int c = class_of_flat(f);
        wid = a.pt[ptrow + c * a.MP + cb[c] + (f - cum[c])];
      }
    };
    load_window(0);
    auto issue = [&](int f) {  // warp-uniform: start the copy of flat page f
      if (f - wbase >= 32) {
        wbase += 32;
        load_window(wbase);
      }
      const int c = class_of_flat(f);
      const int id = __shfl_sync(0xffffffffu, wid, f - wbase);
      const uint32_t slot = (gcount + f) % ka.ns;
      if (lane == 0) {
        const uint8_t* page = a.pool[c] + static_cast<int64_t>(id) * a.page_bytes[c];
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&bars[slot], a.slice[c] + 4 * a.P);
        bulk_g2s(slots + slot * ka.slot_bytes, page + a.hdr + static_cast<int64_t>(kvh) * a.slice[c], a.slice[c],
                 &bars[slot]);
        bulk_g2s(wpos + slot * a.P, page, 4 * a.P, &bars[slot]);
      }
    };
    const int pre = min(T, ka.ns);
    for (int f = 0; f < pre; ++f) issue(f);
    bool timed_out = false;
    for (int f = 0; f < T; ++f) {
      const uint32_t g = gcount + f;
      const uint32_t slot = g % ka.ns;
      const bool arrived = mbar_wait(&bars[slot], (g / ka.ns) & 1);
      if (!__all_sync(0xffffffffu, arrived)) {  // give up together, never half a warp
        timed_out = true;
        // wait (bounded) for the copies still in flight, then give up on this kernel
        for (int r = f + 1; r < min(T, f + ka.ns); ++r) {
          const uint32_t g2 = gcount + r;
          mbar_wait(&bars[g2 % ka.ns], (g2 / ka.ns) & 1);
        }
        break;
      }
      const int c = class_of_flat(f);
      const int kidx = cb[c] + (f - cum[c]);
      const int fill = min(a.P, ntk[c] - kidx * a.P);
      const uint8_t* sl = slots + slot * ka.slot_bytes;
      const int* sp = wpos + slot * a.P;
      switch (c) {
        case 0: consume_page<D, 2>(sl, sp, a.P, a.G, fill, lo, hi, qf, sumq, st, lane); break;
        case 1: consume_page<D, 4>(sl, sp, a.P, a.G, fill, lo, hi, qf, sumq, st, lane); break;
        case 2: consume_page<D, 8>(sl, sp, a.P, a.G, fill, lo, hi, qf, sumq, st, lane); break;
        default: consume_page<D, 16>(sl, sp, a.P, a.G, fill, lo, hi, qf, sumq, st, lane); break;
      }
      __syncwarp();
      if (f + ka.ns < T) issue(f + ka.ns);
    }
    if (timed_out) {
      if (lane == 0) set_status(a.ctrl, TRR_ERR_TIMEOUT);
      return;
    }
    gcount += T;

    // merge the lanes that share a part: max, rescale, sum
    float M = st.m;
#pragma unroll
    for (int o = LPK; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float f = (st.m == kNegInf) ? 0.f : exp2f(st.m - M);
    float L = st.l * f;
#pragma unroll
    for (int o = LPK; o < 32; o <<= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      float x = (st.acc[j] + st.zacc) * f;
#pragma unroll
      for (int o = LPK; o < 32; o <<= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
      st.acc[j] = x;
    }
    const int64_t orow = (static_cast<int64_t>(qi) * a.Hq + qh) * D;
    if (nsplit == 1) {
      if (lane < LPK) {
        const float inv = L > 0.f ? 1.f / L : 0.f;
        uint4* o4 = reinterpret_cast<uint4*>(ka.out + orow + part * 32);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t w[4];
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const __nv_bfloat162 b2 = __floats2bfloat162_rn(st.acc[8 * q + 2 * h] * inv, st.acc[8 * q + 2 * h + 1] * inv);
            w[h] = *reinterpret_cast<const uint32_t*>(&b2);
          }
          o4[q] = make_uint4(w[0], w[1], w[2], w[3]);
        }
      }
      continue;
    }
    // several splits: store this one's partial, the last to arrive merges them all
    const int first_item = s_base[qi] + unit * nsplit;
    float* pp = a.part + static_cast<int64_t>(item) * (D + 4);
    if (lane < LPK) {
      float4* p4 = reinterpret_cast<float4*>(pp + part * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q) p4[q] = make_float4(st.acc[4 * q], st.acc[4 * q + 1], st.acc[4 * q + 2], st.acc[4 * q + 3]);
      if (lane == 0) {
        pp[D] = M;
        pp[D + 1] = L;
      }
    }
    __threadfence();
    __syncwarp();
    int last = 0;
    int32_t* counter = a.cnt + static_cast<int64_t>(qi) * a.units + unit;
    if (lane == 0) last = atomicAdd(counter, 1) == nsplit - 1;
    last = __shfl_sync(0xffffffffu, last, 0);
    if (!last) continue;
    __threadfence();
    constexpr int DPL = D / 32;  // dimensions per lane in the merge
    float Mx = kNegInf;
    for (int s = 0; s < nsplit; ++s) Mx = fmaxf(Mx, __ldcg(a.part + static_cast<int64_t>(first_item + s) * (D + 4) + D));
    float Ls = 0.f, o[DPL];
#pragma unroll
    for (int j = 0; j < DPL; ++j) o[j] = 0.f;
    for (int s = 0; s < nsplit; ++s) {
      const float* ps = a.part + static_cast<int64_t>(first_item + s) * (D + 4);
      const float ms = __ldcg(ps + D);
      const float wgt = (ms == kNegInf) ? 0.f : exp2f(ms - Mx);
      Ls = fmaf(wgt, __ldcg(ps + D + 1), Ls);
#pragma unroll
      for (int j = 0; j < DPL; ++j) o[j] = fmaf(wgt, __ldcg(ps + lane * DPL + j), o[j]);
    }
    const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
    for (int j = 0; j < DPL; j += 2) {
      const __nv_bfloat162 b2 = __floats2bfloat162_rn(o[j] * inv, o[j + 1] * inv);
      *reinterpret_cast<__nv_bfloat162*>(ka.out + orow + lane * DPL + j) = b2;
    }
    if (lane == 0) *counter = 0;
  }
}

constexpr int kAttnSmemLimit = 200 * 1024;  // dynamic shared memory of one attention CTA

// Done once per cache at creation, so that calls stay legal inside stream capture.
cudaError_t attn_configure() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmemLimit);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmemLimit);
  return e;
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
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const LayerArgs a = layer_args(l, cache_views(cache), layer);
  attn_plan_kernel<<<(n + 7) / 8, 256, 0, s>>>(a, n, seq_ids, q_positions, modes, windows, window_scalar,
                                               static_cast<uint16_t*>(out_bf16));
  AttnKernelArgs ka;
  ka.a = a;
  ka.n = n;
  ka.q = static_cast<const uint16_t*>(q_bf16);
  ka.out = static_cast<uint16_t*>(out_bf16);
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.f / sqrtf(static_cast<float>(l.d));
  ka.qscale = scale * 1.4426950408889634f;
  ka.ns = 4;
  ka.slot_bytes = static_cast<int>(l.slice[3]);
  ka.base_bytes = ((n + 1) * 4 + 127) / 128 * 128;
  const int per_warp = ka.ns * (ka.slot_bytes + 4 * l.P + 8);
  const int budget = kAttnSmemLimit - ka.base_bytes;
  const int nwarps = std::min(8, budget / per_warp);
  if (nwarps < 1) return TRR_ERR_UNSUPPORTED;
  const int smem = ka.base_bytes + nwarps * per_warp;
  const int grid = cache_num_sms(cache);
  if (l.d == 64)
    attn_kernel<64><<<grid, nwarps * 32, smem, s>>>(ka);
  else
    attn_kernel<128><<<grid, nwarps * 32, smem, s>>>(ka);
  cache_set_launches(cache, 2);
  return cudaGetLastError() == cudaSuccess ? TRR_OK : TRR_ERR_CUDA;
}
