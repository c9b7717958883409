/*
 * trr.h - C ABI of the TriRoute serving hot path on GB300 (sm_103a).
 *
 * TriRoute (arxiv 2607.06601) routes every token, at every layer, with a policy
 * pi_t = (a_t, e_t, b_t) (Sec. 3.1).  This library implements the inference-time
 * consumer of two of its axes:
 *   - a_t in {skip, local, full}: how much of the past the query reads
 *     (Sec. 3.2(A), Eq. 2);
 *   - b_t in {2, 4, 8, 16}: the bit-width at which the token's own K/V are written
 *     to the cache for later queries (Sec. 3.2(C), Eq. 4; 16 = native bf16).
 * At inference the decisions are hard (argmax), only the selected computation runs,
 * and each token's KV is stored at its chosen width in a paged cache (Sec. 3.8).
 * Sec. 7 names the two kernels a production system needs: mode-aware attention over
 * ragged skip/local/full work, and a mixed-precision paged KV cache that groups tokens
 * by precision.  Those are trr_decode_attn and trr_kv_append below.  The hard
 * decisions themselves (arg max of the router's logits) and their cost under the
 * model of Sec. 3.5 are trr_route_decisions; trr_kv_append_routed and
 * trr_decode_attn_routed take the same decisions inside their own kernels.
 *
 * Conventions shared by every entry point
 *   - Pointers marked "device" are CUDA device pointers on the current device; the
 *     library never takes ownership of them.  "host" pointers are read before return.
 *   - Every call is asynchronous and stream-ordered on `stream` (a cudaStream_t passed
 *     as void*; NULL = legacy default stream).  No call synchronises the device except
 *     trr_get_status and trr_destroy.
 *   - Host-detectable errors (NULL pointers, sizes out of range, layer out of range)
 *     return an error immediately and enqueue nothing.
 *   - Device-detectable errors (see trr_kv_append / trr_decode_attn) are recorded in a
 *     sticky device status word that keeps the FIRST error since it was last read;
 *     trr_get_status reads and clears it.  No kernel traps or asserts.
 *   - One stream at a time per cache: calls on the same cache must not overlap.
 *   - Kernels are launched with programmatic dependent launch.  The index arrays of a
 *     call (sequence ids, positions, bit-widths, modes, windows, router logits of the
 *     *_routed calls) are read while the previous kernel of the stream may still be
 *     running, so they must not be outputs of that kernel (produce them one kernel
 *     earlier, or copy them in from the host).  Query, K and V rows are read after it
 *     has finished.  A decode step (trr_decode_step) whose layer was not touched by the
 *     two calls enqueued before it on the cache also reads the layer's cache state early
 *     (see there); the other calls read the cache only after the previous kernel.
 *
 * Cache memory layout (fixed; the CPU oracle re-derives it independently)
 *   class index c = 0,1,2,3 <-> b = 2,4,8,16.   P = page_size, d = head_dim,
 *   G = group_size, Hkv = num_kv_heads, MP = ceil(max_context / P),
 *   W32 = ceil(max_context / 32).
 *   Metadata (int32 unless noted), all indexed [layer][seq]...:
 *     last_pos  [L][S]          last position appended to (layer, seq), -1 if none
 *     ntok      [L][S][4]       tokens of class c stored for (layer, seq)
 *     presence  [L][S][W32] u32 bit (p % 32) of word p / 32 set <=> token p is stored
 *     page_table[L][S][4][MP]   page ids of class c, in position order
 *     page_first[L][S][4][MP]   position of the first token of each page
 *     page_last [L][S][4][MP]   position of the last token of each page
 *     next_page [4]             pages handed out so far per class (bump allocator)
 *   Pools: class c holds pages_per_class[c] pages of PAGE_BYTES(b) bytes each:
 *     HDR        = roundup(4 * P, 128)           header: int32 positions[P]
 *     TOKB(b)    = 2*(d*b/8) + 2*(d/G)*4   (b < 16)  |  4*d   (b = 16)
 *     SLICE(b)   = P * TOKB(b) + MASKB          one KV head of one page
 *     MASKB      = 16 with head_modes, else 0
 *     PAGE_BYTES = roundup(HDR + Hkv * SLICE(b), 128)
 *     head h starts at HDR + h * SLICE(b); inside it, for b < 16:
 *       K codes [P][d*b/8] | V codes [P][d*b/8] | K sz [P][d/G][2] | V sz [P][d/G][2]
 *     where sz = (scale, zero) as IEEE binary16, and for b = 16:
 *       K [P][d] bf16 | V [P][d] bf16.
 *   Code packing: element j of a head vector sits at byte floor(j*b/8), bit (j*b) % 8,
 *   least significant bits first (2-bit codes 1,2,3,0 -> byte 0x39).
 *   Chunk order of 8- and 16-bit rows: in every cache except those of query groups
 *   g = Hq/Hkv >= 2 with g * (d/G) <= 8 and head_modes = 0, the K and V code regions of
 *   b = 8 and b = 16 slices store byte x of the slice (x counted from the slice's start,
 *   x < 2*P*d*b/8) at x' = 128*n + 16*(k XOR (n % 8)) + x % 16, where n = x / 128 and
 *   k = (x / 16) % 8: each 128-byte line keeps its 16-byte chunks in a permuted order
 *   (the order the attention's lanes read them without shared-memory bank conflicts).
 *   Everything else (b = 2 and 4, scales, positions, masks) is stored as above.
 *   Page allocation: entries are taken in array order; an entry of class c whose
 *   (layer, seq) has ntok % P == 0 opens page next_page[c]++ .
 *   Per-head modes (head_modes = 1): the last 16 bytes of KV head h's slice hold a
 *   little-endian uint64 (then 8 zero bytes): bit `slot` set <=> the token in that slot
 *   stores KV head h.  A page starts with every bit clear when its slot 0 is written.
 */
#ifndef TRR_H
#define TRR_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define TRR_API __attribute__((visibility("default")))
#else
#define TRR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  TRR_OK = 0,
  TRR_ERR_INVALID_ARG = 1,   /* bad pointer, size, enum value (bits, mode) or window */
  TRR_ERR_OUT_OF_MEMORY = 2, /* cudaMalloc failed or caller pool too small */
  TRR_ERR_OUT_OF_PAGES = 3,  /* a class pool is exhausted */
  TRR_ERR_BAD_POSITION = 4,  /* position outside [0, max_context) or not increasing */
  TRR_ERR_CUDA = 5,          /* a CUDA runtime call failed */
  TRR_ERR_UNSUPPORTED = 6,   /* configuration outside the supported set */
  TRR_ERR_BAD_VALUE = 7,     /* non-finite or |x| > 65504 value in a quantised group */
  TRR_ERR_TIMEOUT = 8        /* a bounded wait inside a kernel gave up */
} trr_status;

enum { TRR_MODE_SKIP = 0, TRR_MODE_LOCAL = 1, TRR_MODE_FULL = 2 }; /* a_t, Eq. 2 */

typedef struct trr_cache_config {
  int32_t num_layers;      /* L >= 1 */
  int32_t max_seqs;        /* S >= 1: sequence ids are 0 .. S-1 */
  int32_t num_q_heads;     /* Hq, a multiple of num_kv_heads */
  int32_t num_kv_heads;    /* Hkv >= 1 */
  int32_t head_dim;        /* d: 64 or 128 */
  int32_t group_size;      /* G: 32, 64 or 128 with G <= d (quantiser group along d) */
  int32_t page_size;       /* P: 16, 32 or 64 tokens */
  int32_t max_context;     /* positions are 0 .. max_context-1 */
  int32_t pages_per_class[4]; /* pool capacity for b = 2, 4, 8, 16 */
  int32_t max_append;      /* largest n accepted by trr_kv_append */
  int32_t max_queries;     /* largest n accepted by trr_decode_attn */
  int32_t split_bytes;     /* least KV bytes (of 8-bit tokens) per split-K work item; 0 = 24576 */
  int32_t skip_writes_kv;  /* 0: a skip token stores no KV (default); 1: it stores KV */
  int32_t head_modes;      /* 0: one mode per token, modes[n] (default); 1: one mode per
                              query head, modes[n][Hq] (Sec. 3.2(A): per head by default),
                              with a presence mask per KV head in every page */
  void* pool;              /* device memory of >= trr_cache_required_bytes, or NULL */
  uint64_t pool_bytes;     /* size of `pool` (ignored when pool is NULL) */
} trr_cache_config;

typedef struct trr_cache trr_cache; /* opaque */

/* Bytes of device memory a cache with this configuration needs (metadata, scratch
 * and the four page pools).  Returns TRR_ERR_UNSUPPORTED / TRR_ERR_INVALID_ARG for a
 * configuration outside the supported set. */
TRR_API trr_status trr_cache_required_bytes(const trr_cache_config* cfg, uint64_t* bytes);

/* Create a cache on the current device.  With cfg->pool == NULL the library
 * cudaMallocs the memory and frees it in trr_destroy; otherwise it carves everything
 * out of the caller's buffer (>= trr_cache_required_bytes, 256-byte aligned), which
 * must outlive the cache.  All metadata starts empty.  Synchronous. */
TRR_API trr_status trr_create_cache(const trr_cache_config* cfg, trr_cache** out);

/* Quantise-on-write append (Sec. 3.2(C), Eq. 4; Sec. 3.8).
 *   n entries, taken in array order; entry i is token positions[i] of sequence
 *   seq_ids[i] at `layer`, with K/V rows k[i][Hkv][d], v[i][Hkv][d] (bf16, device,
 *   contiguous), bit-width bits[i] in {2,4,8,16} and attention mode modes[i].
 *   A skip token (modes[i] == 0) stores nothing unless skip_writes_kv == 1.
 *   With head_modes, modes is [n][Hq] (uint8, device): KV head j of entry i is stored
 *   when a query head reading it (h / (Hq / Hkv) == j) has a mode other than skip, or
 *   always with skip_writes_kv == 1; an entry none of whose KV heads is stored takes no
 *   slot.  An entry that takes a slot has every KV head's row written, and its slot's
 *   bit set in the presence mask of each KV head it stores.
 *   For b < 16 each group of G consecutive elements of a head vector is stored as
 *     z = fp16(min x),  s = fp16(fl32(fl32(max x - min x) / (2^b - 1))),
 *     c_j = clamp(rne((x_j - z) / s), 0, 2^b - 1)   (c_j = 0 when s == 0)
 *   with fl32 = IEEE binary32 round-to-nearest-even and rne taken on the EXACT quotient
 *   (c_j is the nearest level z + c*s, ties to the even c); b = 16 stores the bf16 bits.
 *   seq_ids, positions, k, v, bits, modes: device arrays; 0 <= n <= max_append.  They may
 *   be read while the previous kernel of the stream (a trr_* call) is still running:
 *   they must not be outputs of that call.
 *   Device-detected errors: seq id out of range or bits/mode not allowed
 *   (INVALID_ARG), a position outside [0, max_context) or not above the sequence's
 *   last one (BAD_POSITION), a pool running out (OUT_OF_PAGES).  Any of these makes
 *   the whole call a no-op and records the error of the lowest failing index.
 *   A quantised group holding a non-finite value or |x| > 65504 is stored as zeros
 *   and records BAD_VALUE; the rest of the call takes effect. */
TRR_API trr_status trr_kv_append(trr_cache* cache, int32_t layer, int32_t n,
                         const int32_t* seq_ids, const int32_t* positions,
                         const void* k_bf16, const void* v_bf16,
                         const uint8_t* bits, const uint8_t* modes, void* stream);

/* Mode-routed split-K decode attention over the mixed-precision cache (Eq. 2).
 *   n queries; query i belongs to sequence seq_ids[i] at position t = q_positions[i],
 *   has rows q[i][Hq][d] (bf16, device) and mode modes[i]:
 *     skip : out row = 0
 *     local: softmax attention over the stored tokens j with t-w+1 <= j <= t,
 *            w = windows[i] (or window_scalar when windows == NULL), w >= 1
 *     full : softmax attention over the stored tokens j <= t.
 *   With head_modes, modes is [n][Hq] and each query head h runs its own mode over the
 *   tokens that store its KV head (presence bit set); the window check applies when any
 *   head is local, and a mode value outside {0, 1, 2} in any head fails the query.
 *   Query head h reads KV head h / (Hq / Hkv).  Scores are softmax_scale * q.k
 *   (softmax_scale <= 0 means 1/sqrt(d)) with K/V dequantised as z + c*s; fp32
 *   accumulation, bf16 (round-to-nearest-even) output out[i][Hq][d] (device).
 *   A query with no stored token in range gets a zero row.
 *   Device-detected errors (seq id, mode or window invalid: INVALID_ARG; position
 *   outside [0, max_context): BAD_POSITION) zero that query's row and record the
 *   error of the lowest failing index; other queries are computed.
 *   seq_ids, q_positions, q, modes, windows, out: device; 0 <= n <= max_queries.
 *   seq_ids, q_positions, modes and windows may be read while the previous kernel of the
 *   stream (a trr_* call) is still running: they must not be outputs of that call. */
TRR_API trr_status trr_decode_attn(trr_cache* cache, int32_t layer, int32_t n,
                           const int32_t* seq_ids, const int32_t* q_positions,
                           const void* q_bf16, const uint8_t* modes,
                           const int32_t* windows, int32_t window_scalar,
                           float softmax_scale, void* out_bf16, void* stream);

/* One decode step of one layer in one kernel: trr_kv_append of the n entries followed by
 * trr_decode_attn of their queries at the same positions and modes (Sec. 3.8: at
 * inference each token's KV is stored at its chosen width b_t, Sec. 3.2(C) Eq. 4, and its
 * query attends in its mode a_t, Sec. 3.2(A) Eq. 2, over the cache including its own new
 * token).
 *   Entry i is token positions[i] of sequence seq_ids[i] (all distinct: one token per
 *   sequence) with K/V rows k[i][Hkv][d], v[i][Hkv][d] (bf16), bit-width bits[i] and mode
 *   modes[i], as trr_kv_append takes them; its query q[i][Hq][d] (bf16) attends at
 *   t = positions[i] in mode modes[i] with window windows[i] (or window_scalar) and
 *   writes out[i][Hq][d] (bf16), as trr_decode_attn does.  The results are those of the
 *   two calls in that order: the same page bytes and metadata, and attention over every
 *   stored token up to t in range, the entry's own token included.
 *   seq_ids, positions, k, v, bits, modes, q, windows, out: device arrays;
 *   0 <= n <= min(256, max_append, max_queries); k, v, q, out 16-byte aligned.  A cache
 *   with head_modes returns TRR_ERR_UNSUPPORTED.
 *   Errors are those of both calls, checked for the whole call before anything is
 *   stored: sequence id, bit-width or mode not allowed, a sequence named twice, or a
 *   local query with a window below 1 (INVALID_ARG); a position outside
 *   [0, max_context) or not above the sequence's last one (BAD_POSITION); a pool running
 *   out (OUT_OF_PAGES).  Any of these makes the call store nothing and write zero rows
 *   for every query, and records the error of the lowest failing entry.  A group that
 *   cannot be quantised (BAD_VALUE) is handled as trr_kv_append handles it.
 *   The index arrays (seq_ids, positions, bits, modes, windows) may be read while the
 *   previous kernel of the stream is still running: they must not be outputs of that
 *   kernel.  k, v and q are read after it has finished.  When neither of the two calls
 *   enqueued before this one on the cache was for the same layer, the kernel also reads
 *   the layer's cache state and starts its page copies before the previous kernel has
 *   finished; this relies on every kernel of the stream (the caller's included) not
 *   letting its successor start before its own predecessor has finished, which holds
 *   for kernels launched without programmatic dependent launch. */
TRR_API trr_status trr_decode_step(trr_cache* cache, int32_t layer, int32_t n, const int32_t* seq_ids,
                                   const int32_t* positions, const void* k_bf16, const void* v_bf16,
                                   const uint8_t* bits, const uint8_t* modes, const void* q_bf16,
                                   const int32_t* windows, int32_t window_scalar, float softmax_scale,
                                   void* out_bf16, void* stream);

/* trr_decode_attn without any per-call scratch in the cache's memory (this entry point
 * has no counterpart in the paper; it serves callers that cannot allocate).
 *   Same arguments, results and error contract as trr_decode_attn, but its scratch
 *   (control words, split arrival counters, fp32 partials) lives in one
 *   32 MiB array that the library declares as a static device variable: every GPU that
 *   loads the library holds it until the process exits, and no call allocates device
 *   memory.  This is for callers that must not call cudaMalloc at the point of the
 *   call, such as an engine running inside a fixed, fully reserved memory budget, and
 *   that need more queries per call than the cache's max_queries scratch was sized
 *   for: n is bounded by the array instead of by max_queries.
 *   The call needs 256 + n * Hq * (4 * (1 + ceil(S_cap / 16)) + S_cap * (4*d + 16))
 *   bytes (plus 256-byte rounding per region), with S_cap the most splits per query of
 *   this cache; a call above 32 MiB returns TRR_ERR_OUT_OF_MEMORY and launches nothing.
 *   The first call on a device looks up the array's device address (once per device,
 *   with that device current); make that first call before any stream capture.
 *   Every call clears what must start at zero and then overwrites the array, so calls
 *   that overlap on the GPU (on different streams, or from different caches) race;
 *   serialise them. */
TRR_API trr_status trr_decode_attn_static(trr_cache* cache, int32_t layer, int32_t n,
                                          const int32_t* seq_ids, const int32_t* q_positions,
                                          const void* q_bf16, const uint8_t* modes,
                                          const int32_t* windows, int32_t window_scalar,
                                          float softmax_scale, void* out_bf16, void* stream);

/* The router's hard decisions at inference and their cost (Sec. 3.8: the router takes
 * the arg max of its logits and only the selected computation runs; Sec. 3.5 cost
 * model, evaluated at the one-hot policy as Appendix C's expected_cost does).
 *   mode_logits[n][3] (options skip, local, full) and bit_logits[n][4] (options
 *   b = 2, 4, 8, 16): fp32, device.  Decision = index of the largest logit, the first
 *   of equal ones; a NaN logit is never chosen; a row of NaN gives option 0.
 *   Outputs (device, each may be NULL): modes[n], bits[n] (uint8, the values
 *   trr_kv_append / trr_decode_attn take); attn_flops[n] = Hq * 2 * d * kappa with
 *   kappa the key positions the query reads at 0-indexed position p = positions[i]:
 *   full p + 1, local min(p + 1, window), skip 0 (p < 0 is charged as p = 0);
 *   kv_bits[n] = 2 * Hkv * d * b bits (the cost model's 2 d_kv b), 0 for a skip token
 *   when skip_writes_kv == 0 (it stores nothing).
 *   totals[4] (int64, device, ADDED to, so that calls over layers and steps
 *   accumulate): sum of attn_flops, sum of kv_bits, the dense attention cost
 *   sum Hq * 2 * d * (p + 1) and the dense memory cost n * 2 * Hkv * d * 16, the
 *   normalisers of the budget fractions (Appendix C).
 *   positions, window >= 1 and the head shape are needed only when attn_flops,
 *   kv_bits or totals is given.  Float arrays 4-byte aligned, int64 arrays 8-byte.
 *   The logits and positions are read after the previous kernel of the stream has
 *   finished.  The outputs must not be passed to the very next trr_* call on the
 *   stream (trr_kv_append and trr_decode_attn read their index arrays while the
 *   previous kernel still runs): pass the logits to the *_routed calls instead, which
 *   decide the same way. */
TRR_API trr_status trr_route_decisions(int32_t n, const float* mode_logits, const float* bit_logits,
                                       const int32_t* positions, int32_t window, int32_t num_q_heads,
                                       int32_t head_dim, int32_t num_kv_heads, int32_t skip_writes_kv,
                                       uint8_t* modes, uint8_t* bits, int64_t* attn_flops,
                                       int64_t* kv_bits, int64_t* totals, void* stream);

/* trr_kv_append with each entry's mode and bit-width decided in the append's own
 * planning step from the router's logits, exactly as trr_route_decisions decides:
 * bit_logits[n][4] (b = 2, 4, 8, 16) and mode_logits[n][3] (skip, local, full), fp32,
 * device, 4-byte aligned.  Otherwise the same arguments, results and error contract as
 * trr_kv_append (the logits, like the other inputs, may be read while the previous
 * kernel of the stream is still running).  Decisions are per token: a cache with
 * head_modes returns TRR_ERR_UNSUPPORTED. */
TRR_API trr_status trr_kv_append_routed(trr_cache* cache, int32_t layer, int32_t n,
                                        const int32_t* seq_ids, const int32_t* positions,
                                        const void* k_bf16, const void* v_bf16,
                                        const float* bit_logits, const float* mode_logits,
                                        void* stream);

/* trr_decode_attn with each query's mode decided in the attention's planning step from
 * mode_logits[n][3] (skip, local, full; fp32, device, 4-byte aligned), exactly as
 * trr_route_decisions decides.  Otherwise the same as trr_decode_attn.  Decisions are
 * per token: a cache with head_modes returns TRR_ERR_UNSUPPORTED. */
TRR_API trr_status trr_decode_attn_routed(trr_cache* cache, int32_t layer, int32_t n,
                                          const int32_t* seq_ids, const int32_t* q_positions,
                                          const void* q_bf16, const float* mode_logits,
                                          const int32_t* windows, int32_t window_scalar,
                                          float softmax_scale, void* out_bf16, void* stream);

/* Free library-owned memory (waits for the device first).  A caller pool is not
 * freed.  NULL is accepted. */
TRR_API trr_status trr_destroy(trr_cache* cache);

/* Read and clear the sticky device status (synchronises `stream`).  After
 * TRR_ERR_TIMEOUT it also returns the cache's per-call counters to their start values
 * (on `stream`, before returning), so that later calls on the cache run normally. */
TRR_API trr_status trr_get_status(trr_cache* cache, void* stream);

/* Bound of every wait inside this cache's attention and decode-step kernels, in
 * nanoseconds of the GPU's global timer (0 = the default, 2 s; below 20000 the waiting
 * warps poll instead of suspending, so that the limit is kept).  A wait that runs out
 * makes its CTA stop, lets its copies in flight land, records TRR_ERR_TIMEOUT and
 * returns; the call's rows are then undefined and a decode step stores nothing.  No
 * kernel waits without a bound.  Host-side setting, read at each later call. */
TRR_API trr_status trr_set_wait_limit(trr_cache* cache, uint64_t nanoseconds);

/* Forget every sequence of every layer and return all pages to the pools
 * (stream-ordered; metadata only, page bytes are not cleared). */
TRR_API trr_status trr_reset(trr_cache* cache, void* stream);

/* Location of one layout region inside the cache's device memory, for inspection:
 * 0 last_pos, 1 ntok, 2 presence, 3 page_table, 4 page_first, 5 page_last,
 * 6 next_page, 7..10 pools of b = 2, 4, 8, 16.  *ptr is a device pointer. */
TRR_API trr_status trr_get_region(const trr_cache* cache, int32_t region, void** ptr,
                          uint64_t* bytes);

/* Number of SMs and kernels the last trr_decode_attn / trr_kv_append launched
 * (host-side bookkeeping, no synchronisation). */
TRR_API int32_t trr_last_launch_count(const trr_cache* cache);

#ifdef __cplusplus
}
#endif
#endif /* TRR_H */
