/*
 * trr_oracle.c - plain, slow, fp64 CPU oracle for the TriRoute serving path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline / reference leg load this file's library.  It shares no source, header,
 * table or helper with the CUDA library; it re-derives the documented cache layout on
 * its own.  Every step follows the paper in order, with no blocking or fusion:
 *
 *   - quantiser Q_b (Sec. 3.2(C), Eq. 4): z = min(x), s = (max(x) - min(x)) / (2^b - 1),
 *     codes round((x - z) / s), stored code c dequantises to z + c*s; b = 16 keeps
 *     the native value.  Readings where the paper is silent: min/max are taken per
 *     group of G elements along the head dimension; s and z are stored as IEEE
 *     binary16, s computed as fp16(fl32(fl32(max - min) / (2^b - 1))); the code is
 *     round-half-to-even of the EXACT quotient (x - z) / s, clamped to [0, 2^b - 1],
 *     i.e. the index of the nearest of the levels z + c*s, ties to the even index;
 *     native precision is bf16.
 *   - attention modes (Sec. 3.2(A), Eq. 2): skip -> 0; local -> softmax attention over
 *     the last w positions t-w+1..t (w keys, the reading the cost model
 *     kappa_local ~ 2 d min(t, w) of Sec. 3.5 and Appendix C fixes); full -> over
 *     all positions <= t.  Only stored tokens take part.
 *   - hard decisions at inference, KV stored at the chosen width, paged cache
 *     (Sec. 3.8); grouping tokens by precision (Sec. 7) -> one width class per page.
 *   - the hard decision itself (arg max of the router's logits, Sec. 3.8) and the
 *     cost model of Sec. 3.5 / Appendix C evaluated at it (orc_route_decisions).
 *
 * Floating point: fl32(op) is computed as a double operation followed by a cast to
 * float.  For +, -, * and / of binary32 operands this double rounding is innocuous
 * (53 >= 2*24 + 2), so it equals a single binary32 round-to-nearest-even.
 * Attention is computed entirely in double.
 *
 * Parity status: every function here is pinned by tests (see tests/test_oracle_*.py).
 */
#include <fenv.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_INVALID_ARG 1
#define ORC_OUT_OF_MEMORY 2
#define ORC_OUT_OF_PAGES 3
#define ORC_BAD_POSITION 4
#define ORC_UNSUPPORTED 6
#define ORC_BAD_VALUE 7

static const int BITS_OF_CLASS[4] = {2, 4, 8, 16};

typedef struct orc_cache {
  int L, S, Hq, Hkv, d, G, P, maxctx, skip_writes_kv, no_pool, head_modes;
  int chunk_order;     /* 1: 8- and 16-bit code rows keep each 128-byte line's 16-byte
                          chunks in the documented permuted order (see stored_at) */
  int cap[4];
  int MP, W32;
  int32_t* last_pos;   /* [L][S] */
  int32_t* ntok;       /* [L][S][4] */
  uint32_t* presence;  /* [L][S][W32] */
  int32_t* page_table; /* [L][S][4][MP] */
  int32_t* page_first; /* [L][S][4][MP] */
  int32_t* page_last;  /* [L][S][4][MP] */
  int32_t next_page[4];
  int64_t hdr, tokb[4], slice[4], maskb, page_bytes[4];
  uint8_t* pool[4];
} orc_cache;

/* ------------------------------------------------------------------ numbers -- */

double orc_bf16_to_double(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

/* IEEE binary16: 1 sign, 5 exponent (bias 15), 10 fraction bits. */
double orc_f16_to_double(uint16_t h) {
  int sign = (h >> 15) & 1, e = (h >> 10) & 31, m = h & 1023;
  double v;
  if (e == 0)
    v = ldexp((double)m, -24);
  else if (e == 31)
    v = m ? NAN : INFINITY;
  else
    v = ldexp((double)(1024 + m), e - 25);
  return sign ? -v : v;
}

/* Round a finite double to the nearest binary16, ties to even. */
uint16_t orc_double_to_f16(double x) {
  uint16_t sign = (x < 0 || (x == 0 && signbit(x))) ? 0x8000 : 0;
  double a = fabs(x);
  if (a == 0) return sign;
  if (a < ldexp(1.0, -14)) { /* subnormal range: quantum 2^-24 */
    double r = nearbyint(ldexp(a, 24));
    return (uint16_t)(sign | (uint16_t)r); /* r == 1024 encodes the smallest normal */
  }
  int E;
  frexp(a, &E);                   /* a = f * 2^E, f in [0.5, 1) */
  double r = nearbyint(ldexp(a, 11 - E)); /* significand scaled to [1024, 2048] */
  if (r == 2048) { r = 1024; E += 1; }
  int biased = (E - 1) + 15;
  if (biased >= 31) return (uint16_t)(sign | 0x7C00); /* overflow -> inf */
  return (uint16_t)(sign | (biased << 10) | ((int)r - 1024));
}

static double fl32(double x) { return (double)(float)x; }

/* -------------------------------------------------------------- quantiser -- */

/* Eq. 4 for one group of G bf16 values: writes binary16 bits of s and z and one
 * unpacked code per element.  Returns 1 (and all zeros) when the group holds a
 * non-finite value or one with |x| > 65504, which binary16 cannot carry. */
int orc_quantize_group(const uint16_t* x, int G, int b, uint16_t* s16, uint16_t* z16,
                       uint8_t* codes) {
  int i;
  double mn = INFINITY, mx = -INFINITY;
  for (i = 0; i < G; i++) {
    double xi = orc_bf16_to_double(x[i]);
    if (!isfinite(xi) || fabs(xi) > 65504.0) {
      *s16 = 0;
      *z16 = 0;
      memset(codes, 0, (size_t)G);
      return 1;
    }
    if (xi < mn) mn = xi;
    if (xi > mx) mx = xi;
  }
  int levels = (1 << b) - 1;
  uint16_t zb = orc_double_to_f16(mn);                 /* z = min(x) */
  double range = fl32(mx - mn);                         /* max(x) - min(x) */
  uint16_t sb = orc_double_to_f16(fl32(range / (double)levels)); /* s */
  double z = orc_f16_to_double(zb), s = orc_f16_to_double(sb);
  for (i = 0; i < G; i++) {
    /* round((x - z) / s) on the exact quotient, clamped to the levels: walk up the
     * levels z + c*s while x lies above the midpoint between level c and level c+1
     * (or on it with c odd, so that a tie ends on the even level).  The midpoint
     * z + (c + 1/2) s is exact in double: z and s are binary16, so it is a multiple
     * of 2^-25 below 2^18.  x is a bf16 value, exact in double, so every comparison is
     * exact.  With s = 0 every level is z and the code is 0. */
    double xi = orc_bf16_to_double(x[i]);
    int c = 0;
    if (s != 0) {
      while (c < levels) {
        double mid = z + ((double)c + 0.5) * s;
        if (xi > mid || (xi == mid && (c & 1))) c++;
        else break;
      }
    }
    codes[i] = (uint8_t)c;
  }
  *s16 = sb;
  *z16 = zb;
  return 0;
}

/* Pack n codes of b bits, least significant bits first. */
void orc_pack_codes(const uint8_t* codes, int n, int b, uint8_t* out) {
  int j;
  memset(out, 0, (size_t)(n * b / 8));
  for (j = 0; j < n; j++) {
    int bit = j * b;
    out[bit / 8] |= (uint8_t)(codes[j] << (bit % 8));
  }
}

static int unpack_code(const uint8_t* packed, int j, int b) {
  int bit = j * b;
  return (packed[bit / 8] >> (bit % 8)) & ((1 << b) - 1);
}

/* ------------------------------------------------------------------ layout -- */

static int64_t roundup(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

static int class_of_bits(int b) {
  int c;
  for (c = 0; c < 4; c++)
    if (BITS_OF_CLASS[c] == b) return c;
  return -1;
}

static int64_t idx_ls(const orc_cache* o, int l, int s) { return (int64_t)l * o->S + s; }
static int64_t idx_lsc(const orc_cache* o, int l, int s, int c) {
  return idx_ls(o, l, s) * 4 + c;
}
static int64_t idx_pt(const orc_cache* o, int l, int s, int c, int k) {
  return idx_lsc(o, l, s, c) * o->MP + k;
}

static uint8_t* page_ptr(const orc_cache* o, int c, int id) {
  return o->pool[c] + (int64_t)id * o->page_bytes[c];
}

/* Mode of query head h of entry i (modes are [n] or, with head_modes, [n][Hq]). */
static int mode_of(const orc_cache* o, const uint8_t* modes, int i, int h) {
  return o->head_modes ? modes[(int64_t)i * o->Hq + h] : modes[i];
}

/* Whether entry i stores KV for KV head j: always when skip tokens store KV, otherwise
 * when one of the query heads reading KV head j (h / (Hq / Hkv) = j) is not skip. */
static int head_stores(const orc_cache* o, const uint8_t* modes, int i, int j) {
  int g = o->Hq / o->Hkv, h;
  if (o->skip_writes_kv) return 1;
  for (h = j * g; h < (j + 1) * g; h++)
    if (mode_of(o, modes, i, h) != 0) return 1;
  return 0;
}

/* Whether entry i takes a slot: some KV head of it is stored. */
static int entry_stores(const orc_cache* o, const uint8_t* modes, int i) {
  int j;
  for (j = 0; j < o->Hkv; j++)
    if (head_stores(o, modes, i, j)) return 1;
  return 0;
}

/* With head_modes, KV head j's 64-bit presence mask (little-endian): the first 8 of the
 * 16 bytes that end its slice of the page. */
static uint8_t* mask_ptr(const orc_cache* o, const uint8_t* page, int c, int j) {
  return (uint8_t*)page + o->hdr + (int64_t)j * o->slice[c] + o->slice[c] - o->maskb;
}

/* With head_modes, the bit of `slot` in KV head j's presence mask. */
static int slot_present(const orc_cache* o, const uint8_t* page, int c, int slot, int j) {
  uint64_t m;
  if (!o->head_modes) return 1;
  memcpy(&m, mask_ptr(o, page, c, j), 8);
  return (int)((m >> slot) & 1);
}

/* cfg: L, S, Hq, Hkv, d, G, P, max_context, cap[4], skip_writes_kv, no_pool, head_modes.
 * With no_pool = 1 only metadata and nothing of the page bytes is kept.  head_modes = 1:
 * attention modes are chosen per query head (Sec. 3.2(A): per head by default), modes
 * arrays are [n][Hq], and every KV head's slice of a page ends with 16 bytes holding its
 * 64-bit presence mask (then 8 zero bytes). */
int orc_create(const int32_t* cfg, orc_cache** out) {
  int c;
  *out = NULL;
  if (fegetround() != FE_TONEAREST) return ORC_UNSUPPORTED;
  orc_cache* o = (orc_cache*)calloc(1, sizeof(orc_cache));
  if (!o) return ORC_OUT_OF_MEMORY;
  o->L = cfg[0]; o->S = cfg[1]; o->Hq = cfg[2]; o->Hkv = cfg[3];
  o->d = cfg[4]; o->G = cfg[5]; o->P = cfg[6]; o->maxctx = cfg[7];
  for (c = 0; c < 4; c++) o->cap[c] = cfg[8 + c];
  o->skip_writes_kv = cfg[12];
  o->no_pool = cfg[13];
  o->head_modes = cfg[14];
  if (o->L < 1 || o->S < 1 || o->Hkv < 1 || o->Hq < o->Hkv || o->Hq % o->Hkv ||
      (o->d != 64 && o->d != 128) || (o->G != 32 && o->G != 64 && o->G != 128) ||
      o->G > o->d || (o->P != 16 && o->P != 32 && o->P != 64) || o->maxctx < 1 ||
      o->cap[0] < 0 || o->cap[1] < 0 || o->cap[2] < 0 || o->cap[3] < 0 ||
      (o->head_modes != 0 && o->head_modes != 1)) {
    free(o);
    return ORC_UNSUPPORTED;
  }
  o->MP = (o->maxctx + o->P - 1) / o->P;
  o->W32 = (o->maxctx + 31) / 32;
  o->hdr = roundup(4 * (int64_t)o->P, 128);
  o->maskb = o->head_modes ? 16 : 0;
  {
    /* The documented rule: the permuted chunk order applies to every cache except those
     * read by the tensor-core path, i.e. query groups of g >= 2 whose g * (d / G)
     * (head, group) columns fit 8, without per-head modes. */
    int g = o->Hq / o->Hkv, cols = g * (o->d / o->G);
    o->chunk_order = (!o->head_modes && g >= 2 && cols <= 8) ? 0 : 1;
  }
  for (c = 0; c < 4; c++) {
    int b = BITS_OF_CLASS[c];
    o->tokb[c] = b < 16 ? 2 * (o->d * b / 8) + 2 * (o->d / o->G) * 4 : 4 * o->d;
    o->slice[c] = o->P * o->tokb[c] + o->maskb;
    o->page_bytes[c] = roundup(o->hdr + o->Hkv * o->slice[c], 128);
  }
  int64_t nls = (int64_t)o->L * o->S;
  o->last_pos = (int32_t*)malloc(sizeof(int32_t) * nls);
  o->ntok = (int32_t*)calloc((size_t)(nls * 4), sizeof(int32_t));
  o->presence = (uint32_t*)calloc((size_t)(nls * o->W32), sizeof(uint32_t));
  o->page_table = (int32_t*)malloc(sizeof(int32_t) * nls * 4 * o->MP);
  o->page_first = (int32_t*)malloc(sizeof(int32_t) * nls * 4 * o->MP);
  o->page_last = (int32_t*)malloc(sizeof(int32_t) * nls * 4 * o->MP);
  int fail = !o->last_pos || !o->ntok || !o->presence || !o->page_table ||
             !o->page_first || !o->page_last;
  for (c = 0; c < 4 && !fail && !o->no_pool; c++) {
    o->pool[c] = (uint8_t*)calloc((size_t)(o->cap[c] > 0 ? o->cap[c] : 1),
                                  (size_t)o->page_bytes[c]);
    if (!o->pool[c]) fail = 1;
  }
  *out = o;
  if (fail) return ORC_OUT_OF_MEMORY;
  int64_t i;
  for (i = 0; i < nls; i++) o->last_pos[i] = -1;
  for (i = 0; i < nls * 4 * o->MP; i++) {
    o->page_table[i] = -1;
    o->page_first[i] = -1;
    o->page_last[i] = -1;
  }
  return ORC_OK;
}

void orc_destroy(orc_cache* o) {
  int c;
  if (!o) return;
  free(o->last_pos); free(o->ntok); free(o->presence);
  free(o->page_table); free(o->page_first); free(o->page_last);
  for (c = 0; c < 4; c++) free(o->pool[c]);
  free(o);
}

/* ------------------------------------------------------------------ append -- */

/* Checks of one entry against the running state, in the documented order.
 * tmp_last / tmp_ntok / tmp_next describe the cache as if earlier entries of this
 * call had been applied. */
static int check_entry(const orc_cache* o, int seq, int pos, int bits, const uint8_t* modes,
                       int i, const int32_t* tmp_last, const int32_t* tmp_ntok,
                       const int32_t* tmp_next) {
  int h;
  if (seq < 0 || seq >= o->S) return ORC_INVALID_ARG;
  int c = class_of_bits(bits);
  if (c < 0) return ORC_INVALID_ARG;
  for (h = 0; h < (o->head_modes ? o->Hq : 1); h++)
    if (mode_of(o, modes, i, h) > 2) return ORC_INVALID_ARG;
  if (pos < 0 || pos >= o->maxctx) return ORC_BAD_POSITION;
  if (pos <= tmp_last[seq]) return ORC_BAD_POSITION;
  if (!entry_stores(o, modes, i)) return ORC_OK;
  if (tmp_ntok[seq * 4 + c] % o->P == 0 && tmp_next[c] >= o->cap[c]) return ORC_OUT_OF_PAGES;
  return ORC_OK;
}

/* The stored position of byte x of a KV slice (x counted from the slice's start) in an
 * 8- or 16-bit code region of a cache with the permuted chunk order: line n = x / 128
 * keeps its 16-byte chunk k = (x / 16) % 8 at chunk k XOR (n % 8) of the same line. */
static int64_t stored_at(const orc_cache* o, int b, int64_t x) {
  if (!o->chunk_order || b < 8) return x;
  int64_t n = x / 128, k = (x / 16) % 8;
  return n * 128 + (k ^ (n % 8)) * 16 + x % 16;
}

static void write_row(orc_cache* o, uint8_t* page, int c, int slot, int h,
                      const uint16_t* krow, const uint16_t* vrow, int* bad) {
  int b = BITS_OF_CLASS[c], d = o->d, G = o->G, P = o->P;
  uint8_t* sl = page + o->hdr + (int64_t)h * o->slice[c];
  int64_t j;
  uint8_t row[256]; /* one K or V code row in its logical byte order (d * b / 8 <= 256);
                       rows start on 16 bytes and are moved a 16-byte chunk at a time */
  if (b == 16) {
    for (int which = 0; which < 2; which++) {
      int64_t at = (int64_t)which * P * d * 2 + (int64_t)slot * d * 2;
      memcpy(row, which ? vrow : krow, (size_t)d * 2);
      for (j = 0; j < d * 2; j += 16) memcpy(sl + stored_at(o, b, at + j), row + j, 16);
    }
    return;
  }
  int rowb = d * b / 8, ng = d / G, which, g;
  uint8_t codes[128];
  for (which = 0; which < 2; which++) { /* 0 = K, 1 = V */
    const uint16_t* x = which ? vrow : krow;
    int64_t at = (int64_t)which * P * rowb + (int64_t)slot * rowb;
    uint8_t* szrow = sl + 2 * (int64_t)P * rowb + (int64_t)which * P * ng * 4 +
                     (int64_t)slot * ng * 4;
    memset(row, 0, sizeof(row));
    for (g = 0; g < ng; g++) {
      uint16_t s16, z16;
      *bad |= orc_quantize_group(x + g * G, G, b, &s16, &z16, codes);
      orc_pack_codes(codes, G, b, row + g * G * b / 8);
      memcpy(szrow + g * 4, &s16, 2); /* little-endian host, as on the GPU */
      memcpy(szrow + g * 4 + 2, &z16, 2);
    }
    for (j = 0; j < rowb; j += 16) memcpy(sl + stored_at(o, b, at + j), row + j, 16);
  }
}

int orc_append(orc_cache* o, int layer, int n, const int32_t* seq_ids,
               const int32_t* positions, const uint16_t* k, const uint16_t* v,
               const uint8_t* bits, const uint8_t* modes) {
  int i, c;
  if (layer < 0 || layer >= o->L || n < 0) return ORC_INVALID_ARG;
  if (n == 0) return ORC_OK;
  /* pass 1: validate every entry in order against a scratch copy of the state */
  int32_t* tmp_last = (int32_t*)malloc(sizeof(int32_t) * o->S);
  int32_t* tmp_ntok = (int32_t*)malloc(sizeof(int32_t) * o->S * 4);
  int32_t tmp_next[4];
  if (!tmp_last || !tmp_ntok) { free(tmp_last); free(tmp_ntok); return ORC_OUT_OF_MEMORY; }
  memcpy(tmp_last, o->last_pos + idx_ls(o, layer, 0), sizeof(int32_t) * o->S);
  memcpy(tmp_ntok, o->ntok + idx_lsc(o, layer, 0, 0), sizeof(int32_t) * o->S * 4);
  memcpy(tmp_next, o->next_page, sizeof(tmp_next));
  for (i = 0; i < n; i++) {
    int e = check_entry(o, seq_ids[i], positions[i], bits[i], modes, i, tmp_last,
                        tmp_ntok, tmp_next);
    if (e != ORC_OK) { free(tmp_last); free(tmp_ntok); return e; }
    tmp_last[seq_ids[i]] = positions[i];
    if (!entry_stores(o, modes, i)) continue;
    c = class_of_bits(bits[i]);
    if (tmp_ntok[seq_ids[i] * 4 + c] % o->P == 0) tmp_next[c]++;
    tmp_ntok[seq_ids[i] * 4 + c]++;
  }
  free(tmp_last);
  free(tmp_ntok);
  /* pass 2: apply */
  int bad = 0;
  int64_t row = (int64_t)o->Hkv * o->d;
  for (i = 0; i < n; i++) {
    int s = seq_ids[i], pos = positions[i];
    o->last_pos[idx_ls(o, layer, s)] = pos;
    if (!entry_stores(o, modes, i)) continue; /* skip: no KV entry */
    c = class_of_bits(bits[i]);
    int32_t* nt = &o->ntok[idx_lsc(o, layer, s, c)];
    int kidx = *nt / o->P, slot = *nt % o->P;
    if (slot == 0) {
      o->page_table[idx_pt(o, layer, s, c, kidx)] = o->next_page[c]++;
      o->page_first[idx_pt(o, layer, s, c, kidx)] = pos;
    }
    o->page_last[idx_pt(o, layer, s, c, kidx)] = pos;
    (*nt)++;
    o->presence[idx_ls(o, layer, s) * o->W32 + pos / 32] |= 1u << (pos % 32);
    if (o->no_pool) continue;
    uint8_t* page = page_ptr(o, c, o->page_table[idx_pt(o, layer, s, c, kidx)]);
    int32_t p32 = pos;
    memcpy(page + 4 * slot, &p32, 4);
    int h;
    for (h = 0; h < o->Hkv; h++)
      write_row(o, page, c, slot, h, k + i * row + (int64_t)h * o->d,
                v + i * row + (int64_t)h * o->d, &bad);
    /* head_modes: every KV head's row is written; the heads that store it get their
     * presence bit (a new page starts with every bit clear) */
    for (h = 0; h < o->Hkv && o->head_modes; h++) {
      uint8_t* mw = mask_ptr(o, page, c, h);
      uint64_t m;
      memcpy(&m, mw, 8);
      if (slot == 0) m = 0;
      if (head_stores(o, modes, i, h)) m |= (uint64_t)1 << slot;
      memcpy(mw, &m, 8);
    }
  }
  return bad ? ORC_BAD_VALUE : ORC_OK;
}

/* ---------------------------------------------------------------- dequant -- */

/* Dequantised K and V (head h) of the token in `slot` of a class-c page. */
static void dequant_slot(const orc_cache* o, const uint8_t* page, int c, int slot, int h,
                         double* kout, double* vout) {
  int b = BITS_OF_CLASS[c], d = o->d, G = o->G, P = o->P, j, which;
  const uint8_t* sl = page + o->hdr + (int64_t)h * o->slice[c];
  uint8_t r[256]; /* the row in its logical byte order */
  for (which = 0; which < 2; which++) {
    double* outv = which ? vout : kout;
    if (b == 16) {
      int64_t at = (int64_t)which * P * d * 2 + (int64_t)slot * d * 2, x;
      for (x = 0; x < d * 2; x += 16) memcpy(r + x, sl + stored_at(o, b, at + x), 16);
      for (j = 0; j < d; j++) {
        uint16_t h16;
        memcpy(&h16, r + 2 * j, 2);
        outv[j] = orc_bf16_to_double(h16);
      }
      continue;
    }
    int rowb = d * b / 8, ng = d / G;
    int64_t at = (int64_t)which * P * rowb + (int64_t)slot * rowb, x;
    for (x = 0; x < rowb; x += 16) memcpy(r + x, sl + stored_at(o, b, at + x), 16);
    const uint8_t* crow = r;
    const uint8_t* szrow = sl + 2 * (int64_t)P * rowb + (int64_t)which * P * ng * 4 +
                           (int64_t)slot * ng * 4;
    for (j = 0; j < d; j++) {
      uint16_t s16, z16;
      memcpy(&s16, szrow + (j / G) * 4, 2);
      memcpy(&z16, szrow + (j / G) * 4 + 2, 2);
      outv[j] = orc_f16_to_double(z16) + unpack_code(crow, j, b) * orc_f16_to_double(s16);
    }
  }
}

static int tokens_in_page(const orc_cache* o, int layer, int s, int c, int kidx) {
  int nt = o->ntok[idx_lsc(o, layer, s, c)];
  int left = nt - kidx * o->P;
  return left < o->P ? left : o->P;
}

static int32_t slot_position(const uint8_t* page, int slot) {
  int32_t p;
  memcpy(&p, page + 4 * slot, 4);
  return p;
}

/* Dequantised K/V of position pos of (layer, seq), KV head h.  Returns the class index
 * of the stored token, or -1 when the token is not stored. */
int orc_dequant_token(const orc_cache* o, int layer, int s, int pos, int h, double* kout,
                      double* vout) {
  int c, kidx, slot;
  if (o->no_pool) return -1;
  for (c = 0; c < 4; c++) {
    int np = (o->ntok[idx_lsc(o, layer, s, c)] + o->P - 1) / o->P;
    for (kidx = 0; kidx < np; kidx++) {
      const uint8_t* page = page_ptr(o, c, o->page_table[idx_pt(o, layer, s, c, kidx)]);
      int fill = tokens_in_page(o, layer, s, c, kidx);
      for (slot = 0; slot < fill; slot++)
        if (slot_position(page, slot) == pos) {
          if (!slot_present(o, page, c, slot, h)) return -1;
          dequant_slot(o, page, c, slot, h, kout, vout);
          return c;
        }
    }
  }
  return -1;
}

/* --------------------------------------------------------------- attention -- */

typedef struct { int c, kidx; } page_ref;

static uint64_t lcg_next(uint64_t* st) {
  *st = *st * 6364136223846793005ULL + 1442695040888963407ULL;
  return *st >> 33;
}

/* Eq. 2 for every query; out is [n][Hq][d] doubles.  order_seed != 0 visits the pages
 * (and the slots inside each page) in a pseudo-random order instead of page-table
 * order, which must not change the result beyond fp64 rounding. */
int orc_decode_attn(const orc_cache* o, int layer, int n, const int32_t* seq_ids,
                    const int32_t* q_positions, const uint16_t* q, const uint8_t* modes,
                    const int32_t* windows, int window_scalar, double scale,
                    uint64_t order_seed, double* out) {
  int i, h, j, status = ORC_OK;
  if (layer < 0 || layer >= o->L || n < 0) return ORC_INVALID_ARG;
  if (o->no_pool) return ORC_UNSUPPORTED;
  int d = o->d, group = o->Hq / o->Hkv;
  if (scale <= 0) scale = 1.0 / sqrt((double)d);
  page_ref* refs = (page_ref*)malloc(sizeof(page_ref) * 4 * (o->MP + 1));
  double* score = (double*)malloc(sizeof(double) * (o->maxctx + 1));
  double* kv = (double*)malloc(sizeof(double) * 2 * d);
  double* acc = (double*)malloc(sizeof(double) * d);
  double* qd = (double*)malloc(sizeof(double) * d);
  if (!refs || !score || !kv || !acc || !qd) {
    free(refs); free(score); free(kv); free(acc); free(qd);
    return ORC_OUT_OF_MEMORY;
  }
  for (i = 0; i < n; i++) {
    double* orow = out + (int64_t)i * o->Hq * d;
    int s = seq_ids[i], t = q_positions[i];
    int w = windows ? windows[i] : window_scalar;
    int err = ORC_OK, any_local = 0, any_read = 0;
    for (h = 0; h < o->Hq; h++) {
      int m = mode_of(o, modes, i, h);
      if (m > 2) err = ORC_INVALID_ARG;
      any_local |= m == 1;
      any_read |= m != 0;
    }
    if (s < 0 || s >= o->S) err = ORC_INVALID_ARG;
    else if (err == ORC_OK && (t < 0 || t >= o->maxctx)) err = ORC_BAD_POSITION;
    else if (err == ORC_OK && any_local && w < 1) err = ORC_INVALID_ARG;
    for (j = 0; j < o->Hq * d; j++) orow[j] = 0.0;
    if (err != ORC_OK) {
      if (status == ORC_OK) status = err;
      continue;
    }
    if (!any_read) continue; /* Attn^skip = 0 */
    /* the pages of this (layer, seq), all classes */
    int nref = 0, c, kidx;
    for (c = 0; c < 4; c++) {
      int np = (o->ntok[idx_lsc(o, layer, s, c)] + o->P - 1) / o->P;
      for (kidx = 0; kidx < np; kidx++) {
        refs[nref].c = c;
        refs[nref].kidx = kidx;
        nref++;
      }
    }
    uint64_t st = order_seed;
    if (order_seed) { /* Fisher-Yates shuffle of the visiting order */
      for (j = nref - 1; j > 0; j--) {
        int r = (int)(lcg_next(&st) % (uint64_t)(j + 1));
        page_ref tmp = refs[j];
        refs[j] = refs[r];
        refs[r] = tmp;
      }
    }
    for (h = 0; h < o->Hq; h++) {
      int kvh = h / group, r, nk = 0, slot, mode = mode_of(o, modes, i, h);
      if (mode == 0) continue; /* Attn^skip = 0 for this head */
      int lo = mode == 2 ? 0 : (t - w + 1 > 0 ? t - w + 1 : 0);
      for (j = 0; j < d; j++) qd[j] = orc_bf16_to_double(q[((int64_t)i * o->Hq + h) * d + j]);
      /* pass 1: scores of the stored keys lo <= j <= t, and their maximum */
      double mx = -INFINITY;
      for (r = 0; r < nref; r++) {
        int cc = refs[r].c, kk = refs[r].kidx;
        const uint8_t* page = page_ptr(o, cc, o->page_table[idx_pt(o, layer, s, cc, kk)]);
        int fill = tokens_in_page(o, layer, s, cc, kk);
        for (slot = 0; slot < fill; slot++) {
          int sl = order_seed ? fill - 1 - slot : slot;
          int32_t pos = slot_position(page, sl);
          if (pos < lo || pos > t || !slot_present(o, page, cc, sl, kvh)) continue;
          dequant_slot(o, page, cc, sl, kvh, kv, kv + d);
          double dot = 0;
          for (j = 0; j < d; j++) dot += qd[j] * kv[j];
          score[nk] = scale * dot;
          if (score[nk] > mx) mx = score[nk];
          nk++;
        }
      }
      if (nk == 0) continue; /* no stored token in range: zero row */
      /* pass 2: softmax weights and the weighted sum of V */
      double denom = 0;
      for (j = 0; j < d; j++) acc[j] = 0;
      nk = 0;
      for (r = 0; r < nref; r++) {
        int cc = refs[r].c, kk = refs[r].kidx;
        const uint8_t* page = page_ptr(o, cc, o->page_table[idx_pt(o, layer, s, cc, kk)]);
        int fill = tokens_in_page(o, layer, s, cc, kk);
        for (slot = 0; slot < fill; slot++) {
          int sl = order_seed ? fill - 1 - slot : slot;
          int32_t pos = slot_position(page, sl);
          if (pos < lo || pos > t || !slot_present(o, page, cc, sl, kvh)) continue;
          dequant_slot(o, page, cc, sl, kvh, kv, kv + d);
          double p = exp(score[nk] - mx);
          denom += p;
          for (j = 0; j < d; j++) acc[j] += p * kv[d + j];
          nk++;
        }
      }
      for (j = 0; j < d; j++) orow[(int64_t)h * d + j] = acc[j] / denom;
    }
  }
  free(refs); free(score); free(kv); free(acc); free(qd);
  return status;
}

/* -------------------------------------------------------------- inspection -- */

/* Region ids as in the library's documented layout: 0 last_pos, 1 ntok, 2 presence,
 * 3 page_table, 4 page_first, 5 page_last, 6 next_page, 7..10 pools (b = 2,4,8,16).
 * Returns the region's size in bytes and its host pointer. */
int64_t orc_region(orc_cache* o, int id, void** ptr) {
  int64_t nls = (int64_t)o->L * o->S;
  switch (id) {
    case 0: *ptr = o->last_pos; return 4 * nls;
    case 1: *ptr = o->ntok; return 16 * nls;
    case 2: *ptr = o->presence; return 4 * nls * o->W32;
    case 3: *ptr = o->page_table; return 16 * nls * o->MP;
    case 4: *ptr = o->page_first; return 16 * nls * o->MP;
    case 5: *ptr = o->page_last; return 16 * nls * o->MP;
    case 6: *ptr = o->next_page; return 16;
    case 7: case 8: case 9: case 10:
      *ptr = o->pool[id - 7];
      return o->pool[id - 7] ? (int64_t)o->cap[id - 7] * o->page_bytes[id - 7] : 0;
    default: *ptr = NULL; return -1;
  }
}

/* Layout sizes: which = 0 header bytes, 1..4 slice bytes of class 0..3,
 * 5..8 page bytes of class 0..3, 9 bytes that end each slice for its presence mask
 * (16 with head_modes, else 0). */
int64_t orc_layout(const orc_cache* o, int which) {
  if (which == 0) return o->hdr;
  if (which >= 1 && which <= 4) return o->slice[which - 1];
  if (which >= 5 && which <= 8) return o->page_bytes[which - 5];
  if (which == 9) return o->maskb;
  return -1;
}

/* ---------------------------------------------- hard decisions and their cost -- */

/* The hard decision of one controller head (Sec. 3.8: at inference the router takes
 * the arg max of its logits).  Readings where the paper is silent: the first of equal
 * maxima wins; a NaN logit is never the maximum; a row of NaN gives option 0.
 * Returned: the smallest i whose logit is a number no smaller than every other
 * logit that is a number. */
int orc_argmax(const float* z, int k) {
  int i, j;
  for (i = 0; i < k; i++) {
    int top = !isnan(z[i]);
    for (j = 0; j < k && top; j++)
      if (!isnan(z[j]) && z[j] > z[i]) top = 0;
    if (top) return i;
  }
  return 0;
}

/* Hard decisions of n tokens at one layer and what they cost.
 *   mode_logits [n][3]: options skip, local, full (the order of Sec. 3.2(A));
 *   bit_logits  [n][4]: options b = 2, 4, 8, 16 (Sec. 3.2(C)).
 * Cost of the one-hot policy (the cost model of Sec. 3.5 evaluated at the hard
 * decision, as Appendix C's expected_cost does with one-hot a and b):
 *   attention: for each of the Hq heads, 2 d per key interaction, and a query at
 *   0-indexed position p interacts with the positions it reads: full -> every j <= p,
 *   local -> those with j >= p - w + 1 as well (the w-key window), skip -> none.
 *   Appendix C charges at least one position; a negative p is charged as p = 0.
 *   memory: 2 d_kv b bits with d_kv = Hkv d (K and V of every KV head); a skip
 *   token that stores nothing (skip_writes_kv == 0) is charged 0.
 * totals (added to, not overwritten): [0] sum of attention costs, [1] sum of memory
 * costs, [2] the dense attention cost (every head full: 2 d Hq (p + 1)), [3] the
 * dense memory cost (2 d_kv 16), the normalisers C_dense of Appendix C. */
int orc_route_decisions(int n, const float* mode_logits, const float* bit_logits,
                        const int32_t* positions, int window, int Hq, int d, int Hkv,
                        int skip_writes_kv, uint8_t* modes, uint8_t* bits,
                        int64_t* attn_flops, int64_t* kv_bits, int64_t* totals) {
  int i;
  if (n < 0 || window < 1 || Hq < 1 || d < 1 || Hkv < 1) return ORC_INVALID_ARG;
  for (i = 0; i < n; i++) {
    int m = orc_argmax(mode_logits + 3 * (int64_t)i, 3);
    int b = BITS_OF_CLASS[orc_argmax(bit_logits + 4 * (int64_t)i, 4)];
    int64_t p = positions[i] < 0 ? 0 : positions[i];
    /* key interactions, counted one position at a time */
    int64_t keys = 0, dense_keys = 0, j;
    for (j = 0; j <= p; j++) {
      dense_keys++;
      if (m == 2 || (m == 1 && j >= p - window + 1)) keys++;
    }
    int64_t flops = (int64_t)Hq * 2 * d * keys;
    int64_t mem = (m == 0 && !skip_writes_kv) ? 0 : 2 * (int64_t)Hkv * d * b;
    modes[i] = (uint8_t)m;
    bits[i] = (uint8_t)b;
    attn_flops[i] = flops;
    kv_bits[i] = mem;
    totals[0] += flops;
    totals[1] += mem;
    totals[2] += (int64_t)Hq * 2 * d * dense_keys;
    totals[3] += 2 * (int64_t)Hkv * d * 16;
  }
  return ORC_OK;
}
