/*
 * pcs_oracle.c -- plain, slow, scalar CPU oracle for the PCS hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file: only the test-suite, the smoke check of __graft_entry__ and
 * the CPU-baseline leg of bench.py use it.  It shares no code, header, table
 * or constant generator with the CUDA library; every definition below is
 * written out from the paper (or, where the paper is silent, from the frozen
 * reading named in the comment) in the most direct form available.
 *
 * What the paper fixes and what it leaves open
 *   - The paper defines PCS, the partition H = PCS (+) Derivable and the
 *     checkpoint / restore / fork / delete contract with invariants I1-I4
 *     (Sec. 3, Definition 1 and "The contract").  At epsilon = 0 the
 *     acceptance test D <= epsilon is byte identity, so "must snapshot" is
 *     decided by comparing a buffer's content before and after a recompute
 *     (Sec. 3 "The partition"; Sec. 4 procedure FINGERPRINT, step 1).
 *   - It gives no hash, no pack format and no relevance formula.  Where
 *     it is silent this file fixes one reading (content fingerprint
 *     PCSFP64-v1, the PCS1 record layout, fixed-order fp32 cosine,
 *     (score, -index) ranking and the three k-rules), and each function
 *     states the reading it implements.
 *
 * Parity status of each function against the paper
 *   pcso_fmix              pinned: published SplitMix64 output vectors
 *   pcso_lane_value,       the paper prints no hash, so these are pinned to
 *   pcso_chunk_hash,       the frozen definition: a second statement of the
 *   pcso_fingerprint       lane chain vectorised over the 32 lanes (a chunk
 *                          viewed as u64[8][32][2]) with a top-down buffer
 *                          tree, equal bit for bit, and planted slips (rotation,
 *                          word order, seed, segment map) that it catches; and
 *                          to the definition's invariants (per-word bijection,
 *                          order and length sensitivity, aligned-group
 *                          decomposition) and brute force
 *   pcso_classify          pinned: seeded ground truth of which buffers changed
 *   pcso_score_f32         pinned: a second statement of the summation order
 *                          (lanes as a float32[blocks][32][8] view, numpy
 *                          binary32 steps), equal bit for bit, that catches a
 *                          lane map of e mod 32, a sequential sum and a folded
 *                          lane tree; within 1e-3 of the fp64 cosine
 *   pcso_score_f64         pinned: numpy cosine, closed forms (parallel,
 *                          antiparallel, orthogonal, scaled copies)
 *   pcso_topk              pinned: brute-force ranking on tiny inputs, ties
 *   pcso_k_*               pinned: Table tab:keepfrac frame counts (fraction
 *                          rule), budget inequality, closed forms
 *   pcso_pack/_restore     pinned: I1 round-trip after an excursion, I4
 *                          completeness, the paper's byte counts
 *                          (Table tab:pcs, Sec. 7.2 "Cross-check")
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Content fingerprint PCSFP64-v1 (reading of the "fingerprint" that decides */
/* must-snapshot vs recomputable, Sec. 4 step 1 at epsilon = 0).             */
/* ------------------------------------------------------------------------ */

#define PCSO_CHUNK_BYTES 4096u   /* one chunk                                */
#define PCSO_LANES 32u           /* lanes per chunk                          */
#define PCSO_SEGS_PER_LANE 8u    /* 16-byte segments owned by one lane       */

static const uint64_t PCSO_P = 0x9E3779B97F4A7C15ull;    /* odd multiplier  */
static const uint64_t PCSO_SEED = 0x5043534650363401ull; /* lane seed base  */

/* SplitMix64 finaliser (Steele, Lea & Flood, OOPSLA 2014). */
uint64_t pcso_fmix(uint64_t z)
{
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

static uint64_t rotl64(uint64_t x, unsigned r)
{
    return (x << r) | (x >> (64u - r));
}

/* comb(a, b) = fmix(a * P + rotl(b, 31)): the ordered two-input node. */
uint64_t pcso_comb(uint64_t a, uint64_t b)
{
    return pcso_fmix(a * PCSO_P + rotl64(b, 31));
}

/*
 * Fixed-order pairwise tree over a list: each level replaces items
 * (2i, 2i+1) by comb(item 2i, item 2i+1); an odd last item is carried to the
 * next level unchanged; the single survivor is the root.  n >= 1.
 */
uint64_t pcso_tree(const uint64_t *items, uint64_t n)
{
    uint64_t *v = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    uint64_t len = n, i, root;
    if (!v) return 0;
    memcpy(v, items, (size_t)n * sizeof(uint64_t));
    while (len > 1) {
        uint64_t next = 0;
        for (i = 0; i + 1 < len; i += 2) v[next++] = pcso_comb(v[i], v[i + 1]);
        if (len % 2 == 1) v[next++] = v[len - 1];
        len = next;
    }
    root = v[0];
    free(v);
    return root;
}

/* Little-endian 64-bit word at byte offset `off`; bytes at or past L are 0. */
static uint64_t word_at(const uint8_t *data, uint64_t L, uint64_t off)
{
    uint64_t w = 0;
    unsigned b;
    for (b = 0; b < 8; b++) {
        uint64_t pos = off + b;
        uint64_t byte = (pos < L) ? data[pos] : 0;
        w |= byte << (8u * b);
    }
    return w;
}

/*
 * Lane value a_l of chunk c: lane l owns 16-byte segments s = l + 32k
 * (k = 0..7), i.e. words 2s and 2s+1, visited in ascending order.
 */
uint64_t pcso_lane_value(const uint8_t *data, uint64_t L, uint64_t c, unsigned lane)
{
    uint64_t h = pcso_fmix(PCSO_SEED ^ (c * PCSO_LANES + lane));
    unsigned k, j;
    for (k = 0; k < PCSO_SEGS_PER_LANE; k++) {
        uint64_t seg = lane + PCSO_LANES * k;
        for (j = 0; j < 2; j++) {
            uint64_t w = word_at(data, L, c * PCSO_CHUNK_BYTES + 16u * seg + 8u * j);
            h = (rotl64(h, 23) ^ w) * PCSO_P;
        }
    }
    return pcso_fmix(h);
}

/*
 * Chunk hash x_c: the 32 lane values reduced by the lane tree
 *   for d = 1, 2, 4, 8, 16: v[l] = comb(v[l], v[l + d]) for l = 0 mod 2d.
 */
uint64_t pcso_chunk_hash(const uint8_t *data, uint64_t L, uint64_t c)
{
    uint64_t v[PCSO_LANES];
    unsigned l, d;
    for (l = 0; l < PCSO_LANES; l++) v[l] = pcso_lane_value(data, L, c, l);
    for (d = 1; d < PCSO_LANES; d *= 2)
        for (l = 0; l < PCSO_LANES; l += 2 * d) v[l] = pcso_comb(v[l], v[l + d]);
    return v[0];
}

/* Number of chunks of an L-byte buffer: max(1, ceil(L / 4096)). */
uint64_t pcso_n_chunks(uint64_t L)
{
    return L == 0 ? 1 : (L + PCSO_CHUNK_BYTES - 1) / PCSO_CHUNK_BYTES;
}

/* fp(buffer) = fmix(tree(x_0 .. x_{C-1}) ^ (L * P)). */
uint64_t pcso_fingerprint(const uint8_t *data, uint64_t L)
{
    uint64_t C = pcso_n_chunks(L), c, root;
    uint64_t *x = (uint64_t *)malloc((size_t)C * sizeof(uint64_t));
    if (!x) return 0;
    for (c = 0; c < C; c++) x[c] = pcso_chunk_hash(data, L, c);
    root = pcso_tree(x, C);
    free(x);
    return pcso_fmix(root ^ (L * PCSO_P));
}

/* Fingerprints of n buffers given as (pointer, length) pairs. */
void pcso_fingerprint_many(const uint8_t *const *ptrs, const uint64_t *lens, int32_t n,
                           uint64_t *fp_out)
{
    int32_t i;
    for (i = 0; i < n; i++) fp_out[i] = pcso_fingerprint(ptrs[i], lens[i]);
}

/*
 * Classification (Sec. 3 "The partition"; Sec. 4 FINGERPRINT step 1 at
 * epsilon = 0): a buffer whose content is not reproduced by the recompute is
 * non-derivable, i.e. must be snapshotted.  1 = must-snapshot, 0 = derivable.
 */
void pcso_classify(const uint64_t *fp_before, const uint64_t *fp_after, int32_t n,
                   uint8_t *must_snapshot)
{
    int32_t i;
    for (i = 0; i < n; i++) must_snapshot[i] = (fp_before[i] != fp_after[i]) ? 1 : 0;
}

/* ------------------------------------------------------------------------ */
/* Relevance score (Sec. 5, eviction by relevance; Sec. 7.5).  The paper     */
/* ranks bank frames by relevance to the return viewpoint but gives no      */
/* formula; the reading is cosine(query, key) in fp32 with a fixed order.    */
/* ------------------------------------------------------------------------ */

enum { PCSO_DT_F16 = 4, PCSO_DT_BF16 = 5 };

/* IEEE binary16 -> float, from the format's definition (exact). */
static float f16_value(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 0x1F;
    int m = h & 0x3FF;
    float v;
    if (e == 0)
        v = ldexpf((float)m, -24);                 /* subnormal: m * 2^-24 */
    else if (e == 31)
        v = (m == 0) ? INFINITY : NAN;
    else
        v = ldexpf((float)(1024 + m), e - 25);     /* (1 + m/1024) 2^(e-15) */
    return sign ? -v : v;
}

/* bfloat16 -> float: the upper half of a binary32. */
static float bf16_value(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static float elem_value(const uint16_t *v, int e, int dtype)
{
    return dtype == PCSO_DT_BF16 ? bf16_value(v[e]) : f16_value(v[e]);
}

/*
 * cos(q, k) in fp32 with the frozen order: lane l = floor(e / 8) mod 32 owns
 * element e; each lane accumulates s_l = s_l + q_e * k_e in ascending e
 * (separately rounded multiply and add), the 32 lane sums are reduced by the
 * lane tree s[l] = s[l] + s[l + d] (d = 1, 2, 4, 8, 16, l = 0 mod 2d); the
 * same for q.q and k.k; score = dot / (sqrt(qq) * sqrt(kk)), 0 if the
 * denominator is 0.  This is the precision that decides the kept set.
 */
float pcso_score_f32(const uint16_t *q, const uint16_t *key, int32_t D, int32_t dtype)
{
    float sd[PCSO_LANES], sq[PCSO_LANES], sk[PCSO_LANES];
    int32_t e;
    unsigned l, d;
    float den;
    for (l = 0; l < PCSO_LANES; l++) sd[l] = sq[l] = sk[l] = 0.0f;
    for (e = 0; e < D; e++) {
        float qe = elem_value(q, e, dtype), ke = elem_value(key, e, dtype);
        l = (unsigned)((e / 8) % PCSO_LANES);
        sd[l] = sd[l] + qe * ke;   /* built with -ffp-contract=off: the product */
        sq[l] = sq[l] + qe * qe;   /* is rounded to fp32 before the add        */
        sk[l] = sk[l] + ke * ke;
    }
    for (d = 1; d < PCSO_LANES; d *= 2)
        for (l = 0; l < PCSO_LANES; l += 2 * d) {
            sd[l] = sd[l] + sd[l + d];
            sq[l] = sq[l] + sq[l + d];
            sk[l] = sk[l] + sk[l + d];
        }
    den = sqrtf(sq[0]) * sqrtf(sk[0]);
    if (den == 0.0f) return 0.0f;
    return sd[0] / den;
}

/* Plain fp64 cosine: the mathematical value the fp32 score approximates. */
double pcso_score_f64(const uint16_t *q, const uint16_t *key, int32_t D, int32_t dtype)
{
    double dot = 0, qq = 0, kk = 0, den;
    int32_t e;
    for (e = 0; e < D; e++) {
        double qe = elem_value(q, e, dtype), ke = elem_value(key, e, dtype);
        dot += qe * ke;
        qq += qe * qe;
        kk += ke * ke;
    }
    den = sqrt(qq) * sqrt(kk);
    return den == 0 ? 0.0 : dot / den;
}

/* Scores of n keys (rows of D elements) against one query. */
void pcso_score_many(const uint16_t *q, const uint16_t *keys, int32_t n, int32_t D,
                     int32_t dtype, float *out32, double *out64)
{
    int32_t i;
    for (i = 0; i < n; i++) {
        if (out32) out32[i] = pcso_score_f32(q, keys + (size_t)i * D, D, dtype);
        if (out64) out64[i] = pcso_score_f64(q, keys + (size_t)i * D, D, dtype);
    }
}

/* ------------------------------------------------------------------------ */
/* Ranking (selection, never merging: Sec. 9, WorldTrace paragraph).         */
/* ------------------------------------------------------------------------ */

/* Order-preserving map float -> uint32; -0 ranks as +0, NaN ranks lowest. */
uint32_t pcso_ord32(float s)
{
    uint32_t u;
    if (isnan(s)) return 0;
    if (s == 0.0f) s = 0.0f;
    memcpy(&u, &s, sizeof u);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

/* Ranking key: higher score first, equal scores by lower entry index. */
uint64_t pcso_key64(float s, uint32_t idx)
{
    return ((uint64_t)pcso_ord32(s) << 32) | (uint64_t)(0xFFFFFFFFu - idx);
}

static int cmp_u64_desc(const void *a, const void *b)
{
    uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
    return (x < y) - (x > y);
}

static int cmp_i32_asc(const void *a, const void *b)
{
    int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

/*
 * Keep the k largest ranking keys of n entries by a full sort; write the kept
 * entry indices in ascending order (frames re-stacked in their original
 * order, Sec. 7.2 "Cross-check").  Returns the number kept = min(k, n).
 */
int32_t pcso_topk(const float *scores, int32_t n, int32_t k, int32_t *kept)
{
    uint64_t *keys;
    int32_t i, m = k < n ? k : n;
    if (m <= 0) return 0;
    keys = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    if (!keys) return -1;
    for (i = 0; i < n; i++) keys[i] = pcso_key64(scores[i], (uint32_t)i);
    qsort(keys, (size_t)n, sizeof(uint64_t), cmp_u64_desc);
    for (i = 0; i < m; i++) kept[i] = (int32_t)(0xFFFFFFFFu - (uint32_t)(keys[i] & 0xFFFFFFFFu));
    qsort(kept, (size_t)m, sizeof(int32_t), cmp_i32_asc);
    free(keys);
    return m;
}

/* ------------------------------------------------------------------------ */
/* How many entries each bank keeps (Sec. 7.5: under a binding host budget   */
/* every bank is pruned to the same fraction).                               */
/* ------------------------------------------------------------------------ */

/* Fixed cap: k_s = min(n_s, k_max). */
void pcso_k_fixed(const int32_t *n, int32_t count, int32_t k_max, int32_t *k)
{
    int32_t s;
    for (s = 0; s < count; s++) k[s] = n[s] < k_max ? n[s] : k_max;
}

/*
 * Host byte budget B: T = sum n_s * E_s.  If T <= B every bank is kept whole;
 * otherwise k_s = floor(n_s * B / T), so sum k_s E_s <= B and every bank keeps
 * the same fraction B / T, rounded down.
 */
void pcso_k_budget(const int32_t *n, const uint64_t *entry_bytes, int32_t count,
                   uint64_t budget, int32_t *k)
{
    unsigned __int128 T = 0;
    int32_t s;
    for (s = 0; s < count; s++) T += (unsigned __int128)(uint64_t)n[s] * entry_bytes[s];
    for (s = 0; s < count; s++) {
        if (T <= budget)
            k[s] = n[s];
        else
            k[s] = (int32_t)(((unsigned __int128)(uint64_t)n[s] * budget) / T);
    }
}

/* Retention fraction: k_s = frac * n_s rounded to nearest, ties to even. */
void pcso_k_fraction(const int32_t *n, int32_t count, double frac, int32_t *k)
{
    int32_t s;
    for (s = 0; s < count; s++) {
        double v = nearbyint(frac * (double)n[s]);
        if (v < 0) v = 0;
        if (v > n[s]) v = n[s];
        k[s] = (int32_t)v;
    }
}

/*
 * Global relevance threshold under one host byte budget (a variant of the
 * budgeted pruning of Sec. 7.5: instead of pruning every bank to the same
 * fraction, one score threshold is drawn across all banks, so a session with
 * more relevant frames keeps more of them).  All entries of all banks are
 * ranked together by (score desc, bank asc, index asc) -- the ranking key of
 * the entry's position in the bank-major concatenation -- and the longest
 * prefix of that order whose entry bytes sum to at most `budget` is kept.
 * scores: float[sum n] bank-major; kept: int32[sum n] capacity, written per
 * bank in ascending entry index; kept_off: int32[count + 1] offsets into kept.
 * Returns the number kept, -1 on allocation failure.
 */
int64_t pcso_prune_global(const float *scores, const int32_t *n, const uint64_t *entry_bytes,
                          int32_t count, uint64_t budget, int32_t *kept, int32_t *kept_off)
{
    uint64_t total = 0, *keys, j, m;
    uint8_t *keep;
    unsigned __int128 used = 0;
    int64_t written = 0;
    int32_t s, *bank_of;
    uint64_t pos;
    for (s = 0; s < count; s++) total += (uint64_t)n[s];
    keys = (uint64_t *)malloc((size_t)(total ? total : 1) * sizeof(uint64_t));
    keep = (uint8_t *)calloc((size_t)(total ? total : 1), 1);
    bank_of = (int32_t *)malloc((size_t)(total ? total : 1) * sizeof(int32_t));
    if (!keys || !keep || !bank_of) {
        free(keys);
        free(keep);
        free(bank_of);
        return -1;
    }
    pos = 0;
    for (s = 0; s < count; s++) {
        int32_t i;
        for (i = 0; i < n[s]; i++, pos++) {
            keys[pos] = pcso_key64(scores[pos], (uint32_t)pos);
            bank_of[pos] = s;
        }
    }
    qsort(keys, (size_t)total, sizeof(uint64_t), cmp_u64_desc);
    /* Walk the global order; stop at the first entry that does not fit. */
    m = 0;
    for (j = 0; j < total; j++) {
        uint64_t p = 0xFFFFFFFFu - (uint32_t)(keys[j] & 0xFFFFFFFFu);
        used += entry_bytes[bank_of[p]];
        if (used > budget) break;
        keep[p] = 1;
        m++;
    }
    /* Emit per bank, ascending entry index. */
    pos = 0;
    for (s = 0; s < count; s++) {
        int32_t i;
        kept_off[s] = (int32_t)written;
        for (i = 0; i < n[s]; i++, pos++)
            if (keep[pos]) kept[written++] = i;
    }
    kept_off[count] = (int32_t)written;
    free(keys);
    free(keep);
    free(bank_of);
    return (int64_t)m;
}

/* ------------------------------------------------------------------------ */
/* Snapshot record "PCS1": the storage format of one checkpointed session   */
/* (Sec. 3 "Boundary": storage owns serialisation; the layout is a frozen   */
/* reading).  Little-endian throughout.                                      */
/*   header 64 B: u32 magic, u16 version, u16 n_sections, u32 session_id,    */
/*     u32 kind, u64 total_bytes, u64 session_fp, 32 zero bytes             */
/*   n section entries of 64 B: u32 type, u32 dtype, u32 layer, u32 layout, */
/*     u64 offset, u64 bytes, u64 fp, u64 dim0, u64 dim1, u64 aux           */
/*   payloads at 256-byte aligned offsets; every padding byte is 0.         */
/* ------------------------------------------------------------------------ */

#define PCSO_MAGIC 0x31534350u
#define PCSO_VERSION 1u
#define PCSO_HEADER_BYTES 64u
#define PCSO_ENTRY_BYTES 64u
#define PCSO_ALIGN 256u

enum { PCSO_CONTIG = 0, PCSO_ROWS = 1, PCSO_RING = 2 };

/* One section of a session: where its bytes live and how they are laid out. */
typedef struct {
    uint32_t type, dtype, layer, layout;
    uint8_t *base;          /* pack: source; restore: target                */
    uint64_t bytes;         /* payload bytes                                */
    uint64_t row_bytes;     /* ROWS / RING: bytes per row                   */
    const int32_t *index;   /* ROWS: row ids (bytes / row_bytes of them);   */
                            /* RING: page table (window / page_rows ids)    */
    uint32_t ring_start;    /* RING: ring slot of logical row 0             */
    uint32_t window;        /* RING: ring slots                             */
    uint32_t page_rows;     /* RING: rows per page                          */
    uint32_t reserved;
    uint64_t dim0, dim1;    /* shape recorded in the section entry          */
} pcso_section;

static uint64_t round_up(uint64_t x, uint64_t a) { return (x + a - 1) / a * a; }

static void put_u16(uint8_t *p, uint16_t v) { p[0] = (uint8_t)v; p[1] = (uint8_t)(v >> 8); }
static void put_u32(uint8_t *p, uint32_t v)
{
    unsigned b;
    for (b = 0; b < 4; b++) p[b] = (uint8_t)(v >> (8 * b));
}
static void put_u64(uint8_t *p, uint64_t v)
{
    unsigned b;
    for (b = 0; b < 8; b++) p[b] = (uint8_t)(v >> (8 * b));
}
static uint32_t get_u32(const uint8_t *p)
{
    uint32_t v = 0;
    unsigned b;
    for (b = 0; b < 4; b++) v |= (uint32_t)p[b] << (8 * b);
    return v;
}
static uint64_t get_u64(const uint8_t *p)
{
    uint64_t v = 0;
    unsigned b;
    for (b = 0; b < 8; b++) v |= (uint64_t)p[b] << (8 * b);
    return v;
}

/* Byte offset of the first payload: header + table, rounded up to 256. */
uint64_t pcso_payload_start(int32_t n_sections)
{
    return round_up(PCSO_HEADER_BYTES + (uint64_t)PCSO_ENTRY_BYTES * (uint64_t)n_sections,
                    PCSO_ALIGN);
}

/* Record size: every payload starts on a 256-byte boundary, so does the end. */
uint64_t pcso_record_bytes(const pcso_section *s, int32_t n)
{
    uint64_t off = pcso_payload_start(n);
    int32_t i;
    for (i = 0; i < n; i++) off = round_up(off + s[i].bytes, PCSO_ALIGN);
    return off;
}

/* Address of row r of a ROWS or RING section (pack source / restore target). */
static uint8_t *row_address(const pcso_section *s, uint64_t r)
{
    if (s->layout == PCSO_ROWS)
        return s->base + (uint64_t)(uint32_t)s->index[r] * s->row_bytes;
    /* RING: logical row r lives in ring slot (start + r) mod window. */
    {
        uint64_t slot = ((uint64_t)s->ring_start + r) % s->window;
        uint64_t page = (uint64_t)(uint32_t)s->index[slot / s->page_rows];
        return s->base + (page * s->page_rows + slot % s->page_rows) * s->row_bytes;
    }
}

/* Copy one section's logical bytes into a contiguous payload. */
static void gather_section(const pcso_section *s, uint8_t *payload)
{
    uint64_t r, rows;
    if (s->layout == PCSO_CONTIG) {
        memcpy(payload, s->base, (size_t)s->bytes);
        return;
    }
    rows = s->bytes / s->row_bytes;
    for (r = 0; r < rows; r++)
        memcpy(payload + r * s->row_bytes, row_address(s, r), (size_t)s->row_bytes);
}

/* Copy a contiguous payload back to a section's (possibly scattered) bytes. */
static void scatter_section(const pcso_section *s, const uint8_t *payload)
{
    uint64_t r, rows;
    if (s->layout == PCSO_CONTIG) {
        memcpy(s->base, payload, (size_t)s->bytes);
        return;
    }
    rows = s->bytes / s->row_bytes;
    for (r = 0; r < rows; r++)
        memcpy(row_address(s, r), payload + r * s->row_bytes, (size_t)s->row_bytes);
}

/*
 * checkpoint(s) for one session (Sec. 3 "The contract"): write its record
 * into out[0 .. pcso_record_bytes).  Each section fp is PCSFP64-v1 of its
 * payload; the session fp is fmix(tree(section fps) ^ n_sections).
 * Returns the record size, or 0 if cap is too small or n < 1.
 */
uint64_t pcso_pack(const pcso_section *s, int32_t n, uint32_t session_id, uint32_t kind,
                   uint8_t *out, uint64_t cap)
{
    uint64_t total = pcso_record_bytes(s, n), off;
    uint64_t *fps;
    uint8_t *e;
    int32_t i;
    if (n < 1 || cap < total) return 0;
    fps = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    if (!fps) return 0;
    memset(out, 0, (size_t)total);
    off = pcso_payload_start(n);
    for (i = 0; i < n; i++) {
        gather_section(&s[i], out + off);
        fps[i] = pcso_fingerprint(out + off, s[i].bytes);
        e = out + PCSO_HEADER_BYTES + (uint64_t)PCSO_ENTRY_BYTES * (uint64_t)i;
        put_u32(e + 0, s[i].type);
        put_u32(e + 4, s[i].dtype);
        put_u32(e + 8, s[i].layer);
        put_u32(e + 12, s[i].layout);
        put_u64(e + 16, off);
        put_u64(e + 24, s[i].bytes);
        put_u64(e + 32, fps[i]);
        put_u64(e + 40, s[i].dim0);
        put_u64(e + 48, s[i].dim1);
        put_u64(e + 56, s[i].layout == PCSO_RING ? s[i].ring_start : 0);
        off = round_up(off + s[i].bytes, PCSO_ALIGN);
    }
    put_u32(out + 0, PCSO_MAGIC);
    put_u16(out + 4, (uint16_t)PCSO_VERSION);
    put_u16(out + 6, (uint16_t)n);
    put_u32(out + 8, session_id);
    put_u32(out + 12, kind);
    put_u64(out + 16, total);
    put_u64(out + 24, pcso_fmix(pcso_tree(fps, (uint64_t)n) ^ (uint64_t)n));
    free(fps);
    return total;
}

/* Header fields of a record (returns 0 if the magic/version do not match). */
int32_t pcso_record_header(const uint8_t *rec, uint32_t *n_sections, uint32_t *session_id,
                           uint32_t *kind, uint64_t *total, uint64_t *session_fp)
{
    if (get_u32(rec) != PCSO_MAGIC || (get_u32(rec + 4) & 0xFFFFu) != PCSO_VERSION) return 0;
    *n_sections = get_u32(rec + 4) >> 16;
    *session_id = get_u32(rec + 8);
    *kind = get_u32(rec + 12);
    *total = get_u64(rec + 16);
    *session_fp = get_u64(rec + 24);
    return 1;
}

/* Section entry i of a record: offset, bytes, fp and the ring start (aux). */
void pcso_record_section(const uint8_t *rec, int32_t i, uint64_t *offset, uint64_t *bytes,
                         uint64_t *fp, uint64_t *aux)
{
    const uint8_t *e = rec + PCSO_HEADER_BYTES + (uint64_t)PCSO_ENTRY_BYTES * (uint64_t)i;
    *offset = get_u64(e + 16);
    *bytes = get_u64(e + 24);
    *fp = get_u64(e + 32);
    *aux = get_u64(e + 56);
}

/*
 * restore(c) (Sec. 3 "The contract"): write each section payload of the
 * record back to the target sections.  A RING target whose ring_start is
 * 0xFFFFFFFF takes the ring start stored in the record.  With verify != 0
 * the payload fps and the session fp are recomputed first.
 * Returns 0 on success, -1 on a shape mismatch, -6 if verification fails.
 */
int32_t pcso_restore(const uint8_t *rec, pcso_section *t, int32_t n, int32_t verify)
{
    uint32_t ns, sid, kind;
    uint64_t total, sfp, offset, bytes, fp, aux;
    uint64_t *fps;
    int32_t i, bad = 0;
    if (n < 1 || !pcso_record_header(rec, &ns, &sid, &kind, &total, &sfp) || (int32_t)ns != n)
        return -1; /* a record holds at least one section */
    fps = (uint64_t *)malloc((size_t)n * sizeof(uint64_t));
    if (!fps) return -1;
    for (i = 0; i < n; i++) {
        pcso_record_section(rec, i, &offset, &bytes, &fp, &aux);
        if (bytes != t[i].bytes) {
            free(fps);
            return -1;
        }
        fps[i] = fp;
        if (verify && pcso_fingerprint(rec + offset, bytes) != fp) bad = 1;
    }
    if (verify && pcso_fmix(pcso_tree(fps, (uint64_t)n) ^ (uint64_t)n) != sfp) bad = 1;
    free(fps);
    if (bad) return -6;
    for (i = 0; i < n; i++) {
        pcso_section s = t[i];
        pcso_record_section(rec, i, &offset, &bytes, &fp, &aux);
        if (s.layout == PCSO_RING && s.ring_start == 0xFFFFFFFFu) s.ring_start = (uint32_t)aux;
        scatter_section(&s, rec + offset);
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Reactive host-budget plan: shrink, then drop (Sec. 7.10 "Predictive      */
/* eviction": the runtime escalates shrink -> nothing left to shrink ->     */
/* drop, and acts only when the budget binds; Sec. 7.5 "At 16 MB no policy  */
/* evicts at all").  Reading: sessions are visited in ascending priority    */
/* (ties: lower index first); each shrink takes a bank to the retention     */
/* fraction (round-half-even of frac * n); shrinking stops as soon as the   */
/* kept bytes fit; if every bank is shrunk and they still do not fit,       */
/* sessions are dropped (k = 0) in the same order until they do.            */
/* ------------------------------------------------------------------------ */

typedef struct {
    double priority;
    int32_t index;
} pcso_order;

static int cmp_order(const void *a, const void *b)
{
    const pcso_order *x = (const pcso_order *)a, *y = (const pcso_order *)b;
    if (x->priority < y->priority) return -1;
    if (x->priority > y->priority) return 1;
    return (x->index > y->index) - (x->index < y->index);
}

int32_t pcso_budget_plan(const int32_t *n, const uint64_t *entry_bytes, const double *priority,
                         int32_t count, uint64_t budget, double frac, int32_t *k,
                         int32_t *shrinks, int32_t *drops)
{
    pcso_order *ord;
    unsigned __int128 kept = 0;
    int32_t s, i;
    *shrinks = 0;
    *drops = 0;
    for (s = 0; s < count; s++) {
        k[s] = n[s];
        kept += (unsigned __int128)(uint64_t)n[s] * entry_bytes[s];
    }
    if (kept <= budget) return 0;
    ord = (pcso_order *)malloc((size_t)(count > 0 ? count : 1) * sizeof(pcso_order));
    if (!ord) return -1;
    for (s = 0; s < count; s++) {
        ord[s].priority = priority ? priority[s] : (double)s;
        ord[s].index = s;
    }
    qsort(ord, (size_t)count, sizeof(pcso_order), cmp_order);
    for (i = 0; i < count && kept > budget; i++) {
        int32_t target;
        double v;
        s = ord[i].index;
        v = nearbyint(frac * (double)n[s]);
        if (v < 0) v = 0;
        if (v > n[s]) v = n[s];
        target = (int32_t)v;
        if (target < k[s]) {
            kept -= (unsigned __int128)(uint64_t)(k[s] - target) * entry_bytes[s];
            k[s] = target;
            (*shrinks)++;
        }
    }
    for (i = 0; i < count && kept > budget; i++) {
        s = ord[i].index;
        if (k[s] > 0) {
            kept -= (unsigned __int128)(uint64_t)k[s] * entry_bytes[s];
            k[s] = 0;
            (*drops)++;
        }
    }
    free(ord);
    return 0;
}
