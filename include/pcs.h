/*
 * pcs.h -- C ABI of libpcs, the GB300 (sm_103a) data-parallel hot path of
 * Persistent Computational State (PCS).
 *
 * PCS is the minimal non-recomputable state a generative session must keep
 * across requests (Sec. 3, Definition 1).  The paper's runtime exposes four
 * operations over sessions and opaque snapshot handles -- checkpoint,
 * restore, fork, delete (Sec. 3 "The contract") -- with four invariants:
 *   I1 round-trip      restore(checkpoint(s)) reproduces s (here: byte-exact)
 *   I2 durability      a snapshot is immutable; it survives later work and,
 *                      through a file, the death of the process that made it
 *   I3 fork independence   a fork is an independent copy
 *   I4 completeness    a snapshot holds exactly the selected sections
 * This library implements those operations for many sessions per call, plus
 * the content fingerprint that decides must-snapshot vs derivable (Sec. 4,
 * procedure FINGERPRINT, step 1 at epsilon = 0) and the relevance-keyed
 * pruning of memory banks (Sec. 5 "The two semantic decisions"; Sec. 7.5).
 *
 * Conventions for every call
 *   - Return value: PCS_OK (0) or a negative pcs_status.  pcs_last_error()
 *     gives a message for the calling thread's last failure.
 *   - Argument errors are detected on the host before anything is enqueued.
 *     Errors found by a kernel (an index out of range) are recorded on the
 *     device and returned by the next pcs_sync() as PCS_E_RANGE; the kernel
 *     skips the offending access instead of performing it.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  All device work is enqueued on it; calls return before it
 *     finishes unless documented otherwise.
 *   - Pointers marked "device" must be device (or mapped pinned host) memory
 *     reachable from the GPU of the context; the caller owns every buffer it
 *     passes.  Buffers are read or written only by work enqueued on `stream`.
 *   - Alignment: row bases and row sizes (ROWS / RING layouts) and bank
 *     keys / queries must be multiples of 16 bytes (else PCS_E_ALIGN).
 *     Contiguous buffers and sections may have any address and byte count;
 *     16-byte aligned ones take the 128-bit vector path.
 *   - Snapshots are owned by the library (device or pinned host arenas) and
 *     are immutable after checkpoint; a handle is valid until pcs_delete.
 *   - A context may be used from several host threads; calls are serialised
 *     internally.  Work from different streams that uses the same snapshot
 *     is ordered by the library (events), so a restore on stream B after a
 *     checkpoint on stream A reads the finished record.
 */
#ifndef PCS_H
#define PCS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t pcs_status;

#define PCS_OK 0
#define PCS_E_INVAL (-1)    /* bad argument (null, size, count, layout)      */
#define PCS_E_ALIGN (-2)    /* pointer or row size not a multiple of 16 B   */
#define PCS_E_NOMEM (-3)    /* device or pinned host allocation failed      */
#define PCS_E_CUDA (-4)     /* a CUDA runtime call failed                   */
#define PCS_E_BUDGET (-5)   /* a byte budget cannot be met                  */
#define PCS_E_CORRUPT (-6)  /* verified restore / file: fingerprint mismatch */
#define PCS_E_HANDLE (-7)   /* unknown or deleted snapshot handle           */
#define PCS_E_IO (-8)       /* file could not be opened, read or written    */
#define PCS_E_TIMEOUT (-9)  /* a bounded device wait gave up                */
#define PCS_E_RANGE (-10)   /* a device-side index was out of range         */

/* Element type tags recorded in section entries (informational). */
#define PCS_DT_RAW 0
#define PCS_DT_U8 1
#define PCS_DT_I32 2
#define PCS_DT_I64 3
#define PCS_DT_F16 4
#define PCS_DT_BF16 5
#define PCS_DT_F32 6
#define PCS_DT_U64 7

/* Section type tags (caller-chosen; these are the conventional ones). */
#define PCS_SEC_OBS 1       /* uint8 observation (Markovian model)          */
#define PCS_SEC_RNG 2       /* generator state: seed u64, offset u64        */
#define PCS_SEC_KEPT_IDX 3  /* int32 indices of the kept bank entries       */
#define PCS_SEC_KEYS 4      /* bank keys of the kept entries                */
#define PCS_SEC_VALUES 5    /* bank values (latents) of the kept entries    */
#define PCS_SEC_META 6      /* position indices of a KV context             */
#define PCS_SEC_K 7         /* one layer's keys of a KV window              */
#define PCS_SEC_V 8         /* one layer's values of a KV window            */

/* Session kinds (recorded in the record header; informational). */
#define PCS_KIND_MARKOV 1   /* {OBS, RNG}                                   */
#define PCS_KIND_BANK 2     /* {KEPT_IDX, KEYS, VALUES}                     */
#define PCS_KIND_KV 3       /* {META, K_0, V_0, K_1, V_1, ...}              */

/* How a section's logical bytes map onto memory. */
#define PCS_LAYOUT_CONTIG 0 /* bytes [0, bytes) at base                     */
#define PCS_LAYOUT_ROWS 1   /* row r at base + index[r] * row_bytes         */
#define PCS_LAYOUT_RING 2   /* paged ring: row r in ring slot               */
                            /* q = (ring_start + r) mod window, on page     */
                            /* index[q / page_rows], row q mod page_rows:   */
                            /* base + (page * page_rows + q % page_rows)    */
                            /*        * row_bytes                           */

/* Where a snapshot lives. */
#define PCS_PLACE_DEVICE 0       /* HBM of the context's GPU                */
#define PCS_PLACE_PINNED_HOST 1  /* page-locked host memory, GPU-mapped     */

/* Ring start meaning "the one stored in the snapshot" (restore targets). */
#define PCS_RING_START_FROM_SNAPSHOT 0xFFFFFFFFu

/* k-rules of pcs_prune. */
#define PCS_K_FIXED 0     /* k = min(n, k_max)                               */
#define PCS_K_BUDGET 1    /* T = sum n_s*entry_bytes_s; k_s = n_s if T <= B, */
                          /* else floor(n_s * B / T)  (Sec. 7.5); T may be  */
                          /* given for a population split across processes  */
#define PCS_K_FRACTION 2  /* k = round-half-even(fraction * n)              */
                          /* (Table tab:keepfrac)                           */

typedef struct pcs_ctx pcs_ctx;
typedef struct pcs_snapshot pcs_snapshot;
typedef struct pcs_pool pcs_pool;
typedef struct pcs_plan pcs_plan;

/* A runtime buffer to fingerprint: `bytes` bytes at device pointer `ptr`. */
typedef struct pcs_buf {
    const void *ptr;   /* device, any alignment (may be NULL if bytes==0)   */
    uint64_t bytes;
    uint32_t dtype;    /* PCS_DT_* (informational)                          */
    uint32_t flags;    /* reserved, 0                                       */
} pcs_buf;

/*
 * One section of a session.  For pcs_checkpoint `base` is read; for
 * pcs_restore it is written.  Logical bytes of the section:
 *   CONTIG: `bytes` bytes at base.
 *   ROWS:   bytes / row_bytes rows; row r at base + index[r] * row_bytes;
 *           every index[r] must lie in [0, base_rows).
 *   RING:   window rows (bytes == window * row_bytes); see PCS_LAYOUT_RING;
 *           every page id must lie in [0, base_rows); window must be a
 *           multiple of page_rows; ring_start < window (restore targets may
 *           pass PCS_RING_START_FROM_SNAPSHOT).
 * ROWS / RING: row_bytes and base must be multiples of 16; `index` is
 * device int32.  CONTIG: any address.
 */
typedef struct pcs_section {
    uint32_t type;        /* PCS_SEC_*                                      */
    uint32_t dtype;       /* PCS_DT_*                                       */
    uint32_t layer;       /* layer number (KV) or 0                         */
    uint32_t layout;      /* PCS_LAYOUT_*                                   */
    void *base;           /* device                                         */
    uint64_t bytes;       /* logical payload bytes                          */
    uint64_t row_bytes;   /* ROWS / RING                                    */
    const int32_t *index; /* device: ROWS row ids / RING page table         */
    uint64_t base_rows;   /* ROWS: rows at base; RING: pages at base        */
    uint32_t ring_start;  /* RING                                           */
    uint32_t window;      /* RING: ring slots (rows)                        */
    uint32_t page_rows;   /* RING: rows per page                            */
    uint32_t reserved;    /* 0                                              */
    uint64_t dim0, dim1;  /* shape recorded in the snapshot (informational) */
} pcs_section;

/* A session: an ordered list of 1..65535 sections. */
typedef struct pcs_session {
    uint32_t session_id;
    uint32_t kind;                 /* PCS_KIND_*                             */
    int32_t n_sections;
    int32_t reserved;              /* 0                                      */
    const pcs_section *sections;   /* host array of n_sections               */
} pcs_session;

/* A memory bank to prune: n_entries keys of key_dim fp16/bf16 elements. */
typedef struct pcs_bank {
    const void *keys;      /* device [n_entries][key_dim], 16-byte aligned  */
    const void *query;     /* device [key_dim]: the return viewpoint        */
    int32_t n_entries;
    int32_t key_dim;       /* multiple of 8                                 */
    uint32_t key_dtype;    /* PCS_DT_F16 or PCS_DT_BF16                     */
    uint32_t reserved;     /* 0                                             */
    uint64_t entry_bytes;  /* bytes one kept entry costs (PCS_K_BUDGET,     */
                           /* pcs_prune_global)                             */
} pcs_bank;

typedef struct pcs_prune_params {
    int32_t rule;          /* PCS_K_*                                       */
    int32_t k_max;         /* PCS_K_FIXED                                   */
    uint64_t budget_bytes; /* PCS_K_BUDGET: host byte budget B              */
    double fraction;       /* PCS_K_FRACTION, in [0, 1]                     */
    uint64_t total_bytes;  /* PCS_K_BUDGET: T of the whole population when */
                           /* its banks are split over calls or processes   */
                           /* (the sum of every part's T); 0 = the T of the */
                           /* banks of this call                            */
    uint32_t kept_align;   /* pcs_prune: 0 or 1 = kept lists back to back;  */
                           /* 4 = each bank's list starts at a multiple of  */
                           /* 4 entries (16 bytes of a 16-byte aligned      */
                           /* kept_idx), so a checkpoint moves the lists    */
                           /* with bulk copies                              */
    uint32_t reserved;     /* 0                                             */
} pcs_prune_params;

typedef struct pcs_snapshot_info {
    uint32_t session_id;
    uint32_t kind;
    int32_t n_sections;
    uint32_t placement;    /* PCS_PLACE_*                                   */
    uint64_t total_bytes;  /* record bytes (multiple of 256)                */
    uint64_t session_fp;   /* fmix(tree(section fps) ^ n_sections)          */
    const void *data;      /* record address (read-only for the caller)     */
} pcs_snapshot_info;

typedef struct pcs_section_info {
    uint32_t type, dtype, layer, layout;
    uint64_t offset;       /* payload offset within the record              */
    uint64_t bytes;
    uint64_t fp;           /* PCSFP64-v1 of the payload                     */
    uint64_t dim0, dim1;
    uint64_t aux;          /* RING: ring start at checkpoint; else 0        */
} pcs_section_info;

/* Counters of a context. */
typedef struct pcs_stats {
    uint64_t kernel_launches;  /* kernels this context has launched         */
    uint64_t device_reserved;  /* bytes of HBM held by the snapshot arena   */
    uint64_t host_reserved;    /* bytes of pinned host memory held          */
    int32_t live_snapshots;    /* handles not yet deleted                   */
    int32_t sm_count;          /* SMs of the context's GPU                  */
} pcs_stats;

/* Accumulated device time of one kernel (see pcs_timing_enable). */
typedef struct pcs_kernel_time {
    char name[32];             /* kernel name, NUL-terminated               */
    uint64_t launches;         /* launches timed                            */
    double total_ms;           /* sum of CUDA-event durations               */
} pcs_kernel_time;

/* Message of the calling thread's last error ("" if none).  No paper
 * counterpart: error reporting of this C interface. */
const char *pcs_last_error(void);
/* Name of a status code (no paper counterpart). */
const char *pcs_status_string(pcs_status s);

/*
 * Cap the memory the context reserves for snapshots of one placement
 * (no paper counterpart: a runtime control; bytes; 0 = no cap, the default).  Reservations already made stay; empty
 * ones over the cap are returned.  A call that would need more fails with
 * PCS_E_NOMEM before any launch and leaves no snapshot behind.
 */
pcs_status pcs_set_arena_limit(pcs_ctx *ctx, uint32_t placement, uint64_t bytes);

/*
 * Create a context on CUDA device `device`: it owns the snapshot arenas,
 * the workspace of the kernels and the snapshot table.  A context is this
 * library's form of the session runtime's session table and PCS store
 * (Sec. 5, Figure fig:arch; Sec. 8), with the paged allocation that Sec. 3
 * "Boundary" leaves to the lower runtime.  PCS_E_CUDA if the device cannot
 * be used.  Two environment variables, read here, change how the context
 * works but never what it computes: PCS_CHECK=1 checks every call's plan on
 * the host before launching it (node slots, work lists, layouts, payloads
 * inside their records; a violation returns PCS_E_INVAL and launches
 * nothing), and PCS_DISABLE_TMA=1 sends every stream through the register
 * kernel instead of the TMA-staged one.
 */
pcs_status pcs_create(int32_t device, pcs_ctx **out);
/* Destroy a context (the end of the store of Sec. 5 / Sec. 8): waits for
 * its work, frees every snapshot it owns. */
pcs_status pcs_destroy(pcs_ctx *ctx);
/* Fill `out` with the context's counters (host only, no synchronisation).
 * No paper counterpart: monitoring of this library. */
pcs_status pcs_get_stats(pcs_ctx *ctx, pcs_stats *out);

/*
 * Per-kernel timing (no paper counterpart: a measurement aid): with on != 0
 * every kernel launch of the context is bracketed by CUDA events on its own
 * stream; on == 0 stops.  Either call clears the accumulated times.
 */
pcs_status pcs_timing_enable(pcs_ctx *ctx, int32_t on);
/*
 * Wait for the timed launches and write up to `max` per-kernel totals to
 * `out` (host); *n = number of kernels with at least one timed launch.  No
 * paper counterpart.
 */
pcs_status pcs_timing_read(pcs_ctx *ctx, pcs_kernel_time *out, int32_t max, int32_t *n);

/*
 * Wait for `stream`, then report what kernels recorded since the last
 * pcs_sync -- failed asynchronous verifications (PCS_E_CORRUPT), a bounded
 * wait that gave up (PCS_E_TIMEOUT), an out-of-range index (PCS_E_RANGE) --
 * or a CUDA error (PCS_E_CUDA).  Clears them.  No paper counterpart: the
 * paper's runtime is synchronous Python; this is where the asynchronous
 * outcome of a verified restore (the I1 check of Sec. 3) reaches the host.
 */
pcs_status pcs_sync(pcs_ctx *ctx, void *stream);

/*
 * Self-test of the bounded device waits (no paper counterpart: a check of
 * the failure path).  Enqueues on `stream` one kernel thread that waits,
 * with the same helpers and the same bound (about two seconds of SM clock)
 * as the library's kernels, for something that never happens: which = 0,
 * the second arrival at a shared-memory mbarrier that expects two (the wait
 * of the TMA pipeline); which = 1, a device flag that nothing writes (the
 * poll of the grid barrier).  The wait gives up, sets the timeout bit and
 * the kernel returns, so the next pcs_sync on the stream reports
 * PCS_E_TIMEOUT and the context stays usable.  PCS_E_INVAL for another
 * `which`.
 */
pcs_status pcs_selftest_wait(pcs_ctx *ctx, int32_t which, void *stream);

/*
 * Content fingerprint PCSFP64-v1 of n buffers (the measurement that decides
 * must-snapshot, Sec. 4 step 1 at epsilon = 0).  fp_out: device uint64[n].
 * Definition: 4096-byte chunks (bytes past the end read as 0); in chunk c,
 * lane l in [0,32) hashes 16-byte segments l+32k (k = 0..7) with
 * h = fmix(SEED ^ (32c + l)), h = (rotl(h,23) ^ w) * P per little-endian
 * word, a_l = fmix(h); a lane tree comb(a,b) = fmix(a*P + rotl(b,31)) gives
 * the chunk hash; a pairwise tree over chunks (odd item carried up) gives
 * the root; fp = fmix(root ^ bytes * P).  fmix = SplitMix64 finaliser,
 * P = 0x9E3779B97F4A7C15, SEED = 0x5043534650363401.
 */
pcs_status pcs_fingerprint(pcs_ctx *ctx, const pcs_buf *bufs, int32_t n, uint64_t *fp_out,
                           void *stream);

/*
 * Classify n buffers after a recompute (Sec. 3 "The partition"): fingerprint
 * them again and write must_snapshot[i] = (fp_before[i] != fp_after[i]):
 * 1 = non-derivable, must be snapshotted; 0 = derivable.
 * fp_before: device uint64[n]; fp_after: device uint64[n] or NULL;
 * must_snapshot: device uint8[n].
 */
pcs_status pcs_classify(pcs_ctx *ctx, const pcs_buf *bufs, int32_t n, const uint64_t *fp_before,
                        uint64_t *fp_after, uint8_t *must_snapshot, void *stream);

/*
 * Host only: how many entries each bank keeps under `params` (the k-rules:
 * a fixed cap, the same fraction of every bank under a host budget, Sec. 7.5,
 * or a retention fraction, Table tab:keepfrac).  k_out: host int32[n].
 * PCS_E_INVAL on a bad rule or fraction.
 */
pcs_status pcs_prune_counts(const pcs_bank *banks, int32_t n, const pcs_prune_params *params,
                            int32_t *k_out);

/*
 * Relevance-keyed pruning (Sec. 5; Sec. 7.5): score every entry of every
 * bank by cos(query, key) in fp32 (fixed order: lane floor(e/8) mod 32 owns
 * element e, separately rounded multiply and add, lane tree, RN sqrt and
 * division, 0 if a norm is 0), keep per bank the k_s entries with the
 * largest (score, -index) -- ties to the lower index, NaN lowest, -0 == +0 --
 * and write their indices in ascending order.
 *   scores:   device float[sum n] (CSR by bank) or NULL
 *   kept_idx: device int32[sum k] (CSR by bank, k from pcs_prune_counts);
 *             with kept_align = 4, int32[sum round_up(k, 4)]: bank b's list
 *             starts at the sum of round_up(k, 4) over the banks before it
 *             (the entries between lists are left as they were)
 *   kept_off: device int32[n + 1] or NULL: offsets of the lists in kept_idx
 *             (the last one: the entries kept_idx spans)
 * PCS_E_INVAL for a kept_align other than 0, 1 or 4.
 */
pcs_status pcs_prune(pcs_ctx *ctx, const pcs_bank *banks, int32_t n,
                     const pcs_prune_params *params, float *scores, int32_t *kept_idx,
                     int32_t *kept_off, void *stream);

/*
 * Keep-k by caller-supplied rank keys, for the recency-keyed policies the
 * paper compares against relevance (Sec. 7.5, Table tab:evict: lru ranks a
 * frame by its last use, fifo by its insertion order): per bank, keep the k_b
 * entries with the largest (key, -index) -- ties to the lower index, NaN
 * lowest -- and write their indices ascending.
 *   keys:     device float[sum n] (CSR by bank, bank b = n[b] entries)
 *   n, k:     host int32[n_banks]; k_b > n_b keeps the whole bank
 *   kept_idx: device int32[sum min(k, n)]; kept_off: device int32[n+1] or NULL
 */
pcs_status pcs_topk(pcs_ctx *ctx, const float *keys, const int32_t *n, const int32_t *k,
                    int32_t n_banks, int32_t *kept_idx, int32_t *kept_off, void *stream);

/*
 * One relevance threshold across all banks under a host byte budget: the
 * budgeted pruning of Sec. 7.5 with a cross-session threshold instead of the
 * same fraction per bank, so a session with more relevant frames keeps more
 * of them.  Every entry is scored as by pcs_prune; all entries of all banks
 * are ranked together by (score desc, bank asc, index asc) and the longest
 * prefix of that order whose entry_bytes sum to at most `budget` is kept (a
 * budget that does not bind keeps everything).
 *   scores:   device float[sum n] (CSR by bank) or NULL
 *   kept_idx: device int32[sum n] (capacity); kept entries of bank b, in
 *             ascending index, at kept_idx[kept_off[b] .. kept_off[b+1])
 *   kept_off: device int32[n + 1], required; kept_off[n] = entries kept
 * PCS_E_INVAL if the total entry bytes exceed 2^64 - 1; bank errors as for
 * pcs_prune.
 */
pcs_status pcs_prune_global(pcs_ctx *ctx, const pcs_bank *banks, int32_t n, uint64_t budget,
                            float *scores, int32_t *kept_idx, int32_t *kept_off, void *stream);

/*
 * The histogram exchange of a global threshold over banks split across
 * processes: called once per digit pass (the same number of times in every
 * part) with this part's histograms -- counts[i] entries and bytes[i] entry
 * bytes per digit i < bins -- which it must replace, in place, by their sums
 * over all parts (an all-reduce).  Returns 0, or non-zero to stop.
 */
typedef int32_t (*pcs_hist_exchange_fn)(void *user, uint64_t *counts, uint64_t *bytes,
                                        int32_t bins);

/*
 * pcs_prune_global for one part of a population whose banks are split
 * across processes (Sec. 7.5's budget over the whole population; the one
 * exchange is a histogram per digit pass, done by the caller's `exchange`).
 * Entries are ranked over the whole population by (score desc, position
 * asc), this part's entry 0 being at position `pos_base` (the entries of the
 * parts before it); the kept set is the longest prefix of that order within
 * `budget`, and this call writes this part's share of it (kept_idx /
 * kept_off as for pcs_prune_global).  Synchronises `stream` once per pass.
 * PCS_E_INVAL if the exchange fails or positions pass 2^32 - 1.
 */
pcs_status pcs_prune_global_part(pcs_ctx *ctx, const pcs_bank *banks, int32_t n, uint64_t budget,
                                 uint64_t pos_base, pcs_hist_exchange_fn exchange, void *user,
                                 float *scores, int32_t *kept_idx, int32_t *kept_off,
                                 void *stream);

/*
 * Host only: the reactive shrink-then-drop plan of a host budget (Sec. 7.10:
 * the runtime escalates shrink -> nothing left to shrink -> drop, and acts
 * only when the budget binds).  Sessions are visited in ascending priority
 * (ties: lower index first; priority NULL = session index).  While the kept
 * bytes sum(k_s * entry_bytes_s) exceed `budget`, the next bank is shrunk to
 * round-half-even(fraction * n_s); once every bank is shrunk, sessions are
 * dropped (k_s = 0) in the same order.  k_out: host int32[count]; shrinks /
 * drops: host int32 counts (may be NULL).
 */
pcs_status pcs_budget_plan(const int32_t *n, const uint64_t *entry_bytes, const double *priority,
                           int32_t count, uint64_t budget, double fraction, int32_t *k_out,
                           int32_t *shrinks, int32_t *drops);

/*
 * Copy-on-write page pool (Sec. 3, I3: fork independence, which the
 * mechanism realises by copy-on-write; Sec. 3 "Boundary": the runtime owns
 * allocation and copy-on-write; Sec. 7.3: reference-counted blocks whose copy
 * leg fires on the first write).  The pool manages n_pages pages of
 * page_bytes in caller device memory at `base` (the caller keeps owning the
 * bytes; sessions address the pages through int32 page tables, e.g. RING
 * sections).  Each page carries the number of table slots that hold it; free
 * pages sit on a device stack.  Page id -1 marks an empty slot and is skipped
 * by every call.  Work is enqueued on `stream`; calls on one pool must be
 * ordered (one stream, or events).  Device-side failures are sticky on the
 * context and returned by pcs_sync: no free page -> PCS_E_NOMEM (the slot
 * keeps its shared page, or an alloc slot gets -1); an id outside the pool
 * -> PCS_E_RANGE (skipped); a page shared, written or released while held
 * by nobody -> PCS_E_INVAL (skipped).  Pools die with their context.
 *   base: device, 16-byte aligned; page_bytes: multiple of 16.
 */
pcs_status pcs_pool_create(pcs_ctx *ctx, void *base, uint64_t page_bytes, int32_t n_pages,
                           pcs_pool **out);
/* Destroy a pool (of the copy-on-write pool above; the pages' bytes stay the
 * caller's). */
pcs_status pcs_pool_destroy(pcs_ctx *ctx, pcs_pool *pool);

/* n free pages, each held once: ids: device int32[n].  Paged allocation of
 * the lower runtime (Sec. 3 "Boundary"). */
pcs_status pcs_pool_alloc(pcs_ctx *ctx, pcs_pool *pool, int32_t *ids, int32_t n, void *stream);

/*
 * Fork of the tables holding src (fork(c) by copy-on-write, Sec. 3 I3;
 * Sec. 7.3): every page of src gains one holder and, if dst is not NULL,
 * src is copied to dst (the child's table).  No page bytes move.  src, dst:
 * device int32[n].
 */
pcs_status pcs_pool_share(pcs_ctx *ctx, pcs_pool *pool, const int32_t *src, int32_t *dst,
                          int32_t n, void *stream);

/*
 * The copy leg of copy-on-write (Sec. 7.3: it fires on the first write),
 * before the caller writes the pages at table[entries[j]]
 * (j < n; entries NULL: table[0 .. n)): a slot whose page is also held
 * elsewhere gets a fresh page holding a copy of it and gives up its hold on
 * the old one; a page held by that slot alone stays.  Of several holders of
 * one page in one call, all but one copy.  Entries must be distinct.
 *   table: device int32[n_table] (updated in place); entries: device int32[n].
 */
pcs_status pcs_pool_prepare_write(pcs_ctx *ctx, pcs_pool *pool, int32_t *table, int64_t n_table,
                                  const int32_t *entries, int32_t n, void *stream);

/* Every page of ids loses one holder; pages held by nobody become free
 * (delete(c) of a shared table, Sec. 3 "The contract"). */
pcs_status pcs_pool_release(pcs_ctx *ctx, pcs_pool *pool, const int32_t *ids, int32_t n,
                            void *stream);

/*
 * No paper counterpart (inspection of the pool above).
 * Synchronises `stream`, then reads the pool's state: free page count; the
 * holder count of every page (host uint32[n_pages] or NULL); the free pages
 * (host int32[n_pages] or NULL; the first *free_pages entries are valid).
 */
pcs_status pcs_pool_query(pcs_ctx *ctx, pcs_pool *pool, int32_t *free_pages, uint32_t *counts,
                          int32_t *free_ids, void *stream);

/*
 * Distance for the discovery procedure (Sec. 4: a return-consistency metric
 * D with tolerance eps; here D counts differing bytes, so eps = 0 is byte
 * identity): counts[i] = number of byte positions below min(a[i].bytes,
 * b[i].bytes) where the two buffers differ, plus the difference of their
 * lengths.  a, b: host arrays of n device buffers (any alignment; 16-byte
 * aligned pairs take the fast path); counts: device uint64[n].
 */
pcs_status pcs_mismatch(pcs_ctx *ctx, const pcs_buf *a, const pcs_buf *b, int32_t n,
                        uint64_t *counts, void *stream);

/*
 * State versus witness (Sec. 3, "A distinction the implementation forced":
 * a buffer is PCS iff restore reads it).  Given the byte ranges a restore
 * read -- read j covers [addr[j], addr[j] + bytes[j]) -- flags[i] = 1 iff
 * some read of at least one byte overlaps buffer i (a non-empty buffer).
 * Buffers may overlap one another.  bufs: host array of n buffers (only ptr
 * and bytes are used); addr, bytes: device uint64[m]; flags: device uint8[n].
 */
pcs_status pcs_classify_reads(pcs_ctx *ctx, const pcs_buf *bufs, int32_t n, const uint64_t *addr,
                              const uint64_t *bytes, int64_t m, uint8_t *flags, void *stream);

/*
 * Probe of the discovery procedure: run the leave-and-return trajectory with
 * exactly the components keep[i] != 0 restored from the snapshot (the others
 * left to be re-derived), and write the distance D to *distance.  Returns 0,
 * or non-zero to stop the procedure.
 */
typedef int32_t (*pcs_probe_fn)(void *user, const uint8_t *keep, uint64_t *distance);

/*
 * Host only: discovering PCS by measurement (Sec. 4, procedure
 * FINGERPRINT) over k components: (1) necessity -- component i is necessary
 * if D > eps with every component but i restored; (2) sufficiency -- if D <=
 * eps with exactly the necessary set restored, that set is PCS; (3)
 * redundancy fallback -- otherwise add, one at a time, the component whose
 * addition gives the smallest D (ties: lowest index) until D <= eps.
 *   pcs_out: host uint8[k] (1 = PCS, 0 = derivable); probes: probes run;
 *   consistent: 1 if the returned set reaches D <= eps (0 if even every
 *   component does not).  PCS_E_INVAL if the probe fails.
 */
pcs_status pcs_discover(int32_t k, pcs_probe_fn probe, void *user, uint64_t eps,
                        uint8_t *pcs_out, int32_t *probes, int32_t *consistent);

/*
 * Host only: bytes of the PCS1 record a session of these sections packs to:
 * 256-byte aligned header + 64-byte entries, then each payload at a
 * 256-byte aligned offset.  The record layout is this library's (Sec. 3
 * "Boundary": storage owns serialisation; the paper fixes no format).
 */
pcs_status pcs_record_bytes(const pcs_section *sections, int32_t n_sections, uint64_t *out);

/*
 * checkpoint(s) for n sessions (Sec. 3 "The contract"): gather every
 * section into one contiguous PCS1 record per session in a new snapshot of
 * the given placement, with the fingerprint of every section payload fused
 * into the copy, and write the record header (session fp) and section
 * table.  out: host array receiving n handles.  Asynchronous; the live
 * buffers may be changed once `stream` has passed this call (I2).
 */
pcs_status pcs_checkpoint(pcs_ctx *ctx, const pcs_session *sessions, int32_t n,
                          uint32_t placement, pcs_snapshot **out, void *stream);

/*
 * fork(c) (Sec. 3 "The contract"): an independent byte copy of a snapshot,
 * same placement, so the child's continuation cannot affect the parent's
 * (I3).  A full copy because a bank consumed in place cannot share pages
 * (Sec. 7.3); pcs_pool_share is the copy-on-write form.
 */
pcs_status pcs_fork(pcs_ctx *ctx, const pcs_snapshot *parent, pcs_snapshot **child,
                    void *stream);
/* fork(c) (Sec. 3 "The contract") for n snapshots in one call; children:
 * host array of n handles. */
pcs_status pcs_fork_many(pcs_ctx *ctx, pcs_snapshot *const *parents, int32_t n,
                         pcs_snapshot **children, void *stream);

/*
 * restore(c) (Sec. 3 "The contract") for n snapshots, byte-identical to the
 * checkpointed state (I1): scatter each section payload to the
 * target section of targets[i] (same section count and byte counts; any
 * layout).  verify = 1 also recomputes every section fingerprint and the
 * session fp, waits for `stream`, and returns PCS_E_CORRUPT if any differs
 * from the record (the bytes have been written by then).  verify = 2 does
 * the same checks without waiting: failures are counted on the device and
 * the next pcs_sync returns PCS_E_CORRUPT.  verify = 0: no check.
 */
pcs_status pcs_restore(pcs_ctx *ctx, pcs_snapshot *const *snaps, int32_t n,
                       const pcs_session *targets, int32_t verify, void *stream);

/*
 * Prepared calls (no paper counterpart: a runtime form of checkpoint(s) and
 * restore(c) of Sec. 3 "The contract", same records, same verification),
 * for the same checkpoint or restore repeated (a periodic checkpoint of a
 * fixed set of sessions, a restore that recurs): the call is
 * planned once -- validation, descriptors, launch shape, uploaded into a
 * device buffer of the plan -- and each pcs_plan_run only launches kernels.
 * Everything a section describes (pointers, sizes, layouts, ring starts) is
 * fixed at plan time; the bytes it points at are read at run time.  Runs of
 * one plan must be ordered (they share its scratch).
 *
 * pcs_plan_checkpoint: plans checkpoint(s) of n sessions, creates their n
 * snapshots (out, host array) and runs the first checkpoint on `stream`.
 * Every later run overwrites the same records in place (the snapshots are
 * the plan's latest checkpoint); the records stay valid until both the
 * snapshots are deleted and the plan destroyed.
 * pcs_plan_restore: plans restore(c) of n snapshots into n targets; verify
 * 0 or 2 (mismatches reported by pcs_sync).  The plan keeps the snapshots'
 * records alive until it is destroyed.
 */
pcs_status pcs_plan_checkpoint(pcs_ctx *ctx, const pcs_session *sessions, int32_t n,
                               uint32_t placement, pcs_snapshot **out, pcs_plan **plan,
                               void *stream);
pcs_status pcs_plan_restore(pcs_ctx *ctx, pcs_snapshot *const *snaps, int32_t n,
                            const pcs_session *targets, int32_t verify, pcs_plan **plan);
pcs_status pcs_plan_run(pcs_ctx *ctx, pcs_plan *plan, void *stream);
pcs_status pcs_plan_destroy(pcs_ctx *ctx, pcs_plan *plan);

/* delete(c) (Sec. 3 "The contract"): release a snapshot (its memory is
 * reused once pending work that reads it has finished).  The handle is
 * invalid afterwards: a call given it returns PCS_E_HANDLE until a later
 * checkpoint, fork or read issues the same handle value again (handle
 * objects are reused), after which it names that new snapshot. */
pcs_status pcs_delete(pcs_ctx *ctx, pcs_snapshot *snap);

/* delete(c) (Sec. 3 "The contract") for n snapshots at once; PCS_E_HANDLE
 * (and nothing deleted) if any handle is unknown. */
pcs_status pcs_delete_many(pcs_ctx *ctx, pcs_snapshot *const *snaps, int32_t n);

/* Header fields of a snapshot; waits for the work that wrote it.  No paper
 * counterpart: inspection of this library's record (Sec. 3 "Boundary":
 * storage owns serialisation). */
pcs_status pcs_snapshot_get_info(pcs_ctx *ctx, const pcs_snapshot *snap, pcs_snapshot_info *out);
/* Section entry i of a snapshot; waits for the work that wrote it.  No
 * paper counterpart (inspection, as above). */
pcs_status pcs_snapshot_get_section(pcs_ctx *ctx, const pcs_snapshot *snap, int32_t i,
                                pcs_section_info *out);
/* Copy record bytes [offset, offset + bytes) to dst (device or host),
 * enqueued on stream.  No paper counterpart: raw access to the serialised
 * record that storage owns (Sec. 3 "Boundary"). */
pcs_status pcs_snapshot_copy_out(pcs_ctx *ctx, const pcs_snapshot *snap, uint64_t offset,
                                 uint64_t bytes, void *dst, void *stream);

/* Durability across processes (I2): write the record to `path` (written to
 * a temporary file, flushed, then renamed); read one back into a new
 * snapshot after validating its header and section table (PCS_E_CORRUPT on
 * a malformed record, PCS_E_IO on a file error). */
pcs_status pcs_snapshot_write_file(pcs_ctx *ctx, const pcs_snapshot *snap, const char *path);
pcs_status pcs_snapshot_read_file(pcs_ctx *ctx, const char *path, uint32_t placement,
                                  pcs_snapshot **out);

/*
 * Fingerprints without any allocation.  The paper has no counterpart: this is
 * a service of this library for callers that cannot allocate device memory,
 * for example a serving process that has already carved nearly all of HBM
 * into its own page pools (a cudaMalloc would fail or upset its accounting),
 * or a latency-critical loop that cannot afford the device-wide
 * synchronisation that cudaMalloc / cudaFree bring.
 *
 * Same result as pcs_fingerprint (PCSFP64-v1 of each buffer), but no context
 * is needed and nothing is allocated: the plan travels as a kernel
 * parameter, and the only working memory is one fixed array of
 * PCS_STATIC_MAX_NODES tree nodes (512 KiB) that the library's GPU code
 * defines.  Every GPU that runs this call holds that array until the process
 * exits.
 *   bufs    host array of n buffer descriptions (device pointers, any
 *           alignment); n <= PCS_STATIC_MAX_BUFFERS
 *   fp_out  device uint64[n]
 * Limits: each buffer needs ceil(bytes / 131072) nodes (at least 1) and one
 * call may use at most PCS_STATIC_MAX_NODES of them: about 8 GiB per call.
 * A call beyond a limit returns PCS_E_INVAL before anything is enqueued.
 * The first call on a device looks up the array's device address with that
 * device current (this may load the library's GPU code on that device); make
 * that first call before any stream capture.  The address is kept for the
 * rest of the process: after cudaDeviceReset on a device, the module is
 * loaded anew and the kept address is stale, so a process that resets a
 * device must not call this entry point on it again.  All calls share the array: two
 * calls whose work overlaps on the GPU (unordered streams) corrupt each
 * other's results, so order them.  No part of the array needs to start at
 * zero; each call writes every node it later reads.  On success the call
 * allocates neither device nor host memory.
 */
#define PCS_STATIC_MAX_BUFFERS 64
#define PCS_STATIC_MAX_NODES 65536
pcs_status pcs_fingerprint_static(const pcs_buf *bufs, int32_t n, uint64_t *fp_out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PCS_H */
