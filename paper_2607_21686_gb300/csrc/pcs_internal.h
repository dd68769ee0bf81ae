// pcs_internal.h -- descriptors shared by the host runtime (pcs_runtime.cpp)
// and the sm_103a kernels (pcs_kernels.cu).  Plain structs copied to the
// device once per call; no torch types.
#pragma once

#include <atomic>
#include <cstdint>

#include <cuda_runtime.h>

namespace pcs {

constexpr uint32_t kChunkBytes = 4096;   // fingerprint chunk
constexpr uint32_t kRecordAlign = 256;   // record / payload alignment
constexpr uint32_t kHeaderBytes = 64;
constexpr uint32_t kEntryBytes = 64;
constexpr uint32_t kMagic = 0x31534350u;  // "PCS1"
constexpr uint32_t kVersion = 1;
constexpr int kMaxGroupLog2 = 5;         // at most 32 chunks per warp task

// Errors a kernel records (OR-ed into the context's device error word).
constexpr uint32_t kDevErrIndex = 1u;    // a row / page id out of range
constexpr uint32_t kDevErrTimeout = 2u;  // a bounded wait inside a kernel gave up
constexpr uint32_t kDevErrNoPage = 4u;   // a page pool had no free page
constexpr uint32_t kDevErrRefcount = 8u; // a page released, shared or written while held by nobody

enum Layout : uint32_t { kContig = 0, kRows = 1, kRing = 2 };

// Work modes of the streaming kernel.
enum Mode : int {
  kModeHash = 0,       // read a contiguous buffer, fingerprint it
  kModePack = 1,       // gather layout side -> payload, fingerprint
  kModeRestore = 2,    // payload -> scatter layout side (no hashing)
  kModeRestoreV = 3,   // payload -> scatter layout side, fingerprint payload
};

// One fingerprinted stream of bytes (a buffer, or a section payload).
// "Layout side" = where the bytes live in the session (source of a pack,
// target of a restore, the buffer itself when hashing); the other side is
// the contiguous payload inside a record.
struct alignas(16) SecDesc {
  uint8_t* lbase;          // layout-side base
  uint8_t* payload;        // contiguous side (record payload), or null
  const int32_t* index;    // ROWS row ids / RING page table
  uint64_t bytes;          // logical bytes L
  uint64_t row_bytes;      // ROWS / RING
  uint64_t base_rows;      // bound on index values
  uint32_t layout;
  int32_t rb_shift;        // log2(row_bytes) if a power of two, else -1
  uint32_t ring_start;
  uint32_t window;
  uint32_t page_rows;
  int32_t pr_shift;        // log2(page_rows) if a power of two, else -1
  uint32_t task_begin;     // first warp task (= node slot) of this stream
  uint32_t n_tasks;
  uint64_t n_chunks;
  uint32_t align;          // CONTIG layout side: 16, 4 or 1 (largest that divides lbase)
  uint32_t fin_count;      // nodes the finaliser trees: [fin_begin, fin_begin + fin_count)
  uint32_t fin_begin;      // (the task nodes, or their 32-to-1 reduction)
  uint32_t sess;           // checkpoint / restore: the session of this stream
  uint32_t pad[2];
};
static_assert(sizeof(SecDesc) == 112, "SecDesc layout");

// One session: a record and the contiguous range of its sections.
struct alignas(16) SessDesc {
  uint8_t* record;         // record base (pack: written; restore: read)
  uint64_t total_bytes;
  uint64_t payload_start;  // header + table, rounded up to 256
  uint32_t sec_begin;
  uint32_t n_sections;
  uint32_t session_id;
  uint32_t kind;
};
static_assert(sizeof(SessDesc) == 40 || sizeof(SessDesc) == 48, "SessDesc layout");

// Section entry exactly as stored in a record (64 bytes, little-endian).
struct alignas(16) Entry {
  uint32_t type, dtype, layer, layout;
  uint64_t offset, bytes, fp, dim0, dim1, aux;
};
static_assert(sizeof(Entry) == 64, "Entry layout");

// One memory bank to score / prune.
struct alignas(16) BankDesc {
  const uint16_t* keys;    // [n][D] fp16 / bf16 bits
  const uint16_t* query;   // [D]
  uint64_t entry_begin;    // CSR offset of this bank's scores
  uint64_t kept_begin;     // CSR offset of this bank's kept indices
  int32_t n;
  int32_t D;
  int32_t k;
  uint32_t is_bf16;
  uint64_t entry_bytes;    // bytes one kept entry costs (global threshold)
  uint64_t pad;
};
static_assert(sizeof(BankDesc) == 64, "BankDesc layout");

// The streams one streaming kernel processes: item j is stream secs[ids[j]],
// owning this kernel's tasks [begin[j], begin[j+1]) (the last up to n_tasks).
// Task t of item j writes node secs[ids[j]].task_begin + (t - begin[j]).
struct WorkList {
  const uint32_t* ids;
  const uint32_t* begin;
  int n_items;
  uint32_t n_tasks;
};

// Chunks per task of the TMA-staged kernel (an 8 KiB tile).
constexpr int kBulkTileChunks = 2;
constexpr uint32_t kFinRegNodes = 1024;  // nodes a finalising warp trees from registers
// Smallest row size the TMA-staged kernel takes for ROWS / RING streams.
constexpr uint64_t kBulkMinRowBytes = 512;

// Kernel launchers (pcs_kernels.cu).  All enqueue on `stream`, return the
// CUDA error of the launch.

// Register kernel: warp tasks of 2^group_log2 chunks, 128-bit loads/stores.
cudaError_t launch_stream(int mode, const SecDesc* secs, WorkList wl, int group_log2,
                          uint64_t* nodes, uint32_t* dev_err, int sm_count, int blocks_per_sm,
                          cudaStream_t stream);

// TMA-staged kernel: tasks of kBulkTileChunks chunks staged through shared
// memory with cp.async.bulk; one persistent block per SM.  `sched`: two
// device words of the call (zero on entry, left zero) that share out the
// launch's last tiles at run time; launches using the same words must be
// ordered.  (Hash mode runs k_hash and does not use them.)
cudaError_t launch_bulk(int mode, const SecDesc* secs, WorkList wl, uint64_t* nodes,
                        uint32_t* dev_err, uint32_t* sched, int sm_count, cudaStream_t stream);

// One launch for a small call: the register streaming pass over wl (no
// node reduction), then the finaliser of `mode` run by the last block to
// finish (hash: n_items buffers; pack / restore_verify: n_items sessions).
// `ticket` must be zero; the last block resets it.
cudaError_t launch_small(int mode, const SecDesc* secs, WorkList wl, int group_log2,
                         uint64_t* nodes, uint32_t* dev_err, uint32_t* ticket, int n_items,
                         const SessDesc* sess, const Entry* entries, uint64_t* fp_out,
                         const uint64_t* fp_before, uint8_t* flags, uint32_t* bad, int sm_count,
                         int blocks_per_sm, cudaStream_t stream);

// One level of the node reduction of stream i: count nodes at src, reduced
// by aligned groups of 32 to ceil(count / 32) nodes at dst.
struct NodeLevel {
  uint32_t src, count, dst, pad;
};

// Streams with many task nodes: reduce each aligned group of 32 nodes of
// stream i (nodes[lv[i].src ...]) to one node at nodes[lv[i].dst + g].
// Groups of all streams are numbered by dst - base (monotone).
cudaError_t launch_reduce_nodes(const NodeLevel* lv, int n_secs, uint64_t* nodes, uint32_t base,
                                uint32_t n_groups, int sm_count, cudaStream_t stream);

// Section fps from the nodes [fin_begin, fin_begin + fin_count) (in place), then per mode:
//   kModeHash: fp_out[i] = fp; if fp_before: flags[i] = fp != fp_before[i]
//   kModePack: header + section table of each session's record
//   kModeRestoreV: compare with the record's stored fps; corrupt[s] = 1 and
//                  ++*bad on mismatch
cudaError_t launch_finalize(int mode, const SecDesc* secs, const SessDesc* sess, int n_sess,
                            const Entry* entries, uint64_t* nodes, uint64_t* fp_out,
                            const uint64_t* fp_before, uint8_t* flags, uint32_t* bad,
                            int max_secs, cudaStream_t stream);



cudaError_t launch_topk(const BankDesc* banks, int n_banks, const float* scores,
                        int32_t* kept_idx, cudaStream_t stream);
// One thread waits for what never happens (which = 0: an mbarrier's second
// arrival; 1: *never_set >= 1), gives up after the kernels' wait bound and
// sets the timeout bit in *err.
cudaError_t launch_selftest_wait(int which, const uint32_t* never_set, uint32_t* err,
                                 cudaStream_t stream);


// ---- One relevance threshold across all banks (pcs_prune_global) ---------
constexpr int kGTile = 4096;    // entries per tile of the global passes
constexpr int kGPasses = 6;     // digits of the 64-bit key: 11, 11, 10, 11, 11, 10 bits
constexpr int kGBins = 2048;    // bins of the widest digit

// Select state: the kept set is every entry whose ranking key exceeds
// `threshold`.  Set by the host, advanced by the last block of each pass.
struct alignas(16) GState {
  uint64_t prefix, mask;  // key bits fixed so far
  uint64_t remaining;     // budget left for keys inside the prefix
  uint64_t threshold;
  uint32_t done, ticket, total_kept, n_cand;
  uint32_t bar_count, bar_gen, pad[2];  // k_gfinish: arrivals, last barrier released
  uint64_t whist[kGBins]; // entry bytes per digit (mixed entry sizes)
  uint32_t chist[kGBins]; // entries per digit
};

// Summed bins of one later digit pass inside k_gfinish.
struct GBinSet {
  uint64_t w[kGBins];
  uint32_t c[kGBins];
};

// The score kernel's optional epilogue: the first digit pass of the global
// threshold (a histogram of the top key bits, then the digit choice).
struct GHist {
  GState* st;             // NULL: no histogram
  uint64_t uniform_bytes; // entry bytes when every bank costs the same
  int32_t mode;           // 1: uniform entry bytes, 2: per-bank entry bytes
  int32_t pad;
};

// Passed by value as a kernel parameter.
struct GPlan {
  const float* scores;        // [entries], bank-major
  const uint64_t* ebeg;       // [n_banks + 1]: first entry of each bank; ebeg[n_banks] = entries
  const uint64_t* ebytes;     // [n_banks]: bytes one entry of the bank costs
  const uint32_t* tile_bank;  // [tiles + 1]: bank of entry min(t * kGTile, entries - 1)
  uint32_t* tile_cnt;         // [tiles]: kept per tile
  GState* st;
  int32_t* kept_idx;          // [<= entries], CSR by bank
  int32_t* kept_off;          // [n_banks + 1]
  uint64_t entries;
  uint64_t uniform_bytes;     // entry bytes when every bank costs the same
  int32_t n_banks;
  int32_t tiles;
  int32_t uniform;
  int32_t local;              // 1: histogram only, the host sums the parts and picks
  uint64_t pos_base;          // position of entry 0 in the whole (split) population
  int32_t vec;                // 1: scores 16-byte aligned (whole runs read as float4)
  int32_t pad;
  // k_gfinish scratch
  uint32_t* ucand;            // [tiles * 8]: candidates of each 512-entry unit
  uint64_t* ckey;             // [tiles * kGTile]: their keys, unit u's from 512 u
  uint32_t* cbank;            // the same slots: their banks (mixed entry sizes only)
  GBinSet* hb;                // [kGPasses]: summed bins of the passes after the first
  uint32_t* err;              // the context's error word (a barrier that timed out)
};

// Scores of every entry; with gh.st set (and a fixed-width kernel), also the
// first digit pass of the global threshold.  Returns through *fused whether
// that pass was done.
cudaError_t launch_score(const BankDesc* banks, int n_banks, uint64_t n_entries, int max_dim,
                         int key_types, float* scores, int sm_count, cudaStream_t stream,
                         GHist gh = GHist{}, bool* fused = nullptr);

// The bins of pass `pass` (0..kGPasses-1) of the byte-weighted radix select
// over a part of a split population (local plan: the host sums and picks);
// a no-op once the threshold is known.
cudaError_t launch_gselect(const GPlan& p, int pass, int sm_count, cudaStream_t stream);
// The digit passes from `first_pass` on (none once the state is done) and
// the compaction: kept indices and bank offsets.  One cooperative launch.
cudaError_t launch_gfinish(const GPlan& p, int first_pass, int sm_count, cudaStream_t stream);

// ---- Copy-on-write page pool (pcs_pool_*) ---------------------------------
// Reference counts and a free stack over caller memory.  A kernel either only
// takes pages off the stack (alloc, copy leg) or only puts pages back
// (release), never both, so the stack needs no lock.
struct PoolDev {
  uint8_t* base;       // n_pages * page_bytes, caller memory
  uint32_t* rc;        // [n_pages] table slots holding each page
  int32_t* free_ids;   // [n_pages] stack of free pages; [0, *top) valid
  int32_t* top;
  uint32_t* err;       // the context's error word
  uint64_t page_bytes; // multiple of 16
  int32_t n_pages;
  int32_t pad;
};

cudaError_t launch_pool_alloc(const PoolDev& p, int32_t* ids, int32_t n, cudaStream_t stream);
cudaError_t launch_pool_share(const PoolDev& p, const int32_t* src, int32_t* dst, int32_t n,
                              cudaStream_t stream);
// The copy leg before a write of table[entries[j]] (j < n; entries NULL: j).
cudaError_t launch_pool_cow(const PoolDev& p, int32_t* table, int64_t n_table,
                            const int32_t* entries, int32_t n, int sm_count, cudaStream_t stream);
cudaError_t launch_pool_release(const PoolDev& p, const int32_t* ids, int32_t n,
                                cudaStream_t stream);

// ---- Byte-mismatch distance (pcs_mismatch) --------------------------------
constexpr uint32_t kMmUnit = 2048;  // bytes of each pair per warp iteration

struct MmPair {
  const uint8_t* a;
  const uint8_t* b;
  uint64_t bytes;       // bytes compared: min of the two lengths
  uint32_t vec;         // both 16-byte aligned: 16-byte loads
  uint32_t pad;
};

// Pair i owns units [unit_begin[i], unit_begin[i+1]); counts[i] += mismatches.
cudaError_t launch_mismatch(const MmPair* pairs, const uint64_t* unit_begin, int32_t n,
                            uint64_t units, uint64_t* counts, int sm_count, cudaStream_t stream);

// ---- Reads against buffers (pcs_classify_reads) ---------------------------
// Buffers sorted by start; maxend[i] = max(end[0..i]).
struct ReadPlan {
  const uint64_t* start;
  const uint64_t* end;
  const uint64_t* maxend;
  const uint32_t* orig;   // caller index of each sorted buffer
  int32_t n;
  int32_t pad;
};
cudaError_t launch_classify_reads(const ReadPlan& p, const uint64_t* addr, const uint64_t* bytes,
                                  int64_t m, uint8_t* flags, int sm_count, cudaStream_t stream);

// Occupancy of the streaming kernel (blocks per SM) for the launch shape.
int stream_blocks_per_sm();

// ---- Fingerprints with no allocation (pcs_fingerprint_static) -------------
constexpr int kStaticMaxBufs = 64;         // buffers per call
constexpr uint32_t kStaticMaxNodes = 65536;  // tree nodes per call (512 KiB)

struct StaticBuf {
  const uint8_t* ptr;
  uint64_t bytes;
  uint64_t n_chunks;
  uint32_t task_begin;  // first node slot of this buffer
  uint32_t n_tasks;
  uint32_t align;       // 16, 4 or 1
  uint32_t pad;
};

// Passed by value as a kernel parameter (no device copy of the plan).
struct StaticPlan {
  StaticBuf b[kStaticMaxBufs];
  int32_t n;
  uint32_t n_tasks;
  int32_t glog2;
  int32_t pad;
};

// Device address of the fixed node scratch on the current device; the first
// call on a device looks it up (cudaGetSymbolAddress) with that device current.
cudaError_t static_scratch(uint64_t** nodes);
cudaError_t launch_fingerprint_static(const StaticPlan& plan, uint64_t* nodes, uint64_t* fp_out,
                                      cudaStream_t stream);

}  // namespace pcs
