// pcs_runtime.cpp -- host side of libpcs: argument validation, planning of
// records and kernel work, the snapshot table, the arena allocator, files.
//
// The paper's runtime (Sec. 5, Sec. 8) is a single-process Python service
// that keeps, per session, the PCS a later restore needs; the byte movement
// is delegated to the layer below.  This file is that layer's host half: it
// turns a batch of sessions into one launch of the streaming kernel over
// every section of every session, and owns the snapshots behind opaque
// handles (Sec. 3 "The contract": checkpoint / restore / fork / delete).
#include <nvtx3/nvToolsExt.h>
#include <cuda_runtime.h>
#include <fcntl.h>
#include <unistd.h>

#include <algorithm>
#include <cerrno>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <unordered_map>
#include <map>
#include <memory>
#include <mutex>
#include <string>
#include <unordered_set>
#include <vector>

#include "pcs.h"
#include "pcs_internal.h"
#include "pcs_ptrset.h"

using namespace pcs;

// ---------------------------------------------------------------------------
// Errors
// ---------------------------------------------------------------------------

namespace {

thread_local std::string g_err;

// An NVTX range around each data-path call of the library, named after the
// call, for Nsight tools (for example `ncu --nvtx --nvtx-include
// "pcs_checkpoint/"` profiles only the kernels a checkpoint launched).
// Without a tool attached a range costs a few nanoseconds.
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};
#define PCS_TRACE(name) TraceRange pcs_trace_range_(name)

pcs_status fail(pcs_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return s;
}

pcs_status cuda_fail(cudaError_t e, const char* what) {
  return fail(PCS_E_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define PCS_CUDA(call)                                  \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
  } while (0)

uint64_t round_up(uint64_t x, uint64_t a) { return (x + a - 1) / a * a; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
int log2_exact(uint64_t x) {
  if (x == 0 || (x & (x - 1)) != 0) return -1;
  int s = 0;
  while ((1ull << s) != x) ++s;
  return s;
}

// ---------------------------------------------------------------------------
// Events: pooled, shared; a range of freed memory keeps the events of the
// work that last used it, and whoever reuses it first waits for them on its
// own stream (stream-ordered reuse; the host never blocks for it).
// ---------------------------------------------------------------------------

struct EventPool {
  std::vector<cudaEvent_t> free_;
  ~EventPool() {
    for (auto e : free_) cudaEventDestroy(e);
  }
  cudaEvent_t get() {
    if (!free_.empty()) {
      cudaEvent_t e = free_.back();
      free_.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return nullptr;
    return e;
  }
  void put(cudaEvent_t e) { free_.push_back(e); }
};

struct Event {
  cudaEvent_t ev = nullptr;
  std::shared_ptr<EventPool> pool;
  ~Event() {
    if (ev) pool->put(ev);
  }
  bool done() const { return ev && cudaEventQuery(ev) == cudaSuccess; }
};
using Ev = std::shared_ptr<Event>;

Ev record_event(const std::shared_ptr<EventPool>& pool, cudaStream_t s) {
  auto e = std::make_shared<Event>();
  e->pool = pool;
  e->ev = pool->get();
  if (!e->ev || cudaEventRecord(e->ev, s) != cudaSuccess) return nullptr;
  return e;
}

void prune_done(std::vector<Ev>& deps) {
  deps.erase(std::remove_if(deps.begin(), deps.end(), [](const Ev& e) { return !e || e->done(); }),
             deps.end());
}

// ---------------------------------------------------------------------------
// Arena allocator: slabs of device (HBM) or pinned, GPU-mapped host memory,
// first fit with coalescing, 256-byte granules.
// ---------------------------------------------------------------------------

struct Range {
  uint64_t size = 0;
  std::vector<Ev> deps;  // work that must finish before the bytes are reused
};

struct Slab {
  uint8_t* base = nullptr;  // device-usable address
  uint64_t size = 0;
  uint64_t used = 0;
  std::map<uint64_t, Range> free;  // offset -> free range
};

struct Block {
  Slab* slab = nullptr;
  uint64_t off = 0;
  uint64_t size = 0;
  uint8_t* ptr = nullptr;
  uint32_t placement = PCS_PLACE_DEVICE;
  int refs = 0;
  Ev written;                                 // completion of the write
  std::map<cudaStream_t, Ev> uses;            // latest use per stream
};

class Arena {
 public:
  Arena(uint32_t placement, std::shared_ptr<EventPool> pool) : placement_(placement), pool_(pool) {}
  ~Arena() { release_all(); }

  // Reserve `bytes`; `stream` is made to wait for earlier users of the range.
  pcs_status alloc(uint64_t bytes, cudaStream_t stream, Block** out) {
    bytes = round_up(std::max<uint64_t>(bytes, kRecordAlign), kRecordAlign);
    for (int attempt = 0; attempt < 3; ++attempt) {
      for (auto& sp : slabs_) {
        Slab* s = sp.get();
        for (auto it = s->free.begin(); it != s->free.end(); ++it) {
          if (it->second.size < bytes) continue;
          const uint64_t off = it->first;
          Range r = std::move(it->second);
          s->free.erase(it);
          prune_done(r.deps);
          for (auto& e : r.deps)
            if (cudaStreamWaitEvent(stream, e->ev, 0) != cudaSuccess)
              return fail(PCS_E_CUDA, "cudaStreamWaitEvent failed");
          if (r.size > bytes) {
            Range rest;
            rest.size = r.size - bytes;
            rest.deps = r.deps;
            s->free.emplace(off + bytes, std::move(rest));
          }
          auto* b = new Block();
          b->slab = s;
          b->off = off;
          b->size = bytes;
          b->ptr = s->base + off;
          b->placement = placement_;
          s->used += bytes;
          *out = b;
          return PCS_OK;
        }
      }
      if (attempt == 0) {
        if (new_slab(bytes) == PCS_OK) continue;
        // Out of memory: return empty slabs, then try once more.
        trim();
        cudaGetLastError();
      } else if (attempt == 1) {
        if (new_slab(bytes) == PCS_OK) continue;
        cudaGetLastError();
      }
    }
    return fail(PCS_E_NOMEM, "cannot allocate %llu bytes of %s memory",
                static_cast<unsigned long long>(bytes),
                placement_ == PCS_PLACE_DEVICE ? "device" : "pinned host");
  }

  // Return a block; its bytes are reused only after its recorded uses.
  void free(Block* b) {
    Slab* s = b->slab;
    Range r;
    r.size = b->size;
    for (auto& kv : b->uses) r.deps.push_back(kv.second);
    if (b->written) r.deps.push_back(b->written);
    prune_done(r.deps);
    uint64_t off = b->off;
    s->used -= b->size;
    delete b;
    // Coalesce with the following and preceding free ranges.
    auto next = s->free.lower_bound(off);
    if (next != s->free.end() && next->first == off + r.size) {
      r.size += next->second.size;
      r.deps.insert(r.deps.end(), next->second.deps.begin(), next->second.deps.end());
      s->free.erase(next);
    }
    auto it = s->free.lower_bound(off);
    if (it != s->free.begin()) {
      auto prev = std::prev(it);
      if (prev->first + prev->second.size == off) {
        prev->second.size += r.size;
        prev->second.deps.insert(prev->second.deps.end(), r.deps.begin(), r.deps.end());
        prune_done(prev->second.deps);
        return;
      }
    }
    prune_done(r.deps);
    s->free.emplace(off, std::move(r));
  }

  void trim() {
    for (auto it = slabs_.begin(); it != slabs_.end();) {
      Slab* s = it->get();
      if (s->used == 0) {
        for (auto& kv : s->free)
          for (auto& e : kv.second.deps) cudaEventSynchronize(e->ev);
        free_memory(s->base);
        it = slabs_.erase(it);
      } else {
        ++it;
      }
    }
  }

  void release_all() {
    for (auto& s : slabs_) free_memory(s->base);
    slabs_.clear();
  }

  uint64_t reserved() const {
    uint64_t t = 0;
    for (auto& s : slabs_) t += s->size;
    return t;
  }

  // Cap on the bytes this arena reserves (0: none).
  void set_limit(uint64_t bytes) {
    limit_ = bytes;
    if (limit_ && reserved() > limit_) trim();
  }

 private:
  pcs_status new_slab(uint64_t bytes) {
    const uint64_t min_slab = placement_ == PCS_PLACE_DEVICE ? (256ull << 20) : (64ull << 20);
    uint64_t size = round_up(std::max(bytes, min_slab), 2ull << 20);
    if (limit_) {
      const uint64_t have = reserved();
      if (have + size > limit_) size = round_up(bytes, 2ull << 20);  // no headroom slab
      if (have + size > limit_) return PCS_E_NOMEM;
    }
    void* p = nullptr;
    if (placement_ == PCS_PLACE_DEVICE) {
      if (cudaMalloc(&p, size) != cudaSuccess) return PCS_E_NOMEM;
    } else {
      void* h = nullptr;
      if (cudaHostAlloc(&h, size, cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess)
        return PCS_E_NOMEM;
      if (cudaHostGetDevicePointer(&p, h, 0) != cudaSuccess) {
        cudaFreeHost(h);
        return PCS_E_NOMEM;
      }
      host_of_[p] = h;
    }
    auto s = std::make_unique<Slab>();
    s->base = static_cast<uint8_t*>(p);
    s->size = size;
    Range r;
    r.size = size;
    s->free.emplace(0, std::move(r));
    slabs_.push_back(std::move(s));
    return PCS_OK;
  }

  void free_memory(uint8_t* p) {
    if (placement_ == PCS_PLACE_DEVICE) {
      cudaFree(p);
    } else {
      auto it = host_of_.find(p);
      if (it != host_of_.end()) {
        cudaFreeHost(it->second);
        host_of_.erase(it);
      }
    }
  }

  uint32_t placement_;
  uint64_t limit_ = 0;
  std::shared_ptr<EventPool> pool_;
  std::vector<std::unique_ptr<Slab>> slabs_;
  std::map<void*, void*> host_of_;
};

}  // namespace

// ---------------------------------------------------------------------------
// Snapshots and the context
// ---------------------------------------------------------------------------

struct pcs_snapshot {
  Block* block = nullptr;
  uint64_t offset = 0;         // record offset within the block
  uint64_t total_bytes = 0;
  uint64_t payload_start = 0;
  uint32_t session_id = 0;
  uint32_t kind = 0;
  // Host copy of the section table (fp = 0): n_sections entries from
  // `first` of an array shared by the snapshots of one call and their forks.
  std::shared_ptr<const std::vector<Entry>> tables;
  uint32_t first = 0;
  uint32_t n_sections = 0;
  const Entry* table() const { return tables->data() + first; }
  uint8_t* record() const { return block->ptr + offset; }
};

struct pcs_pool {
  pcs::PoolDev d{};
  void* meta = nullptr;  // counts, free stack and top in one allocation
};

struct pcs_plan;

struct pcs_ctx {
  int device = 0;
  int sm_count = 0;
  int stream_bps = 1;          // resident blocks per SM of the streaming kernel
  bool use_bulk = true;        // TMA-staged kernel for eligible streams
  bool check_plans = false;    // PCS_CHECK=1: check every plan before launching
  std::mutex mu;
  std::shared_ptr<EventPool> events = std::make_shared<EventPool>();
  std::unique_ptr<Arena> dev_arena, host_arena;
  PtrSet<pcs_snapshot> live;
  std::vector<pcs_snapshot*> spare;  // deleted handles' objects, for the next ones
  // Workspaces, one per stream: the descriptors and tree nodes of a call,
  // after a header of per-call device words ([0] the fused kernel's ticket,
  // [1] failures of a verify = 1 restore, [4] and [5] the TMA kernel's work
  // sharing).  Calls on one stream are ordered
  // by the stream; calls on different streams do not share one, so they can
  // run side by side.
  struct Workspace {
    uint8_t* buf = nullptr;
    uint64_t bytes = 0;
    Ev busy;  // the last call's end
  };
  std::unordered_map<cudaStream_t, Workspace> ws;
  Workspace* ws_cur = nullptr;    // of the call in progress (calls hold mu)
  uint32_t* call_words = nullptr;  // its header words
  // Context-wide device words: [0] kernel error bits, [2] verify = 2
  // failures until the next pcs_sync, [4] a flag nothing writes (self-test).
  uint32_t* words = nullptr;
  std::vector<uint8_t> plan;   // host staging of the descriptors
  // Pinned slots for the plans of calls: a true async copy, no driver-side
  // staging of pageable memory (which can hold the host until the stream
  // has caught up).  Each slot grows to the largest plan it has carried.
  uint8_t* plan_slot_buf[8] = {};
  uint64_t plan_slot_cap[8] = {};
  Ev plan_slot_busy[8];
  int plan_slot = 0;
  int plan_slot_used = -1;     // slot of the call in progress, or -1
  uint8_t* stage = nullptr;    // pinned staging for file I/O
  uint64_t stage_bytes = 0;
  uint64_t launches = 0;       // kernels launched by this context
  // Per-kernel CUDA-event timing (pcs_timing_enable).
  bool timing = false;
  struct Timed {
    int kind;
    cudaEvent_t start, stop;
  };
  std::vector<Timed> timed;
  std::vector<cudaEvent_t> timing_events;  // free timing-capable events
  double kernel_ms[32] = {};
  uint64_t kernel_n[32] = {};
  std::unordered_set<pcs_pool*> pools;  // live page pools
  std::unordered_set<pcs_plan*> plans;  // live prepared calls
};

namespace {

constexpr uint64_t kStageBytes = 64ull << 20;

pcs_status set_device(pcs_ctx* c) {
  PCS_CUDA(cudaSetDevice(c->device));
  return PCS_OK;
}

// Kernels the context launches, for counting and timing.
enum KernelKind {
  kKStreamHash, kKStreamPack, kKStreamRestore, kKStreamRestoreV, kKFinalizeHash,
  kKFinalizePack, kKFinalizeRestoreV, kKScore, kKTopk, kKBulkHash, kKBulkPack,
  kKBulkRestore, kKBulkRestoreV, kKReduce, kKGSelect, kKGFinish, kKPoolAlloc, kKPoolShare,
  kKPoolCow, kKPoolRelease, kKMismatch, kKClassifyReads, kKernelKinds
};
static_assert(kKernelKinds <= 32, "kernel timing table");
const char* kKernelNames[kKernelKinds] = {
    "k_stream<hash>", "k_stream<pack>", "k_stream<restore>", "k_stream<restore_verify>",
    "k_finalize<hash>", "k_finalize<pack>", "k_finalize<restore_verify>", "k_score", "k_topk",
    "k_hash", "k_bulk<pack>", "k_bulk<restore>", "k_bulk<restore_verify>",
    "k_reduce_nodes", "k_gselect", "k_gfinish", "k_pool_alloc", "k_pool_share", "k_pool_cow",
    "k_pool_release", "k_mismatch", "k_classify_reads"};

cudaEvent_t timing_event(pcs_ctx* c) {
  if (!c->timing_events.empty()) {
    cudaEvent_t e = c->timing_events.back();
    c->timing_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Brackets one kernel launch: counts it and, when timing is on, records
// CUDA events around it on the launching stream.
struct LaunchScope {
  pcs_ctx* c;
  int kind;
  cudaStream_t stream;
  cudaEvent_t start = nullptr;
  LaunchScope(pcs_ctx* c_, int kind_, cudaStream_t s) : c(c_), kind(kind_), stream(s) {
    c->launches += 1;
    if (c->timing) {
      start = timing_event(c);
      if (start) cudaEventRecord(start, stream);
    }
  }
  ~LaunchScope() {
    if (!start) return;
    cudaEvent_t stop = timing_event(c);
    if (!stop) return;
    cudaEventRecord(stop, stream);
    c->timed.push_back({kind, start, stop});
  }
};

int stream_kind(int mode) {
  switch (mode) {
    case kModeHash: return kKStreamHash;
    case kModePack: return kKStreamPack;
    case kModeRestore: return kKStreamRestore;
    default: return kKStreamRestoreV;
  }
}

int bulk_kind(int mode) {
  switch (mode) {
    case kModeHash: return kKBulkHash;
    case kModePack: return kKBulkPack;
    case kModeRestore: return kKBulkRestore;
    default: return kKBulkRestoreV;
  }
}

Arena* arena_of(pcs_ctx* c, uint32_t placement) {
  return placement == PCS_PLACE_DEVICE ? c->dev_arena.get() : c->host_arena.get();
}

constexpr uint64_t kWsHeader = 256;  // per-call device words before the descriptors
constexpr int kWordBulkSched = 4;    // header words [4], [5]: the TMA kernel's work sharing

// The header words of a call: they sit just below its descriptors, in a
// stream's workspace and in a prepared call's buffer alike.
uint32_t* header_words(uint8_t* ws) { return reinterpret_cast<uint32_t*>(ws - kWsHeader); }

// The workspace of `stream` for the call in progress: grown if needed (after
// its last call has finished), else `stream` waits for its last call (a no-op
// on the same stream; a stream handle may be reused after its stream was
// destroyed).  Returns the base of the call's descriptors; the call's header
// words are c->call_words, zero on entry.
pcs_status ws_acquire(pcs_ctx* c, uint64_t bytes, cudaStream_t stream, uint8_t** out) {
  bytes = round_up(std::max<uint64_t>(bytes, 1), kRecordAlign) + kWsHeader;
  pcs_ctx::Workspace& W = c->ws[stream];
  if (bytes > W.bytes) {
    if (W.busy) PCS_CUDA(cudaEventSynchronize(W.busy->ev));
    W.busy.reset();
    if (W.buf) cudaFree(W.buf);
    W.buf = nullptr;
    W.bytes = 0;
    const uint64_t want = round_up(std::max<uint64_t>(bytes, 1ull << 20) * 5 / 4, 2ull << 20);
    if (cudaMalloc(&W.buf, want) != cudaSuccess) {
      cudaGetLastError();
      W.buf = nullptr;
      return fail(PCS_E_NOMEM, "cannot allocate %llu bytes of workspace",
                  static_cast<unsigned long long>(want));
    }
    PCS_CUDA(cudaMemset(W.buf, 0, kWsHeader));
    W.bytes = want;
  } else if (W.busy && !W.busy->done()) {
    PCS_CUDA(cudaStreamWaitEvent(stream, W.busy->ev, 0));
  }
  c->ws_cur = &W;
  c->call_words = reinterpret_cast<uint32_t*>(W.buf);
  *out = W.buf + kWsHeader;
  return PCS_OK;
}

constexpr uint64_t kPlanSlotBytes = 256 << 10;  // smallest pinned plan slot
constexpr uint64_t kPlanSlotMax = 64ull << 20;  // larger plans are copied from pageable memory
constexpr int kPlanSlots = 8;

// A free pinned plan slot for `bytes` of descriptors (round robin over
// kPlanSlots, grown to the largest plan it carries), which the call then
// holds until ws_release records its end -- a call that fails before then
// leaves the slot held for good, never reused early; null when the next slot
// is still busy or the plan is huge.
uint8_t* plan_slot(pcs_ctx* c, uint64_t bytes) {
  c->plan_slot_used = -1;
  if (bytes <= kPlanSlotMax) {
    const int i = c->plan_slot;
    Ev& busy = c->plan_slot_busy[i];
    if (!busy || busy->done()) {
      if (c->plan_slot_cap[i] < bytes) {
        if (c->plan_slot_buf[i]) cudaFreeHost(c->plan_slot_buf[i]);
        c->plan_slot_buf[i] = nullptr;
        c->plan_slot_cap[i] = 0;
        uint64_t cap = kPlanSlotBytes;
        while (cap < bytes) cap *= 2;
        void* p = nullptr;
        if (cudaHostAlloc(&p, cap, cudaHostAllocDefault) == cudaSuccess) {
          c->plan_slot_buf[i] = static_cast<uint8_t*>(p);
          c->plan_slot_cap[i] = cap;
        } else {
          cudaGetLastError();
        }
      }
      if (c->plan_slot_buf[i]) {
        c->plan_slot = (i + 1) % kPlanSlots;
        busy = std::make_shared<Event>();
        c->plan_slot_used = i;
        return c->plan_slot_buf[i];
      }
    }
  }
  return nullptr;
}

// Where a call writes `bytes` of descriptors: a pinned plan slot, else
// `fallback` (pageable memory).
uint8_t* plan_dst(pcs_ctx* c, uint64_t bytes, std::vector<uint8_t>& fallback) {
  if (uint8_t* slot = plan_slot(c, bytes)) return slot;
  fallback.resize(bytes);
  return fallback.data();
}

// Send descriptors written where plan_dst said into the workspace.
cudaError_t plan_send(pcs_ctx* c, uint8_t* ws, uint64_t bytes,
                        const std::vector<uint8_t>& fallback, cudaStream_t stream) {
  const uint8_t* src = c->plan_slot_used >= 0 ? c->plan_slot_buf[c->plan_slot_used] : fallback.data();
  return cudaMemcpyAsync(ws, src, bytes, cudaMemcpyHostToDevice, stream);
}

// Copy the call's descriptors (c->plan, `bytes`) into the workspace, through
// a pinned slot when one is free.
cudaError_t plan_copy(pcs_ctx* c, uint8_t* ws, uint64_t bytes, cudaStream_t stream) {
  if (uint8_t* slot = plan_slot(c, bytes)) std::memcpy(slot, c->plan.data(), bytes);
  return plan_send(c, ws, bytes, c->plan, stream);
}

// End of a call's use of the workspace (and of its plan slot): `done`, if
// given, is an event already recorded at this point of the stream.
pcs_status ws_release(pcs_ctx* c, cudaStream_t stream, Ev done = nullptr) {
  Ev& busy = c->ws_cur->busy;
  busy = done ? done : record_event(c->events, stream);
  if (!busy) return fail(PCS_E_CUDA, "cudaEventRecord failed");
  if (c->plan_slot_used >= 0) c->plan_slot_busy[c->plan_slot_used] = busy;
  c->plan_slot_used = -1;
  return PCS_OK;
}

// Record a use of a block on `stream` (kept until the block is freed).
pcs_status note_use(pcs_ctx* c, Block* b, cudaStream_t stream) {
  auto it = b->uses.find(stream);
  if (it != b->uses.end() && it->second.use_count() == 1) {
    PCS_CUDA(cudaEventRecord(it->second->ev, stream));
    return PCS_OK;
  }
  Ev e = record_event(c->events, stream);
  if (!e) return fail(PCS_E_CUDA, "cudaEventRecord failed");
  b->uses[stream] = e;
  return PCS_OK;
}

pcs_status wait_written(Block* b, cudaStream_t stream) {
  if (b->written && !b->written->done()) PCS_CUDA(cudaStreamWaitEvent(stream, b->written->ev, 0));
  return PCS_OK;
}

void release_block(pcs_ctx* c, Block* b) {
  if (--b->refs == 0) arena_of(c, b->placement)->free(b);
}

// Layout of one call's descriptors inside the workspace.
struct WsLayout {
  uint64_t secs = 0, sess = 0, entries = 0, banks = 0, nodes = 0, total = 0;
};

// Choose 2^g chunks per warp task: at least ~4 tasks per resident warp,
// at most 32 chunks per task.
int choose_group_log2(const pcs_ctx* c, uint64_t total_chunks) {
  const uint64_t warps = static_cast<uint64_t>(c->sm_count) * c->stream_bps * 8;
  int g = 0;
  while (g < kMaxGroupLog2 && (total_chunks >> (g + 1)) >= 4 * warps) ++g;
  return g;
}

uint64_t n_chunks_of(uint64_t bytes) { return bytes == 0 ? 1 : (bytes + kChunkBytes - 1) / kChunkBytes; }

// Validate a section used as a checkpoint source or a restore target.
pcs_status check_section(const pcs_section& s, int sess, int i, bool target) {
  if (s.layout > PCS_LAYOUT_RING)
    return fail(PCS_E_INVAL, "session %d section %d: unknown layout %u", sess, i, s.layout);
  if (s.layout == PCS_LAYOUT_CONTIG) {
    if (s.bytes > 0 && !s.base)
      return fail(PCS_E_INVAL, "session %d section %d: null base", sess, i);
    return PCS_OK;
  }
  if (s.row_bytes == 0 || s.row_bytes % 16 != 0)
    return fail(PCS_E_ALIGN, "session %d section %d: row_bytes %llu not a positive multiple of 16",
                sess, i, static_cast<unsigned long long>(s.row_bytes));
  if (s.bytes % s.row_bytes != 0)
    return fail(PCS_E_INVAL, "session %d section %d: bytes not a multiple of row_bytes", sess, i);
  if (s.bytes == 0) return PCS_OK;
  if (!s.base || !s.index)
    return fail(PCS_E_INVAL, "session %d section %d: null base or index", sess, i);
  if (!aligned16(s.base))
    return fail(PCS_E_ALIGN, "session %d section %d: base not 16-byte aligned", sess, i);
  if ((reinterpret_cast<uintptr_t>(s.index) & 3u) != 0)
    return fail(PCS_E_ALIGN, "session %d section %d: index not 4-byte aligned", sess, i);
  if (s.base_rows == 0)
    return fail(PCS_E_INVAL, "session %d section %d: base_rows must bound the index values", sess, i);
  if (s.layout == PCS_LAYOUT_ROWS) {
    if (s.bytes / s.row_bytes > 0x7FFFFFFFull)
      return fail(PCS_E_INVAL, "session %d section %d: too many rows", sess, i);
    return PCS_OK;
  }
  if (s.page_rows == 0 || s.window == 0 || s.window % s.page_rows != 0)
    return fail(PCS_E_INVAL, "session %d section %d: window must be a positive multiple of page_rows",
                sess, i);
  if (s.bytes != static_cast<uint64_t>(s.window) * s.row_bytes)
    return fail(PCS_E_INVAL, "session %d section %d: bytes != window * row_bytes", sess, i);
  if (s.ring_start >= s.window && !(target && s.ring_start == PCS_RING_START_FROM_SNAPSHOT))
    return fail(PCS_E_INVAL, "session %d section %d: ring_start %u >= window %u", sess, i,
                s.ring_start, s.window);
  return PCS_OK;
}

SecDesc make_desc(const pcs_section& s, uint8_t* payload, uint32_t ring_start) {
  SecDesc d{};
  d.lbase = static_cast<uint8_t*>(s.base);
  d.payload = payload;
  d.index = s.index;
  d.bytes = s.bytes;
  d.layout = s.layout;
  d.row_bytes = s.layout == PCS_LAYOUT_CONTIG ? 0 : s.row_bytes;
  d.rb_shift = s.layout == PCS_LAYOUT_CONTIG ? 0 : log2_exact(s.row_bytes);
  d.base_rows = s.base_rows;
  d.ring_start = ring_start;
  d.window = s.window;
  d.page_rows = s.page_rows;
  d.pr_shift = s.layout == PCS_LAYOUT_RING ? log2_exact(s.page_rows) : 0;
  d.n_chunks = n_chunks_of(s.bytes);
  const uintptr_t a = reinterpret_cast<uintptr_t>(s.base);
  d.align = (a & 15u) == 0 ? 16u : ((a & 3u) == 0 ? 4u : 1u);
  return d;
}

// Device allocations known to one call, as [lo, hi) address ranges, and the
// verdict for pointers outside them.
struct PtrCache {
  std::vector<std::pair<uintptr_t, uintptr_t>> dev;
  std::unordered_map<const void*, bool> other;
  size_t last = 0;  // the range that answered last (sections of a call share a few)
};

// cuMemGetAddressRange, looked up once through the runtime (no libcuda link).
using AddrRangeFn = int (*)(unsigned long long*, size_t*, unsigned long long);
AddrRangeFn addr_range_fn() {
  static AddrRangeFn fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      f = nullptr;
    }
    return reinterpret_cast<AddrRangeFn>(f);
  }();
  return fn;
}

// Is `p` device memory of the current device (not host, managed or unknown)?
// One query per device allocation: its whole address range is remembered.
bool is_device_ptr(const void* p, PtrCache& cache) {
  if (!p) return true;
  const uintptr_t u = reinterpret_cast<uintptr_t>(p);
  if (cache.last < cache.dev.size() && u >= cache.dev[cache.last].first &&
      u < cache.dev[cache.last].second)
    return true;
  for (size_t i = 0; i < cache.dev.size(); ++i) {
    if (u >= cache.dev[i].first && u < cache.dev[i].second) {
      cache.last = i;
      return true;
    }
  }
  auto it = cache.other.find(p);
  if (it != cache.other.end()) return it->second;
  cudaPointerAttributes a{};
  bool dev = false;
  if (cudaPointerGetAttributes(&a, p) == cudaSuccess) dev = a.type == cudaMemoryTypeDevice;
  else cudaGetLastError();
  unsigned long long base = 0;
  size_t size = 0;
  AddrRangeFn fn = addr_range_fn();
  if (dev && fn && fn(&base, &size, u) == 0 && size > 0) {
    cache.dev.emplace_back(static_cast<uintptr_t>(base), static_cast<uintptr_t>(base + size));
  } else {
    cache.other.emplace(p, dev);
  }
  return dev;
}

// How the streams of one call are split between the two kernels.
struct StreamPlan {
  std::vector<uint32_t> bulk_ids, bulk_begin, reg_ids, reg_begin;
  uint32_t bulk_tasks = 0, reg_tasks = 0;
  uint64_t nodes = 0;          // task nodes
  uint32_t reduce_groups = 0;  // 32-to-1 groups reduced before finalising (0 = none)
  uint64_t nodes_total = 0;    // task nodes + reduced nodes
  // Reduction levels: levels[k * n_streams + i] for stream i at level k,
  // with level_groups[k] groups numbered from level_base[k].
  std::vector<NodeLevel> levels;
  std::vector<uint32_t> level_groups, level_base;
  int glog2 = 0;
  bool link_bound = false;     // every stream crosses the host link (see link_bound_call)
};

// The TMA-staged kernel takes a stream whose bytes on both sides live in
// device memory and can be moved as whole 16-byte pieces: a 16-byte aligned
// contiguous buffer, or rows of at least 512 bytes.
bool bulk_eligible(const pcs_ctx* c, const SecDesc& d, bool payload_device, bool small_call,
                   PtrCache& cache) {
  if (!c->use_bulk || !payload_device || small_call) return false;
  if (!is_device_ptr(d.lbase, cache)) return false;
  if (d.layout == kContig) return d.align == 16 || d.bytes == 0;
  return d.row_bytes >= kBulkMinRowBytes && d.row_bytes % 16 == 0;
}

// A call whose every non-empty stream has one side in host memory (a record
// in pinned host memory, or a section that lives there) moves its bytes over
// the host link, a few hundred GB/s that half the SMs keep busy (measured:
// 256 KV sessions suspend at 193 GB/s and resume at 210 GB/s on half the SMs,
// as on all of them; on a quarter the resume lost 6 %, on an eighth 43 %): its
// register kernel gets a grid of 1 / kLinkSmDiv of the GPU, so a suspend and
// a resume on two streams, or a suspend beside other work, can run side by
// side instead of one after the other.
#ifndef PCS_LINK_SM_DIV
#define PCS_LINK_SM_DIV 2
#endif
constexpr int kLinkSmDiv = PCS_LINK_SM_DIV;

bool link_bound_call(const std::vector<SecDesc>& d, const std::vector<char>& bulk,
                     const std::vector<char>& payload_device, PtrCache& cache) {
  bool any = false;
  for (size_t i = 0; i < d.size(); ++i) {
    if (d[i].bytes == 0) continue;
    if (bulk[i]) return false;
    if (payload_device[i] && is_device_ptr(d[i].lbase, cache)) return false;
    any = true;
  }
  return any;
}

int grid_sms(const pcs_ctx* c, const StreamPlan& P) {
  return P.link_bound ? std::max(1, c->sm_count / kLinkSmDiv) : c->sm_count;
}

// Calls moving at most this many bytes take the register kernel: their time
// is launch latency, which the shared-memory pipeline does not shorten.
constexpr uint64_t kSmallCallBytes = 1ull << 20;

uint64_t total_bytes(const std::vector<SecDesc>& d) {
  uint64_t t = 0;
  for (const auto& x : d) t += x.bytes;
  return t;
}

// Give every stream its node slots and its kernel.  bulk[i] says which.
bool plan_streams(const pcs_ctx* c, std::vector<SecDesc>& d, const std::vector<char>& bulk,
                  StreamPlan& P, bool allow_reduce = true) {
  uint64_t reg_chunks = 0;
  size_t n_bulk = 0;
  for (size_t i = 0; i < d.size(); ++i) {
    if (!bulk[i]) reg_chunks += d[i].n_chunks;
    n_bulk += bulk[i] ? 1 : 0;
  }
  P.bulk_ids.reserve(n_bulk);
  P.bulk_begin.reserve(n_bulk);
  P.reg_ids.reserve(d.size() - n_bulk);
  P.reg_begin.reserve(d.size() - n_bulk);
  P.glog2 = choose_group_log2(c, reg_chunks);
  uint64_t node = 0, tb = 0, tr = 0;
  for (size_t i = 0; i < d.size(); ++i) {
    uint64_t n;
    if (bulk[i]) {
      n = (d[i].n_chunks + kBulkTileChunks - 1) / kBulkTileChunks;
      P.bulk_ids.push_back(static_cast<uint32_t>(i));
      P.bulk_begin.push_back(static_cast<uint32_t>(tb));
      tb += n;
    } else {
      n = (d[i].n_chunks + (1ull << P.glog2) - 1) >> P.glog2;
      P.reg_ids.push_back(static_cast<uint32_t>(i));
      P.reg_begin.push_back(static_cast<uint32_t>(tr));
      tr += n;
    }
    d[i].task_begin = static_cast<uint32_t>(node);
    d[i].n_tasks = static_cast<uint32_t>(n);
    node += n;
  }
  P.bulk_tasks = static_cast<uint32_t>(tb);
  P.reg_tasks = static_cast<uint32_t>(tr);
  P.nodes = node;
  // A stream with many task nodes would leave one finalising warp a long
  // serial tree: reduce aligned groups of 32 nodes across the GPU, level by
  // level, until no stream has more than 32 nodes left.  Aligned groups of
  // 32^k nodes reduce to the nodes of the global pairwise tree.  Up to
  // kFinRegNodes (1,024) nodes the finalising warp trees them from its
  // registers quicker than another launch (measured with the lane-local
  // register tree: the 64-bank step, whose latent sections have up to 512
  // tiles, 0.236 -> 0.234 ms without its two reduction launches; with the
  // earlier tree of 32-node groups a threshold of 256 was the better one).
  for (auto& x : d) {
    x.fin_begin = x.task_begin;
    x.fin_count = x.n_tasks;
  }
  uint64_t max_count = 0;
  for (const auto& x : d) max_count = std::max<uint64_t>(max_count, x.n_tasks);
  uint64_t groups = 0;
  if (allow_reduce && max_count > kFinRegNodes) {
    while (max_count > 32) {
      const uint64_t level_base = node + groups;
      uint64_t level_groups = 0;
      max_count = 0;
      for (auto& x : d) {
        NodeLevel L{};
        L.src = x.fin_begin;
        L.count = x.fin_count;
        L.dst = static_cast<uint32_t>(level_base + level_groups);
        const uint32_t out = (x.fin_count + 31) / 32;
        level_groups += out;
        x.fin_begin = L.dst;
        x.fin_count = out;
        max_count = std::max<uint64_t>(max_count, out);
        P.levels.push_back(L);
      }
      P.level_base.push_back(static_cast<uint32_t>(level_base));
      P.level_groups.push_back(static_cast<uint32_t>(level_groups));
      groups += level_groups;
    }
  }
  P.reduce_groups = static_cast<uint32_t>(groups);
  P.nodes_total = node + groups;
  return P.nodes_total < (1ull << 32);
}

// ---------------------------------------------------------------------------
// Plan checks (PCS_CHECK=1 at pcs_create): before anything is uploaded or
// launched, every descriptor, work list and reduction level of a call is
// checked against the invariants the kernels rely on -- node slots inside
// the call's node array, work lists that cover each stream's tasks exactly
// once, layouts the kernels can address, and record payloads inside their
// record and block.  A failure is a planner bug: the call returns
// PCS_E_INVAL naming the broken invariant and launches nothing.  compute-
// sanitizer being unavailable, this is the bounds check of host-planned
// offsets; index values read on the device are bounds-checked by the
// kernels themselves.
// ---------------------------------------------------------------------------

std::string check_streams(const std::vector<SecDesc>& d, const std::vector<char>& bulk,
                          const StreamPlan& P) {
  char msg[256];
  auto bad = [&](const char* fmt, auto... a) {
    std::snprintf(msg, sizeof msg, fmt, a...);
    return std::string(msg);
  };
  std::vector<int> seen(d.size(), 0);
  auto walk = [&](const std::vector<uint32_t>& ids, const std::vector<uint32_t>& begin,
                  uint32_t total, bool is_bulk) -> std::string {
    if (ids.size() != begin.size()) return bad("work list of %zu ids, %zu begins", ids.size(), begin.size());
    uint64_t t = 0;
    for (size_t j = 0; j < ids.size(); ++j) {
      if (ids[j] >= d.size()) return bad("work list item %zu names stream %u of %zu", j, ids[j], d.size());
      if (begin[j] != t) return bad("work list item %zu begins at task %u, expected %llu", j,
                                    begin[j], static_cast<unsigned long long>(t));
      if (static_cast<bool>(bulk[ids[j]]) != is_bulk) return bad("stream %u in the wrong kernel's list", ids[j]);
      ++seen[ids[j]];
      t += d[ids[j]].n_tasks;
    }
    if (t != total) return bad("work list covers %llu tasks, plan says %u",
                               static_cast<unsigned long long>(t), total);
    return {};
  };
  std::string e = walk(P.bulk_ids, P.bulk_begin, P.bulk_tasks, true);
  if (e.empty()) e = walk(P.reg_ids, P.reg_begin, P.reg_tasks, false);
  if (!e.empty()) return e;
  for (size_t i = 0; i < d.size(); ++i) {
    const SecDesc& x = d[i];
    if (seen[i] != 1) return bad("stream %zu appears in %d work lists", i, seen[i]);
    if (x.n_chunks != n_chunks_of(x.bytes)) return bad("stream %zu: %llu chunks for %llu bytes", i,
                                                        static_cast<unsigned long long>(x.n_chunks),
                                                        static_cast<unsigned long long>(x.bytes));
    const uint64_t per = bulk[i] ? kBulkTileChunks : (1ull << P.glog2);
    if (x.n_tasks != (x.n_chunks + per - 1) / per) return bad("stream %zu: %u tasks for %llu chunks", i,
                                                              x.n_tasks,
                                                              static_cast<unsigned long long>(x.n_chunks));
    if (static_cast<uint64_t>(x.task_begin) + x.n_tasks > P.nodes)
      return bad("stream %zu: task nodes end past the %llu nodes", i,
                 static_cast<unsigned long long>(P.nodes));
    if (x.fin_count < 1 || static_cast<uint64_t>(x.fin_begin) + x.fin_count > P.nodes_total)
      return bad("stream %zu: finalisation nodes [%u, +%u) outside %llu", i, x.fin_begin, x.fin_count,
                 static_cast<unsigned long long>(P.nodes_total));
    if (x.layout == kContig) {
      if (x.bytes && !x.lbase) return bad("stream %zu: no base", i);
      if (reinterpret_cast<uintptr_t>(x.lbase) % x.align) return bad("stream %zu: alignment %u wrong", i, x.align);
      if (bulk[i] && x.bytes && x.align != 16) return bad("stream %zu: TMA stream off 16 bytes", i);
    } else {
      if (x.layout != kRows && x.layout != kRing) return bad("stream %zu: layout %u", i, x.layout);
      if (x.row_bytes == 0 || (x.bytes && !x.index) || x.base_rows == 0)
        return bad("stream %zu: rows without size, index or bound", i);
      if (bulk[i] && (x.row_bytes < kBulkMinRowBytes || x.row_bytes % 16))
        return bad("stream %zu: TMA rows of %llu bytes", i, static_cast<unsigned long long>(x.row_bytes));
      if (x.layout == kRing &&
          (x.window == 0 || x.page_rows == 0 || x.window % x.page_rows || x.ring_start >= x.window ||
           x.bytes > static_cast<uint64_t>(x.window) * x.row_bytes))
        return bad("stream %zu: ring window %u, pages of %u rows, start %u", i, x.window, x.page_rows,
                   x.ring_start);
    }
  }
  const size_t ns = d.size();
  for (size_t k = 0; k < P.level_groups.size(); ++k)
    for (size_t i = 0; i < ns; ++i) {
      const NodeLevel& L = P.levels[k * ns + i];
      if (static_cast<uint64_t>(L.src) + L.count > P.nodes_total ||
          static_cast<uint64_t>(L.dst) + (L.count + 31) / 32 > P.nodes_total ||
          L.dst < P.level_base[k] || L.dst + (L.count + 31) / 32 > P.level_base[k] + P.level_groups[k])
        return bad("reduction level %zu of stream %zu outside its nodes", k, i);
    }
  return {};
}

// Records of a checkpoint or restore: sessions cover the streams in order,
// record s lies in its block [block[s].first, block[s].second), each payload
// inside its record.
std::string check_sessions(const std::vector<SecDesc>& d, const std::vector<SessDesc>& sd,
                           const std::vector<std::pair<const uint8_t*, const uint8_t*>>& block) {
  char msg[256];
  uint32_t next = 0;
  for (size_t s = 0; s < sd.size(); ++s) {
    const SessDesc& S = sd[s];
    if (S.sec_begin != next || S.n_sections < 1 || S.sec_begin + S.n_sections > d.size()) {
      std::snprintf(msg, sizeof msg, "session %zu: sections [%u, +%u) out of order", s, S.sec_begin,
                    S.n_sections);
      return msg;
    }
    next = S.sec_begin + S.n_sections;
    if (S.record < block[s].first || S.record + S.total_bytes > block[s].second ||
        S.payload_start > S.total_bytes ||
        S.payload_start % kRecordAlign ||
        S.payload_start < kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * S.n_sections) {
      std::snprintf(msg, sizeof msg, "session %zu: record outside its block or table overlap", s);
      return msg;
    }
    for (uint32_t j = 0; j < S.n_sections; ++j) {
      const SecDesc& x = d[S.sec_begin + j];
      const uint64_t off = static_cast<uint64_t>(x.payload - S.record);
      if (x.payload < S.record + S.payload_start || off % kRecordAlign ||
          off + round_up(x.bytes, kRecordAlign) > S.total_bytes || x.sess != s) {
        std::snprintf(msg, sizeof msg, "session %zu section %u: payload outside its record", s, j);
        return msg;
      }
    }
  }
  if (next != d.size()) {
    std::snprintf(msg, sizeof msg, "sessions cover %u of %zu streams", next, d.size());
    return msg;
  }
  return {};
}

// A small call whose streams all take the register kernel runs in one
// launch (k_small): the streaming pass and its finalisation.
constexpr int kSmallMaxItems = 64;

bool fused_ok(const std::vector<char>& bulk, bool small, int n_items) {
  if (!small || n_items > kSmallMaxItems) return false;
  for (char b : bulk)
    if (b) return false;
  return true;
}

// Workspace offsets of a stream plan's lists, after `base` bytes.
struct ListLayout {
  uint64_t bulk_ids, bulk_begin, reg_ids, reg_begin, levels, end;
};

ListLayout list_layout(const StreamPlan& P, uint64_t base) {
  ListLayout L;
  L.bulk_ids = round_up(base, kRecordAlign);
  L.bulk_begin = L.bulk_ids + 4 * P.bulk_ids.size();
  L.reg_ids = L.bulk_begin + 4 * P.bulk_begin.size();
  L.reg_begin = L.reg_ids + 4 * P.reg_ids.size();
  L.levels = round_up(L.reg_begin + 4 * P.reg_begin.size(), 16);
  L.end = L.levels + sizeof(NodeLevel) * P.levels.size();
  return L;
}

template <class T>
void put(uint8_t* plan, uint64_t off, const std::vector<T>& v) {
  if (!v.empty()) std::memcpy(plan + off, v.data(), v.size() * sizeof(T));
}
template <class T>
void put(std::vector<uint8_t>& plan, uint64_t off, const std::vector<T>& v) {
  put(plan.data(), off, v);
}

void put_lists(uint8_t* plan, const StreamPlan& P, const ListLayout& L) {
  put(plan, L.bulk_ids, P.bulk_ids);
  put(plan, L.bulk_begin, P.bulk_begin);
  put(plan, L.reg_ids, P.reg_ids);
  put(plan, L.reg_begin, P.reg_begin);
  put(plan, L.levels, P.levels);
}
void put_lists(std::vector<uint8_t>& plan, const StreamPlan& P, const ListLayout& L) {
  put_lists(plan.data(), P, L);
}

// Launch both streaming kernels of a plan (TMA-staged first).
cudaError_t launch_streams(pcs_ctx* c, int mode, const SecDesc* dsecs, const StreamPlan& P,
                           const ListLayout& L, uint8_t* ws, uint64_t* nodes,
                           cudaStream_t stream);

// Fingerprint (and optionally classify) contiguous buffers.
pcs_status fingerprint_impl(pcs_ctx* c, const pcs_buf* bufs, int32_t n, uint64_t* fp_out,
                            const uint64_t* fp_before, uint8_t* flags, void* stream_) {
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  if (n < 0 || (n > 0 && !bufs)) return fail(PCS_E_INVAL, "bad buffer list");
  if (n == 0) return PCS_OK;
  std::vector<SecDesc> d(n);
  uint64_t chunks = 0;
  for (int i = 0; i < n; ++i) {
    if (bufs[i].bytes > 0 && !bufs[i].ptr) return fail(PCS_E_INVAL, "buffer %d: null pointer", i);
    pcs_section s{};
    s.layout = PCS_LAYOUT_CONTIG;
    s.base = const_cast<void*>(bufs[i].ptr);
    s.bytes = bufs[i].bytes;
    d[i] = make_desc(s, nullptr, 0);
    chunks += d[i].n_chunks;
  }
  (void)chunks;
  PtrCache cache;
  std::vector<char> bulk(n);
  const bool small = total_bytes(d) <= kSmallCallBytes;
  for (int i = 0; i < n; ++i) bulk[i] = bulk_eligible(c, d[i], true, small, cache);
  const bool fused = fused_ok(bulk, small, n);
  StreamPlan P;
  if (!plan_streams(c, d, bulk, P, !fused)) return fail(PCS_E_INVAL, "too much data in one call");
  P.link_bound = link_bound_call(d, bulk, std::vector<char>(n, 1), cache);
  if (c->check_plans) {
    const std::string e = check_streams(d, bulk, P);
    if (!e.empty()) return fail(PCS_E_INVAL, "plan check: %s", e.c_str());
  }
  WsLayout L;
  L.secs = 0;
  const ListLayout LL = list_layout(P, sizeof(SecDesc) * n);
  L.nodes = round_up(LL.end, kRecordAlign);
  L.total = L.nodes + 8 * P.nodes_total;
  uint8_t* ws = nullptr;
  pcs_status st = ws_acquire(c, L.total, stream, &ws);
  if (st) return st;
  c->plan.resize(L.nodes);
  put(c->plan, L.secs, d);
  put_lists(c->plan, P, LL);
  PCS_CUDA(plan_copy(c, ws, L.nodes, stream));
  auto* dsecs = reinterpret_cast<const SecDesc*>(ws + L.secs);
  auto* nodes = reinterpret_cast<uint64_t*>(ws + L.nodes);
  if (fused) {
    WorkList wl{reinterpret_cast<const uint32_t*>(ws + LL.reg_ids),
                reinterpret_cast<const uint32_t*>(ws + LL.reg_begin),
                static_cast<int>(P.reg_ids.size()), P.reg_tasks};
    LaunchScope ls(c, kKStreamHash, stream);
    PCS_CUDA(launch_small(kModeHash, dsecs, wl, P.glog2, nodes, c->words, c->call_words, n, nullptr,
                          nullptr, fp_out, fp_before, flags, nullptr, c->sm_count, c->stream_bps,
                          stream));
    return ws_release(c, stream);
  }
  PCS_CUDA(launch_streams(c, kModeHash, dsecs, P, LL, ws, nodes, stream));
  {
    LaunchScope ls(c, kKFinalizeHash, stream);
    PCS_CUDA(launch_finalize(kModeHash, dsecs, nullptr, n, nullptr, nodes, fp_out, fp_before,
                             flags, nullptr, 0, stream));
  }
  return ws_release(c, stream);
}

cudaError_t launch_streams(pcs_ctx* c, int mode, const SecDesc* dsecs, const StreamPlan& P,
                           const ListLayout& L, uint8_t* ws, uint64_t* nodes,
                           cudaStream_t stream) {
  cudaError_t e = cudaSuccess;
  if (P.bulk_tasks) {
    WorkList wl{reinterpret_cast<const uint32_t*>(ws + L.bulk_ids),
                reinterpret_cast<const uint32_t*>(ws + L.bulk_begin),
                static_cast<int>(P.bulk_ids.size()), P.bulk_tasks};
    LaunchScope ls(c, bulk_kind(mode), stream);
    e = launch_bulk(mode, dsecs, wl, nodes, c->words, header_words(ws) + kWordBulkSched, c->sm_count,
                    stream);
    if (e != cudaSuccess) return e;
  }
  if (P.reg_tasks) {
    WorkList wl{reinterpret_cast<const uint32_t*>(ws + L.reg_ids),
                reinterpret_cast<const uint32_t*>(ws + L.reg_begin),
                static_cast<int>(P.reg_ids.size()), P.reg_tasks};
    LaunchScope ls(c, stream_kind(mode), stream);
    e = launch_stream(mode, dsecs, wl, P.glog2, nodes, c->words, grid_sms(c, P), c->stream_bps,
                      stream);
    if (e != cudaSuccess) return e;
  }
  if (nodes && P.reduce_groups) {
    const int n_streams = static_cast<int>(P.bulk_ids.size() + P.reg_ids.size());
    const auto* lv = reinterpret_cast<const NodeLevel*>(ws + L.levels);
    for (size_t k = 0; k < P.level_groups.size() && e == cudaSuccess; ++k) {
      LaunchScope ls(c, kKReduce, stream);
      e = launch_reduce_nodes(lv + k * n_streams, n_streams, nodes, P.level_base[k],
                              P.level_groups[k], c->sm_count, stream);
    }
  }
  return e;
}

pcs_snapshot* check_handle(pcs_ctx* c, const pcs_snapshot* h) {
  return c->live.count(h) ? const_cast<pcs_snapshot*>(h) : nullptr;
}

// Handle objects: a deleted handle's object serves the next snapshot (calls
// on thousands of sessions make and drop that many handles each).
constexpr size_t kMaxSpareHandles = 1 << 20;

std::unique_ptr<pcs_snapshot> new_snapshot(pcs_ctx* c) {
  if (c->spare.empty()) return std::make_unique<pcs_snapshot>();
  pcs_snapshot* h = c->spare.back();
  c->spare.pop_back();
  return std::unique_ptr<pcs_snapshot>(h);
}

void drop_snapshot(pcs_ctx* c, pcs_snapshot* h) {
  *h = pcs_snapshot{};
  if (c->spare.size() < kMaxSpareHandles) {
    c->spare.push_back(h);
  } else {
    delete h;
  }
}

// A checkpoint or a restore, planned: the descriptors (host bytes, uploaded
// to [0, L.nodes) of a workspace) and how to launch its kernels.
struct Prepared {
  int mode = kModePack;  // kModePack, kModeRestore, kModeRestoreV
  bool fused = false;    // one k_small launch (small calls)
  int verify = 0;        // restore: 0, 1 or 2
  int32_t n = 0;         // sessions
  int32_t max_secs = 0;  // most sections in one session
  StreamPlan P;
  ListLayout LL{};
  WsLayout L;
  std::vector<uint8_t> plan;
};

// The bytes [0, L.nodes) of a plan's descriptors: a plain call writes them
// straight into a pinned plan slot (one copy less; plan_send then sends
// them), a prepared call into pr->plan, which it keeps.
uint8_t* plan_target(pcs_ctx* c, Prepared* pr, bool to_slot) {
  if (to_slot) return plan_dst(c, pr->L.nodes, pr->plan);
  pr->plan.resize(pr->L.nodes);
  return pr->plan.data();
}

}  // namespace

// A prepared call: its descriptors in a device buffer of its own, and one
// reference on every record block it writes or reads.
struct pcs_plan {
  Prepared pr;
  uint8_t* dev = nullptr;
  std::vector<Block*> blocks;
};

namespace {

void destroy_plan(pcs_ctx* c, pcs_plan* p) {
  if (p->dev) cudaFree(p->dev);  // waits for the device
  for (Block* b : p->blocks) release_block(c, b);
  delete p;
}

void destroy_plans(pcs_ctx* c) {
  for (auto* p : c->plans) destroy_plan(c, p);
  c->plans.clear();
}

// The plan's own device copy of its descriptors, with room for its nodes,
// after a header of its own device words (zero), as in a workspace.
pcs_status plan_upload(pcs_plan* p) {
  PCS_CUDA(cudaMalloc(&p->dev, kWsHeader + std::max<uint64_t>(p->pr.L.total, 16)));
  PCS_CUDA(cudaMemset(p->dev, 0, kWsHeader));
  if (!p->pr.plan.empty())
    PCS_CUDA(cudaMemcpy(p->dev + kWsHeader, p->pr.plan.data(), p->pr.plan.size(),
                        cudaMemcpyHostToDevice));
  return PCS_OK;
}

uint8_t* plan_ws(const pcs_plan* p) { return p->dev + kWsHeader; }
uint32_t* plan_words(const pcs_plan* p) { return reinterpret_cast<uint32_t*>(p->dev); }

// Launch a prepared call whose descriptors are at `ws` (nodes after them);
// `words` are the call's header words (ticket of the fused kernel).
cudaError_t launch_prepared(pcs_ctx* c, const Prepared& pr, uint8_t* ws, uint32_t* words,
                            cudaStream_t stream) {
  const auto* dsecs = reinterpret_cast<const SecDesc*>(ws + pr.L.secs);
  const auto* dsess = reinterpret_cast<const SessDesc*>(ws + pr.L.sess);
  auto* nodes = reinterpret_cast<uint64_t*>(ws + pr.L.nodes);
  WorkList wl{reinterpret_cast<const uint32_t*>(ws + pr.LL.reg_ids),
              reinterpret_cast<const uint32_t*>(ws + pr.LL.reg_begin),
              static_cast<int>(pr.P.reg_ids.size()), pr.P.reg_tasks};
  if (pr.mode == kModePack) {
    const auto* dent = reinterpret_cast<const Entry*>(ws + pr.L.entries);
    if (pr.fused) {
      LaunchScope ls(c, kKStreamPack, stream);
      return launch_small(kModePack, dsecs, wl, pr.P.glog2, nodes, c->words, words, pr.n,
                          dsess, dent, nullptr, nullptr, nullptr, nullptr, c->sm_count,
                          c->stream_bps, stream);
    }
    cudaError_t e = launch_streams(c, kModePack, dsecs, pr.P, pr.LL, ws, nodes, stream);
    if (e != cudaSuccess) return e;
    LaunchScope ls(c, kKFinalizePack, stream);
    return launch_finalize(kModePack, dsecs, dsess, pr.n, dent, nodes, nullptr, nullptr, nullptr,
                           nullptr, pr.max_secs, stream);
  }
  uint32_t* bad = pr.verify == 1 ? words + 1 : c->words + 2;
  if (pr.fused) {
    LaunchScope ls(c, kKStreamRestoreV, stream);
    return launch_small(kModeRestoreV, dsecs, wl, pr.P.glog2, nodes, c->words, words, pr.n,
                        dsess, nullptr, nullptr, nullptr, nullptr, bad, c->sm_count,
                        c->stream_bps, stream);
  }
  cudaError_t e = launch_streams(c, pr.verify ? kModeRestoreV : kModeRestore, dsecs, pr.P, pr.LL,
                                 ws, pr.verify ? nodes : nullptr, stream);
  if (e != cudaSuccess || !pr.verify) return e;
  LaunchScope ls(c, kKFinalizeRestoreV, stream);
  return launch_finalize(kModeRestoreV, dsecs, dsess, pr.n, nullptr, nodes, nullptr, nullptr,
                         nullptr, bad, pr.max_secs, stream);
}

// Plan a checkpoint of n sessions: validate, reserve one block for their
// records (on `stream`), create the handles (not yet live), build the
// descriptors.  On failure nothing is left reserved.
pcs_status build_checkpoint(pcs_ctx* c, const pcs_session* sessions, int32_t n, uint32_t placement,
                            cudaStream_t stream, Prepared* pr, Block** blk_out,
                            std::vector<std::unique_ptr<pcs_snapshot>>* handles,
                            bool to_slot = false) {
  if (placement != PCS_PLACE_DEVICE && placement != PCS_PLACE_PINNED_HOST)
    return fail(PCS_E_INVAL, "unknown placement %u", placement);
  // Plan records: sizes, offsets, entries.
  std::vector<uint64_t> rec_off(n + 1, 0), pstart(n);
  uint64_t total_secs = 0;
  for (int s = 0; s < n; ++s) {
    const pcs_session& S = sessions[s];
    if (S.n_sections < 1 || S.n_sections > 65535 || !S.sections)
      return fail(PCS_E_INVAL, "session %d: needs 1..65535 sections", s);
    for (int i = 0; i < S.n_sections; ++i) {
      pcs_status st = check_section(S.sections[i], s, i, false);
      if (st) return st;
    }
    uint64_t bytes = 0;
    pcs_record_bytes(S.sections, S.n_sections, &bytes);
    pstart[s] = round_up(kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * S.n_sections, kRecordAlign);
    rec_off[s + 1] = rec_off[s] + bytes;
    total_secs += S.n_sections;
  }
  if (total_secs > 0x7FFFFFFFull) return fail(PCS_E_INVAL, "too many sections in one call");
  Block* blk = nullptr;
  pcs_status st = arena_of(c, placement)->alloc(rec_off[n], stream, &blk);
  if (st) return st;
  std::vector<SecDesc> d;
  std::vector<SessDesc> sd(n);
  auto ent_shared = std::make_shared<std::vector<Entry>>();
  std::vector<Entry>& ent = *ent_shared;  // the section tables of every record
  d.reserve(total_secs);
  ent.reserve(total_secs);
  handles->resize(n);
  for (int s = 0; s < n; ++s) {
    const pcs_session& S = sessions[s];
    uint8_t* rec = blk->ptr + rec_off[s];
    auto h = new_snapshot(c);
    h->block = blk;
    h->offset = rec_off[s];
    h->total_bytes = rec_off[s + 1] - rec_off[s];
    h->payload_start = pstart[s];
    h->session_id = S.session_id;
    h->kind = S.kind;
    h->first = static_cast<uint32_t>(ent.size());
    h->n_sections = static_cast<uint32_t>(S.n_sections);
    sd[s].record = rec;
    sd[s].total_bytes = h->total_bytes;
    sd[s].payload_start = pstart[s];
    sd[s].sec_begin = static_cast<uint32_t>(d.size());
    sd[s].n_sections = static_cast<uint32_t>(S.n_sections);
    sd[s].session_id = S.session_id;
    sd[s].kind = S.kind;
    uint64_t off = pstart[s];
    for (int i = 0; i < S.n_sections; ++i) {
      const pcs_section& x = S.sections[i];
      d.push_back(make_desc(x, rec + off, x.ring_start));
      d.back().sess = static_cast<uint32_t>(s);
      Entry e{};
      e.type = x.type;
      e.dtype = x.dtype;
      e.layer = x.layer;
      e.layout = x.layout;
      e.offset = off;
      e.bytes = x.bytes;
      e.fp = 0;
      e.dim0 = x.dim0;
      e.dim1 = x.dim1;
      e.aux = x.layout == PCS_LAYOUT_RING ? x.ring_start : 0;
      ent.push_back(e);
      off = round_up(off + x.bytes, kRecordAlign);
    }
    (*handles)[s] = std::move(h);
  }
  for (auto& h : *handles) h->tables = ent_shared;
  PtrCache cache;
  std::vector<char> bulk(d.size());
  const bool small = total_bytes(d) <= kSmallCallBytes;
  for (size_t i = 0; i < d.size(); ++i)
    bulk[i] = bulk_eligible(c, d[i], placement == PCS_PLACE_DEVICE, small, cache);
  uint32_t max_secs = 0;
  for (int s = 0; s < n; ++s) max_secs = std::max<uint32_t>(max_secs, sd[s].n_sections);
  pr->mode = kModePack;
  pr->n = n;
  pr->max_secs = static_cast<int32_t>(max_secs);
  pr->fused = fused_ok(bulk, small, n) && max_secs <= 2048;
  if (!plan_streams(c, d, bulk, pr->P, !pr->fused)) {
    arena_of(c, placement)->free(blk);
    return fail(PCS_E_INVAL, "too much data in one call");
  }
  pr->P.link_bound =
      link_bound_call(d, bulk, std::vector<char>(d.size(), placement == PCS_PLACE_DEVICE), cache);
  if (c->check_plans) {
    std::string e = check_streams(d, bulk, pr->P);
    if (e.empty())
      e = check_sessions(d, sd, std::vector<std::pair<const uint8_t*, const uint8_t*>>(
                                    n, {blk->ptr, blk->ptr + blk->size}));
    if (!e.empty()) {
      arena_of(c, placement)->free(blk);
      return fail(PCS_E_INVAL, "plan check: %s", e.c_str());
    }
  }
  WsLayout& L = pr->L;
  L.secs = 0;
  L.sess = round_up(sizeof(SecDesc) * d.size(), kRecordAlign);
  L.entries = round_up(L.sess + sizeof(SessDesc) * n, kRecordAlign);
  pr->LL = list_layout(pr->P, L.entries + sizeof(Entry) * ent.size());
  L.nodes = round_up(pr->LL.end, kRecordAlign);
  L.total = L.nodes + 8 * pr->P.nodes_total;
  uint8_t* dst = plan_target(c, pr, to_slot);
  put(dst, L.secs, d);
  put(dst, L.sess, sd);
  put(dst, L.entries, ent);
  put_lists(dst, pr->P, pr->LL);
  *blk_out = blk;
  return PCS_OK;
}

// Plan a restore of n snapshots into n target sessions.
pcs_status build_restore(pcs_ctx* c, pcs_snapshot* const* snaps, int32_t n,
                         const pcs_session* targets, int verify, Prepared* pr,
                         bool to_slot = false) {
  std::vector<SecDesc> d;
  std::vector<SessDesc> sd(n);
  std::vector<char> payload_dev;
  uint64_t want = 0;
  for (int s = 0; s < n; ++s) want += targets[s].n_sections > 0 ? targets[s].n_sections : 0;
  d.reserve(std::min<uint64_t>(want, 1ull << 24));
  payload_dev.reserve(d.capacity());
  for (int s = 0; s < n; ++s) {
    pcs_snapshot* h = check_handle(c, snaps[s]);
    if (!h) return fail(PCS_E_HANDLE, "snapshot %d: unknown handle", s);
    const pcs_session& T = targets[s];
    if (T.n_sections != static_cast<int32_t>(h->n_sections) || !T.sections)
      return fail(PCS_E_INVAL, "session %d: target has %d sections, snapshot %zu", s,
                  T.n_sections, h->n_sections);
    sd[s].record = h->record();
    sd[s].total_bytes = h->total_bytes;
    sd[s].payload_start = h->payload_start;
    sd[s].sec_begin = static_cast<uint32_t>(d.size());
    sd[s].n_sections = static_cast<uint32_t>(T.n_sections);
    sd[s].session_id = h->session_id;
    sd[s].kind = h->kind;
    for (int i = 0; i < T.n_sections; ++i) {
      const pcs_section& x = T.sections[i];
      pcs_status st = check_section(x, s, i, true);
      if (st) return st;
      const Entry& e = h->table()[i];
      if (x.bytes != e.bytes)
        return fail(PCS_E_INVAL, "session %d section %d: target bytes %llu != snapshot %llu", s, i,
                    static_cast<unsigned long long>(x.bytes), static_cast<unsigned long long>(e.bytes));
      uint32_t rs = x.ring_start;
      if (x.layout == PCS_LAYOUT_RING && rs == PCS_RING_START_FROM_SNAPSHOT) {
        if (e.layout != PCS_LAYOUT_RING || e.aux >= x.window)
          return fail(PCS_E_INVAL, "session %d section %d: no stored ring start fits", s, i);
        rs = static_cast<uint32_t>(e.aux);
      }
      d.push_back(make_desc(x, h->record() + e.offset, rs));
      d.back().sess = static_cast<uint32_t>(s);
      payload_dev.push_back(h->block->placement == PCS_PLACE_DEVICE);
    }
  }
  PtrCache cache;
  std::vector<char> bulk(d.size());
  const bool small = total_bytes(d) <= kSmallCallBytes;
  for (size_t i = 0; i < d.size(); ++i) bulk[i] = bulk_eligible(c, d[i], payload_dev[i], small, cache);
  uint32_t max_secs = 0;
  for (int s = 0; s < n; ++s) max_secs = std::max<uint32_t>(max_secs, sd[s].n_sections);
  pr->mode = verify ? kModeRestoreV : kModeRestore;
  pr->verify = verify;
  pr->n = n;
  pr->max_secs = static_cast<int32_t>(max_secs);
  pr->fused = verify && fused_ok(bulk, small, n) && max_secs <= 2048;
  if (!plan_streams(c, d, bulk, pr->P, !pr->fused))
    return fail(PCS_E_INVAL, "too much data in one call");
  pr->P.link_bound = link_bound_call(d, bulk, payload_dev, cache);
  if (c->check_plans) {
    std::vector<std::pair<const uint8_t*, const uint8_t*>> blocks(n);
    for (int s = 0; s < n; ++s)
      blocks[s] = {snaps[s]->block->ptr, snaps[s]->block->ptr + snaps[s]->block->size};
    std::string e = check_streams(d, bulk, pr->P);
    if (e.empty()) e = check_sessions(d, sd, blocks);
    if (!e.empty()) return fail(PCS_E_INVAL, "plan check: %s", e.c_str());
  }
  WsLayout& L = pr->L;
  L.secs = 0;
  L.sess = round_up(sizeof(SecDesc) * d.size(), kRecordAlign);
  pr->LL = list_layout(pr->P, L.sess + sizeof(SessDesc) * n);
  L.nodes = round_up(pr->LL.end, kRecordAlign);
  L.total = L.nodes + (verify ? 8 * pr->P.nodes_total : 0);
  uint8_t* dst = plan_target(c, pr, to_slot);
  put(dst, L.secs, d);
  put(dst, L.sess, sd);
  put_lists(dst, pr->P, pr->LL);
  return PCS_OK;
}


}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" {

const char* pcs_last_error(void) { return g_err.c_str(); }

const char* pcs_status_string(pcs_status s) {
  switch (s) {
    case PCS_OK: return "PCS_OK";
    case PCS_E_INVAL: return "PCS_E_INVAL";
    case PCS_E_ALIGN: return "PCS_E_ALIGN";
    case PCS_E_NOMEM: return "PCS_E_NOMEM";
    case PCS_E_CUDA: return "PCS_E_CUDA";
    case PCS_E_BUDGET: return "PCS_E_BUDGET";
    case PCS_E_CORRUPT: return "PCS_E_CORRUPT";
    case PCS_E_HANDLE: return "PCS_E_HANDLE";
    case PCS_E_IO: return "PCS_E_IO";
    case PCS_E_TIMEOUT: return "PCS_E_TIMEOUT";
    case PCS_E_RANGE: return "PCS_E_RANGE";
    default: return "PCS_E_UNKNOWN";
  }
}

pcs_status pcs_create(int32_t device, pcs_ctx** out) {
  if (!out) return fail(PCS_E_INVAL, "out is null");
  *out = nullptr;
  int count = 0;
  cudaError_t e = cudaGetDeviceCount(&count);
  if (e != cudaSuccess || count == 0) {
    cudaGetLastError();
    return fail(PCS_E_CUDA, "no CUDA device available (%s)", cudaGetErrorString(e));
  }
  if (device < 0 || device >= count) return fail(PCS_E_INVAL, "device %d out of range", device);
  auto c = std::make_unique<pcs_ctx>();
  c->device = device;
  PCS_CUDA(cudaSetDevice(device));
  PCS_CUDA(cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, device));
  c->stream_bps = stream_blocks_per_sm();
  const char* no_tma = std::getenv("PCS_DISABLE_TMA");
  c->use_bulk = !(no_tma && no_tma[0] == '1');
  const char* check = std::getenv("PCS_CHECK");
  c->check_plans = check && check[0] == '1';
  c->dev_arena = std::make_unique<Arena>(PCS_PLACE_DEVICE, c->events);
  c->host_arena = std::make_unique<Arena>(PCS_PLACE_PINNED_HOST, c->events);
  PCS_CUDA(cudaMalloc(&c->words, 256));
  PCS_CUDA(cudaMemset(c->words, 0, 256));
  *out = c.release();
  return PCS_OK;
}

pcs_status pcs_destroy(pcs_ctx* c) {
  if (!c) return PCS_OK;
  {
    std::lock_guard<std::mutex> lk(c->mu);
    cudaSetDevice(c->device);
    cudaDeviceSynchronize();
    c->live.for_each([&](pcs_snapshot* h) {
      release_block(c, h->block);
      delete h;
    });
    c->live.clear();
    for (auto* h : c->spare) delete h;
    c->spare.clear();
    for (auto* pl : c->pools) {
      cudaFree(pl->meta);
      delete pl;
    }
    c->pools.clear();
    destroy_plans(c);
    for (auto& kv : c->ws) {
      kv.second.busy.reset();
      if (kv.second.buf) cudaFree(kv.second.buf);
    }
    c->ws.clear();
    if (c->words) cudaFree(c->words);
    if (c->stage) cudaFreeHost(c->stage);
    for (auto& e : c->plan_slot_busy) e.reset();
    for (uint8_t* b : c->plan_slot_buf)
      if (b) cudaFreeHost(b);
    for (auto& t : c->timed) {
      cudaEventDestroy(t.start);
      cudaEventDestroy(t.stop);
    }
    for (auto e : c->timing_events) cudaEventDestroy(e);
    c->dev_arena.reset();
    c->host_arena.reset();
  }
  delete c;
  return PCS_OK;
}

pcs_status pcs_set_arena_limit(pcs_ctx* c, uint32_t placement, uint64_t bytes) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (placement != PCS_PLACE_DEVICE && placement != PCS_PLACE_PINNED_HOST)
    return fail(PCS_E_INVAL, "unknown placement %u", placement);
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  arena_of(c, placement)->set_limit(bytes);
  return PCS_OK;
}

pcs_status pcs_get_stats(pcs_ctx* c, pcs_stats* out) {
  if (!c || !out) return fail(PCS_E_INVAL, "null argument");
  std::lock_guard<std::mutex> lk(c->mu);
  out->kernel_launches = c->launches;
  out->device_reserved = c->dev_arena->reserved();
  out->host_reserved = c->host_arena->reserved();
  out->live_snapshots = static_cast<int32_t>(c->live.size());
  out->sm_count = c->sm_count;
  return PCS_OK;
}

pcs_status pcs_timing_enable(pcs_ctx* c, int32_t on) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  for (auto& t : c->timed) {
    cudaEventSynchronize(t.stop);
    c->timing_events.push_back(t.start);
    c->timing_events.push_back(t.stop);
  }
  c->timed.clear();
  for (int i = 0; i < kKernelKinds; ++i) {
    c->kernel_ms[i] = 0;
    c->kernel_n[i] = 0;
  }
  c->timing = on != 0;
  return PCS_OK;
}

pcs_status pcs_timing_read(pcs_ctx* c, pcs_kernel_time* out, int32_t max, int32_t* n) {
  if (!c || !n || (max > 0 && !out)) return fail(PCS_E_INVAL, "null argument");
  std::lock_guard<std::mutex> lk(c->mu);
  for (auto& t : c->timed) {
    float ms = 0;
    PCS_CUDA(cudaEventSynchronize(t.stop));
    PCS_CUDA(cudaEventElapsedTime(&ms, t.start, t.stop));
    c->kernel_ms[t.kind] += ms;
    c->kernel_n[t.kind] += 1;
    c->timing_events.push_back(t.start);
    c->timing_events.push_back(t.stop);
  }
  c->timed.clear();
  int32_t k = 0;
  for (int i = 0; i < kKernelKinds; ++i) {
    if (c->kernel_n[i] == 0) continue;
    if (k < max) {
      std::snprintf(out[k].name, sizeof out[k].name, "%s", kKernelNames[i]);
      out[k].launches = c->kernel_n[i];
      out[k].total_ms = c->kernel_ms[i];
    }
    ++k;
  }
  *n = k;
  return PCS_OK;
}

pcs_status pcs_sync(pcs_ctx* c, void* stream) {
  PCS_TRACE("pcs_sync");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  PCS_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  uint32_t w3[3] = {0, 0, 0};
  PCS_CUDA(cudaMemcpy(w3, c->words, sizeof w3, cudaMemcpyDeviceToHost));
  const uint32_t w = w3[0];
  if (w3[2] != 0) {
    PCS_CUDA(cudaMemset(c->words + 2, 0, 4));
    if (w) PCS_CUDA(cudaMemset(c->words, 0, 4));
    return fail(PCS_E_CORRUPT, "%u restored sessions failed asynchronous verification", w3[2]);
  }
  if (w != 0) {
    PCS_CUDA(cudaMemset(c->words, 0, 4));
    if (w & kDevErrTimeout)
      return fail(PCS_E_TIMEOUT, "a bounded wait inside a kernel gave up (error bits 0x%x)", w);
    if (w & kDevErrNoPage)
      return fail(PCS_E_NOMEM, "a page pool had no free page (error bits 0x%x)", w);
    if (w & kDevErrRefcount)
      return fail(PCS_E_INVAL,
                  "a pool page was shared, written or released while held by nobody "
                  "(error bits 0x%x)", w);
    return fail(PCS_E_RANGE, "a kernel met a row or page id out of range (error bits 0x%x)", w);
  }
  return PCS_OK;
}

pcs_status pcs_selftest_wait(pcs_ctx* c, int32_t which, void* stream) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (which != 0 && which != 1) return fail(PCS_E_INVAL, "which must be 0 or 1, got %d", which);
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  // words[4] is zeroed at creation and never written: nothing will set it.
  PCS_CUDA(launch_selftest_wait(which, c->words + 4, c->words, static_cast<cudaStream_t>(stream)));
  ++c->launches;
  return PCS_OK;
}

pcs_status pcs_fingerprint(pcs_ctx* c, const pcs_buf* bufs, int32_t n, uint64_t* fp_out,
                           void* stream) {
  PCS_TRACE("pcs_fingerprint");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (n > 0 && !fp_out) return fail(PCS_E_INVAL, "fp_out is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  return fingerprint_impl(c, bufs, n, fp_out, nullptr, nullptr, stream);
}

pcs_status pcs_classify(pcs_ctx* c, const pcs_buf* bufs, int32_t n, const uint64_t* fp_before,
                        uint64_t* fp_after, uint8_t* must_snapshot, void* stream) {
  PCS_TRACE("pcs_classify");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (n > 0 && (!fp_before || !must_snapshot))
    return fail(PCS_E_INVAL, "fp_before and must_snapshot are required");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  return fingerprint_impl(c, bufs, n, fp_after, fp_before, must_snapshot, stream);
}

pcs_status pcs_prune_counts(const pcs_bank* banks, int32_t n, const pcs_prune_params* p,
                            int32_t* k_out) {
  if (n < 0 || (n > 0 && (!banks || !k_out)) || !p) return fail(PCS_E_INVAL, "bad arguments");
  for (int s = 0; s < n; ++s)
    if (banks[s].n_entries < 0) return fail(PCS_E_INVAL, "bank %d: negative n_entries", s);
  switch (p->rule) {
    case PCS_K_FIXED:
      if (p->k_max < 0) return fail(PCS_E_INVAL, "k_max < 0");
      for (int s = 0; s < n; ++s) k_out[s] = std::min(banks[s].n_entries, p->k_max);
      return PCS_OK;
    case PCS_K_BUDGET: {
      unsigned __int128 T = 0;
      for (int s = 0; s < n; ++s)
        T += static_cast<unsigned __int128>(static_cast<uint64_t>(banks[s].n_entries)) *
             banks[s].entry_bytes;
      // A population split over processes: every part uses the whole T.
      if (p->total_bytes != 0) {
        if (p->total_bytes < T)
          return fail(PCS_E_INVAL, "total_bytes is below the bytes of these banks");
        T = p->total_bytes;
      }
      for (int s = 0; s < n; ++s) {
        if (T <= p->budget_bytes) {
          k_out[s] = banks[s].n_entries;
        } else {
          const unsigned __int128 num =
              static_cast<unsigned __int128>(static_cast<uint64_t>(banks[s].n_entries)) *
              p->budget_bytes;
          k_out[s] = static_cast<int32_t>(num / T);
        }
      }
      return PCS_OK;
    }
    case PCS_K_FRACTION: {
      if (!(p->fraction >= 0.0 && p->fraction <= 1.0))
        return fail(PCS_E_INVAL, "fraction must lie in [0, 1]");
      for (int s = 0; s < n; ++s) {
        // Round to nearest, ties to even (default rounding mode).
        double v = __builtin_nearbyint(p->fraction * static_cast<double>(banks[s].n_entries));
        v = std::min<double>(std::max(v, 0.0), banks[s].n_entries);
        k_out[s] = static_cast<int32_t>(v);
      }
      return PCS_OK;
    }
    default:
      return fail(PCS_E_INVAL, "unknown k-rule %d", p->rule);
  }
}

// Validated scoring descriptors of n banks (k per bank, or all 0 if k is
// NULL), entry offsets bank-major; *entries = total entries.
pcs_status bank_descs(const pcs_bank* banks, int32_t n, const int32_t* k,
                      std::vector<BankDesc>* d, uint64_t* entries_out, uint32_t kept_align = 1) {
  d->assign(std::max(n, 0), BankDesc{});
  uint64_t entries = 0, kept = 0;
  for (int s = 0; s < n; ++s) {
    const pcs_bank& b = banks[s];
    if (b.key_dtype != PCS_DT_F16 && b.key_dtype != PCS_DT_BF16)
      return fail(PCS_E_INVAL, "bank %d: key_dtype must be F16 or BF16", s);
    if (b.key_dim <= 0 || b.key_dim % 8 != 0)
      return fail(PCS_E_ALIGN, "bank %d: key_dim must be a positive multiple of 8", s);
    if (b.n_entries < 0) return fail(PCS_E_INVAL, "bank %d: negative n_entries", s);
    if (b.n_entries > 0 && (!b.keys || !b.query))
      return fail(PCS_E_INVAL, "bank %d: null keys or query", s);
    if (b.n_entries > 0 && (!aligned16(b.keys) || !aligned16(b.query)))
      return fail(PCS_E_ALIGN, "bank %d: keys / query not 16-byte aligned", s);
    BankDesc& x = (*d)[s];
    x.keys = static_cast<const uint16_t*>(b.keys);
    x.query = static_cast<const uint16_t*>(b.query);
    x.entry_begin = entries;
    x.kept_begin = kept;
    x.n = b.n_entries;
    x.D = b.key_dim;
    x.k = k ? k[s] : 0;
    x.is_bf16 = b.key_dtype == PCS_DT_BF16;
    x.entry_bytes = b.entry_bytes;
    entries += b.n_entries;
    kept += round_up(static_cast<uint64_t>(x.k), kept_align);
  }
  if (entries > 0x7FFFFFFFull) return fail(PCS_E_INVAL, "too many entries in one call");
  *entries_out = entries;
  return PCS_OK;
}

// The relevance score of every entry (descriptors already on the device);
// with gh.st set, also the first digit pass of the global threshold where the
// score kernel can take it (*fused says whether it did).
cudaError_t launch_bank_scores(pcs_ctx* c, const pcs_bank* banks, int32_t n,
                               const BankDesc* dbanks, uint64_t entries, float* sc,
                               cudaStream_t stream, GHist gh = GHist{}, bool* fused = nullptr) {
  LaunchScope ls(c, kKScore, stream);
  int max_dim = 0, n_bf16 = 0;
  for (int s = 0; s < n; ++s) {
    max_dim = std::max(max_dim, banks[s].key_dim);
    n_bf16 += banks[s].key_dtype == PCS_DT_BF16;
  }
  const int key_types = n_bf16 == 0 ? 0 : (n_bf16 == n ? 1 : 2);
  return launch_score(dbanks, n, entries, max_dim, key_types, sc, c->sm_count, stream, gh, fused);
}

pcs_status pcs_prune(pcs_ctx* c, const pcs_bank* banks, int32_t n, const pcs_prune_params* p,
                     float* scores, int32_t* kept_idx, int32_t* kept_off, void* stream_) {
  PCS_TRACE("pcs_prune");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::vector<int32_t> k(std::max(n, 0));
  pcs_status st = pcs_prune_counts(banks, n, p, k.data());
  if (st) return st;
  if (n == 0) return PCS_OK;
  const uint32_t align = p->kept_align == 0 ? 1u : p->kept_align;
  if (align != 1 && align != 4) return fail(PCS_E_INVAL, "kept_align must be 0, 1 or 4");
  std::vector<BankDesc> d;
  uint64_t entries = 0;
  st = bank_descs(banks, n, k.data(), &d, &entries, align);
  if (st) return st;
  std::vector<int32_t> koff(n + 1, 0);
  uint64_t kept = 0;
  for (int s = 0; s < n; ++s) {
    kept += round_up(static_cast<uint64_t>(k[s]), align);
    koff[s + 1] = static_cast<int32_t>(kept);
  }
  if (kept > 0 && !kept_idx) return fail(PCS_E_INVAL, "kept_idx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  st = set_device(c);
  if (st) return st;
  WsLayout L;
  L.banks = 0;
  L.secs = round_up(sizeof(BankDesc) * n, kRecordAlign);       // kept offsets (int32)
  L.nodes = round_up(L.secs + 4ull * (n + 1), kRecordAlign);   // scores if caller gives none
  L.total = L.nodes + (scores ? 0 : 4 * entries);
  uint8_t* ws = nullptr;
  st = ws_acquire(c, L.total, stream, &ws);
  if (st) return st;
  c->plan.resize(L.nodes);
  put(c->plan, L.banks, d);
  put(c->plan, L.secs, koff);
  PCS_CUDA(plan_copy(c, ws, L.nodes, stream));
  if (kept_off)
    PCS_CUDA(cudaMemcpyAsync(kept_off, ws + L.secs, 4ull * (n + 1), cudaMemcpyDeviceToDevice, stream));
  float* sc = scores ? scores : reinterpret_cast<float*>(ws + L.nodes);
  auto* dbanks = reinterpret_cast<const BankDesc*>(ws + L.banks);
  PCS_CUDA(launch_bank_scores(c, banks, n, dbanks, entries, sc, stream));
  {
    LaunchScope ls(c, kKTopk, stream);
    PCS_CUDA(launch_topk(dbanks, n, sc, kept_idx, stream));
  }
  return ws_release(c, stream);
}

pcs_status pcs_topk(pcs_ctx* c, const float* keys, const int32_t* n, const int32_t* k,
                    int32_t n_banks, int32_t* kept_idx, int32_t* kept_off, void* stream_) {
  PCS_TRACE("pcs_topk");
  if (!c || n_banks < 0 || (n_banks > 0 && (!n || !k))) return fail(PCS_E_INVAL, "bad arguments");
  if (n_banks == 0) return PCS_OK;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::vector<BankDesc> d(n_banks);
  std::vector<int32_t> koff(n_banks + 1, 0);
  uint64_t entries = 0, kept = 0;
  for (int b = 0; b < n_banks; ++b) {
    if (n[b] < 0 || k[b] < 0) return fail(PCS_E_INVAL, "bank %d: negative n or k", b);
    d[b].entry_begin = entries;
    d[b].kept_begin = kept;
    d[b].n = n[b];
    d[b].k = std::min(k[b], n[b]);
    entries += n[b];
    kept += d[b].k;
    koff[b + 1] = static_cast<int32_t>(kept);
  }
  if (entries > 0 && !keys) return fail(PCS_E_INVAL, "keys is null");
  if (kept > 0 && !kept_idx) return fail(PCS_E_INVAL, "kept_idx is null");
  if (entries > 0x7FFFFFFFull) return fail(PCS_E_INVAL, "too many entries in one call");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  const uint64_t off_at = round_up(sizeof(BankDesc) * n_banks, kRecordAlign);
  const uint64_t total = off_at + 4ull * (n_banks + 1);
  uint8_t* ws = nullptr;
  st = ws_acquire(c, total, stream, &ws);
  if (st) return st;
  c->plan.resize(total);
  put(c->plan, 0, d);
  put(c->plan, off_at, koff);
  PCS_CUDA(plan_copy(c, ws, total, stream));
  if (kept_off)
    PCS_CUDA(cudaMemcpyAsync(kept_off, ws + off_at, 4ull * (n_banks + 1), cudaMemcpyDeviceToDevice,
                             stream));
  {
    LaunchScope ls(c, kKTopk, stream);
    PCS_CUDA(launch_topk(reinterpret_cast<const BankDesc*>(ws), n_banks, keys, kept_idx, stream));
  }
  return ws_release(c, stream);
}

// Digit schedule of the 64-bit ranking key (the same as the kernels'):
// 11, 11, 10 bits of ord32(score), then 11, 11, 10 bits of the position.
static const int kGDigitBits[kGPasses] = {11, 11, 10, 11, 11, 10};
static const int kGDigitShift[kGPasses] = {53, 42, 32, 21, 10, 0};

// The digit choice of one pass from histograms summed over all parts (the
// device's gselect_pick, on the host).  Returns true once the threshold is
// known.
static bool host_pick(int pass, const uint64_t* counts, const uint64_t* bytes, GState* g) {
  const int bits = kGDigitBits[pass], shift = kGDigitShift[pass];
  const uint64_t top = (1ull << bits) - 1;
  uint64_t cum = 0;
  for (int64_t bin = static_cast<int64_t>(top); bin >= 0; --bin) {
    if (cum + bytes[bin] > g->remaining) {
      g->prefix |= static_cast<uint64_t>(bin) << shift;
      g->mask |= top << shift;
      g->remaining -= cum;
      if (counts[bin] == 1 || shift == 0) {
        g->threshold = g->prefix | ~g->mask;
        return true;
      }
      return false;
    }
    cum += bytes[bin];
  }
  g->threshold = 0;  // every candidate fits
  return true;
}

// The digit passes of one part of a split population: histogram here, sum
// over the parts through `ex`, pick on the host, send the state back.
static pcs_status exchange_passes(pcs_ctx* c, const GPlan& gp, uint64_t budget,
                                  pcs_hist_exchange_fn ex, void* user, cudaStream_t stream) {
  std::vector<uint32_t> c32(kGBins);
  std::vector<uint64_t> counts(kGBins), bytes(kGBins);
  GState g{};
  g.remaining = budget;
  for (int pass = 0; pass < kGPasses; ++pass) {
    const int nb = 1 << kGDigitBits[pass];
    std::fill(counts.begin(), counts.end(), 0);
    std::fill(bytes.begin(), bytes.end(), 0);
    if (gp.tiles > 0) {
      {
        LaunchScope ls(c, kKGSelect, stream);
        PCS_CUDA(launch_gselect(gp, pass, c->sm_count, stream));
      }
      PCS_CUDA(cudaMemcpyAsync(c32.data(), gp.st->chist, 4ull * nb, cudaMemcpyDeviceToHost, stream));
      if (!gp.uniform)
        PCS_CUDA(cudaMemcpyAsync(bytes.data(), gp.st->whist, 8ull * nb, cudaMemcpyDeviceToHost,
                                 stream));
      PCS_CUDA(cudaMemsetAsync(gp.st->chist, 0, 4ull * kGBins, stream));
      PCS_CUDA(cudaMemsetAsync(gp.st->whist, 0, 8ull * kGBins, stream));
      PCS_CUDA(cudaStreamSynchronize(stream));
      for (int i = 0; i < nb; ++i) {
        counts[i] = c32[i];
        if (gp.uniform) bytes[i] = counts[i] * gp.uniform_bytes;
      }
    }
    const int32_t rc = ex(user, counts.data(), bytes.data(), nb);
    if (rc != 0) return fail(PCS_E_INVAL, "histogram exchange of pass %d returned %d", pass, rc);
    const bool done = host_pick(pass, counts.data(), bytes.data(), &g);
    g.done = done ? 1 : 0;
    // The header fields (prefix .. done) for the next pass and the compaction.
    PCS_CUDA(cudaMemcpyAsync(gp.st, &g, offsetof(GState, ticket), cudaMemcpyHostToDevice, stream));
    PCS_CUDA(cudaStreamSynchronize(stream));
    if (done) break;
  }
  return PCS_OK;
}

// The global threshold over these banks; with `ex`, these banks are one part
// of a population split over processes: each digit pass's histogram is
// summed over the parts by `ex` and the digit is picked on the host.
static pcs_status prune_global_impl(pcs_ctx* c, const pcs_bank* banks, int32_t n,
                                    uint64_t budget, float* scores, int32_t* kept_idx,
                                    int32_t* kept_off, void* stream_, pcs_hist_exchange_fn ex,
                                    void* user, uint64_t pos_base) {
  if (!c || n < 0 || (n > 0 && !banks)) return fail(PCS_E_INVAL, "bad arguments");
  if (!kept_off) return fail(PCS_E_INVAL, "kept_off is null");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::vector<BankDesc> d;
  uint64_t entries = 0;
  pcs_status st = bank_descs(banks, n, nullptr, &d, &entries);
  if (st) return st;
  if (entries > 0 && !kept_idx) return fail(PCS_E_INVAL, "kept_idx is null");
  std::vector<uint64_t> ebeg(n + 1), ebytes(n);
  unsigned __int128 total = 0;
  bool uniform = true;
  for (int s = 0; s < n; ++s) {
    ebeg[s] = d[s].entry_begin;
    ebytes[s] = banks[s].entry_bytes;
    total += static_cast<unsigned __int128>(banks[s].n_entries) * banks[s].entry_bytes;
    uniform = uniform && banks[s].entry_bytes == banks[0].entry_bytes;
  }
  ebeg[n] = entries;
  if (total > static_cast<unsigned __int128>(~0ull))
    return fail(PCS_E_INVAL, "total entry bytes exceed 2^64");
  std::lock_guard<std::mutex> lk(c->mu);
  st = set_device(c);
  if (st) return st;
  if (pos_base + entries > 0xFFFFFFFFull)
    return fail(PCS_E_INVAL, "positions past 2^32 - 1 in the whole population");
  if (entries == 0 && !ex) {
    // Nothing to rank: every bank keeps nothing.
    PCS_CUDA(cudaMemsetAsync(kept_off, 0, 4ull * (n + 1), stream));
    return PCS_OK;
  }
  const uint64_t tiles = (entries + kGTile - 1) / kGTile;
  // Bank of entry min(t * kGTile, entries - 1), t = 0..tiles.
  std::vector<uint32_t> tile_bank(tiles + 1);
  {
    int b = 0;
    for (uint64_t t = 0; t <= tiles && entries > 0; ++t) {
      const uint64_t i = std::min<uint64_t>(t * kGTile, entries - 1);
      while (b + 1 < n && ebeg[b + 1] <= i) ++b;
      tile_bank[t] = static_cast<uint32_t>(b);
    }
  }
  GState g0{};
  g0.remaining = budget;
  // The budget does not bind: threshold 0 keeps all.  (A part cannot tell:
  // the first summed histogram shows it.)
  g0.done = !ex && total <= budget;
  uint64_t at = round_up(sizeof(BankDesc) * n, kRecordAlign);
  const uint64_t o_ebeg = at;
  at = round_up(at + 8ull * (n + 1), 16);
  const uint64_t o_ebytes = at;
  at = round_up(at + 8ull * n, 16);
  const uint64_t o_tb = at;
  at = round_up(at + 4ull * (tiles + 1), kRecordAlign);
  const uint64_t o_st = at;
  at = round_up(at + sizeof(GState), kRecordAlign);
  const uint64_t plan_bytes = at;
  const uint64_t o_tc = at;
  at = round_up(at + 4ull * tiles, kRecordAlign);
  const uint64_t o_ucand = at;
  at = round_up(at + 4ull * 8 * tiles, kRecordAlign);
  const uint64_t o_hb = at;
  at = round_up(at + sizeof(GBinSet) * kGPasses, kRecordAlign);
  const uint64_t o_ckey = at;
  at = round_up(at + 8ull * kGTile * tiles, kRecordAlign);
  const uint64_t o_cbank = at;
  if (!uniform) at = round_up(at + 4ull * kGTile * tiles, kRecordAlign);
  const uint64_t o_sc = at;
  const uint64_t ws_bytes = at + (scores ? 0 : 4ull * entries);
  uint8_t* ws = nullptr;
  st = ws_acquire(c, ws_bytes, stream, &ws);
  if (st) return st;
  c->plan.assign(plan_bytes, 0);
  put(c->plan, 0, d);
  put(c->plan, o_ebeg, ebeg);
  put(c->plan, o_ebytes, ebytes);
  put(c->plan, o_tb, tile_bank);
  std::memcpy(c->plan.data() + o_st, &g0, sizeof g0);
  PCS_CUDA(plan_copy(c, ws, plan_bytes, stream));
  float* sc = scores ? scores : reinterpret_cast<float*>(ws + o_sc);
  GHist gh{};
  if (!g0.done && !ex) {
    gh.st = reinterpret_cast<GState*>(ws + o_st);
    gh.uniform_bytes = n > 0 ? banks[0].entry_bytes : 0;
    gh.mode = uniform ? 1 : 2;
  }
  bool fused = false;
  PCS_CUDA(launch_bank_scores(c, banks, n, reinterpret_cast<const BankDesc*>(ws), entries, sc,
                              stream, gh, &fused));
  GPlan gp{};
  gp.scores = sc;
  gp.ebeg = reinterpret_cast<const uint64_t*>(ws + o_ebeg);
  gp.ebytes = reinterpret_cast<const uint64_t*>(ws + o_ebytes);
  gp.tile_bank = reinterpret_cast<const uint32_t*>(ws + o_tb);
  gp.tile_cnt = reinterpret_cast<uint32_t*>(ws + o_tc);
  gp.st = reinterpret_cast<GState*>(ws + o_st);
  gp.kept_idx = kept_idx;
  gp.kept_off = kept_off;
  gp.entries = entries;
  gp.uniform_bytes = n > 0 ? banks[0].entry_bytes : 0;
  gp.n_banks = n;
  gp.tiles = static_cast<int32_t>(tiles);
  gp.uniform = uniform ? 1 : 0;
  gp.pos_base = pos_base;
  gp.vec = aligned16(sc) ? 1 : 0;
  gp.ucand = reinterpret_cast<uint32_t*>(ws + o_ucand);
  gp.ckey = reinterpret_cast<uint64_t*>(ws + o_ckey);
  gp.cbank = uniform ? nullptr : reinterpret_cast<uint32_t*>(ws + o_cbank);
  gp.hb = reinterpret_cast<GBinSet*>(ws + o_hb);
  gp.err = c->words;
  if (ex) {
    // Every pass summed over the parts and picked on the host; the state
    // reaches k_gfinish done.
    gp.local = 1;
    st = exchange_passes(c, gp, budget, ex, user, stream);
    if (st) return st;
  }
  if (entries == 0) {
    PCS_CUDA(cudaMemsetAsync(kept_off, 0, 4ull * (n + 1), stream));
  } else {
    // The passes the score kernel did not take (at most six, none once the
    // threshold is known) and the compaction, in one launch.
    LaunchScope ls(c, kKGFinish, stream);
    PCS_CUDA(launch_gfinish(gp, fused ? 1 : 0, c->sm_count, stream));
  }
  return ws_release(c, stream);
}

pcs_status pcs_prune_global(pcs_ctx* c, const pcs_bank* banks, int32_t n, uint64_t budget,
                            float* scores, int32_t* kept_idx, int32_t* kept_off, void* stream) {
  PCS_TRACE("pcs_prune_global");
  return prune_global_impl(c, banks, n, budget, scores, kept_idx, kept_off, stream, nullptr,
                           nullptr, 0);
}

pcs_status pcs_prune_global_part(pcs_ctx* c, const pcs_bank* banks, int32_t n, uint64_t budget,
                                 uint64_t pos_base, pcs_hist_exchange_fn exchange, void* user,
                                 float* scores, int32_t* kept_idx, int32_t* kept_off,
                                 void* stream) {
  PCS_TRACE("pcs_prune_global_part");
  if (!exchange) return fail(PCS_E_INVAL, "exchange is null");
  return prune_global_impl(c, banks, n, budget, scores, kept_idx, kept_off, stream, exchange,
                           user, pos_base);
}

pcs_status pcs_budget_plan(const int32_t* n, const uint64_t* entry_bytes, const double* priority,
                           int32_t count, uint64_t budget, double fraction, int32_t* k_out,
                           int32_t* shrinks, int32_t* drops) {
  if (count < 0 || (count > 0 && (!n || !entry_bytes || !k_out)))
    return fail(PCS_E_INVAL, "bad arguments");
  if (!(fraction >= 0.0 && fraction <= 1.0)) return fail(PCS_E_INVAL, "fraction must lie in [0, 1]");
  int32_t n_shrink = 0, n_drop = 0;
  unsigned __int128 kept = 0;
  for (int s = 0; s < count; ++s) {
    if (n[s] < 0) return fail(PCS_E_INVAL, "session %d: negative n", s);
    k_out[s] = n[s];
    kept += static_cast<unsigned __int128>(static_cast<uint64_t>(n[s])) * entry_bytes[s];
  }
  if (kept > budget) {
    std::vector<int32_t> order(count);
    for (int s = 0; s < count; ++s) order[s] = s;
    std::stable_sort(order.begin(), order.end(), [&](int32_t a, int32_t b) {
      const double pa = priority ? priority[a] : a, pb = priority ? priority[b] : b;
      return pa < pb;
    });
    auto bytes_of = [&](int32_t s, int32_t rows) {
      return static_cast<unsigned __int128>(static_cast<uint64_t>(rows)) * entry_bytes[s];
    };
    for (int i = 0; i < count && kept > budget; ++i) {  // shrink
      const int32_t s = order[i];
      double v = __builtin_nearbyint(fraction * static_cast<double>(n[s]));
      v = std::min<double>(std::max(v, 0.0), n[s]);
      const int32_t target = static_cast<int32_t>(v);
      if (target < k_out[s]) {
        kept -= bytes_of(s, k_out[s] - target);
        k_out[s] = target;
        ++n_shrink;
      }
    }
    for (int i = 0; i < count && kept > budget; ++i) {  // nothing left to shrink: drop
      const int32_t s = order[i];
      if (k_out[s] > 0) {
        kept -= bytes_of(s, k_out[s]);
        k_out[s] = 0;
        ++n_drop;
      }
    }
  }
  if (shrinks) *shrinks = n_shrink;
  if (drops) *drops = n_drop;
  return PCS_OK;
}

pcs_status pcs_record_bytes(const pcs_section* sections, int32_t n, uint64_t* out) {
  if (!out || n < 1 || n > 65535 || !sections) return fail(PCS_E_INVAL, "bad section list");
  uint64_t off = round_up(kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * n, kRecordAlign);
  for (int i = 0; i < n; ++i) off = round_up(off + sections[i].bytes, kRecordAlign);
  *out = off;
  return PCS_OK;
}

pcs_status pcs_checkpoint(pcs_ctx* c, const pcs_session* sessions, int32_t n, uint32_t placement,
                          pcs_snapshot** out, void* stream_) {
  PCS_TRACE("pcs_checkpoint");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  if (n < 0 || (n > 0 && (!sessions || !out))) return fail(PCS_E_INVAL, "bad session list");
  if (n == 0) return PCS_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  Prepared pr;
  Block* blk = nullptr;
  std::vector<std::unique_ptr<pcs_snapshot>> handles;
  st = build_checkpoint(c, sessions, n, placement, stream, &pr, &blk, &handles, true);
  if (st) return st;
  auto undo = [&](pcs_status s) {
    arena_of(c, placement)->free(blk);
    return s;
  };
  uint8_t* ws = nullptr;
  st = ws_acquire(c, pr.L.total, stream, &ws);
  if (st) return undo(st);
  cudaError_t e = plan_send(c, ws, pr.L.nodes, pr.plan, stream);
  if (e == cudaSuccess) e = launch_prepared(c, pr, ws, c->call_words, stream);
  if (e != cudaSuccess) return undo(cuda_fail(e, "checkpoint launch"));
  blk->written = record_event(c->events, stream);
  st = ws_release(c, stream, blk->written);
  if (st) return undo(st);
  blk->refs = n;
  c->live.reserve(n);
  for (int s = 0; s < n; ++s) {
    out[s] = handles[s].release();
    c->live.insert(out[s]);
  }
  return PCS_OK;
}

pcs_status pcs_fork_many(pcs_ctx* c, pcs_snapshot* const* parents, int32_t n,
                         pcs_snapshot** children, void* stream_) {
  PCS_TRACE("pcs_fork_many");
  if (!c || n < 0 || (n > 0 && (!parents || !children))) return fail(PCS_E_INVAL, "bad arguments");
  if (n == 0) return PCS_OK;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::lock_guard<std::mutex> lk(c->mu);
  for (int i = 0; i < n; ++i)
    if (!check_handle(c, parents[i])) return fail(PCS_E_HANDLE, "snapshot %d: unknown handle", i);
  pcs_status st = set_device(c);
  if (st) return st;
  // One new block per placement holds the children of that placement.
  uint64_t need[2] = {0, 0};
  std::vector<uint64_t> off(n);
  for (int i = 0; i < n; ++i) {
    const uint32_t pl = parents[i]->block->placement;
    off[i] = need[pl];
    need[pl] += parents[i]->total_bytes;
  }
  Block* blk[2] = {nullptr, nullptr};
  auto undo = [&](pcs_status s) {
    for (int pl = 0; pl < 2; ++pl)
      if (blk[pl]) arena_of(c, pl)->free(blk[pl]);
    return s;
  };
  for (uint32_t pl = 0; pl < 2; ++pl) {
    if (!need[pl]) continue;
    st = arena_of(c, pl)->alloc(need[pl], stream, &blk[pl]);
    if (st) return undo(st);
  }
  // Snapshots of one call share a block: one wait (one event query) per run
  // of equal blocks, not per snapshot.
  for (int i = 0; i < n; ++i) {
    if (i > 0 && parents[i]->block == parents[i - 1]->block) continue;
    st = wait_written(parents[i]->block, stream);
    if (st) return undo(st);
  }
  // A fork is a restore of the whole record into a contiguous target: the
  // streaming kernels copy it (no hashing), TMA-staged when both are in HBM.
  std::vector<SecDesc> d(n);
  std::vector<char> bulk(n);
  PtrCache cache;
  uint64_t bytes = 0;
  for (int i = 0; i < n; ++i) {
    pcs_section x{};
    x.layout = PCS_LAYOUT_CONTIG;
    x.base = blk[parents[i]->block->placement]->ptr + off[i];
    x.bytes = parents[i]->total_bytes;
    d[i] = make_desc(x, parents[i]->record(), 0);
    bytes += x.bytes;
  }
  const bool small = bytes <= kSmallCallBytes;
  for (int i = 0; i < n; ++i)
    bulk[i] = c->use_bulk && !small && parents[i]->block->placement == PCS_PLACE_DEVICE;
  StreamPlan P;
  if (!plan_streams(c, d, bulk, P)) return undo(fail(PCS_E_INVAL, "too much data in one call"));
  if (c->check_plans) {
    const std::string e = check_streams(d, bulk, P);
    if (!e.empty()) return undo(fail(PCS_E_INVAL, "plan check: %s", e.c_str()));
  }
  const ListLayout LL = list_layout(P, sizeof(SecDesc) * n);
  const uint64_t total = round_up(LL.end, kRecordAlign);
  uint8_t* ws = nullptr;
  st = ws_acquire(c, total, stream, &ws);
  if (st) return undo(st);
  c->plan.resize(total);
  put(c->plan, 0, d);
  put_lists(c->plan, P, LL);
  cudaError_t e = plan_copy(c, ws, total, stream);
  if (e == cudaSuccess)
    e = launch_streams(c, kModeRestore, reinterpret_cast<const SecDesc*>(ws), P, LL, ws, nullptr,
                       stream);
  if (e != cudaSuccess) return undo(cuda_fail(e, "fork copy"));
  Ev done = record_event(c->events, stream);
  st = ws_release(c, stream, done);
  if (st) return undo(st);
  for (int i = 0; i < n; ++i)
    if (i == 0 || parents[i]->block != parents[i - 1]->block) note_use(c, parents[i]->block, stream);
  for (int pl = 0; pl < 2; ++pl) {
    if (!blk[pl]) continue;
    blk[pl]->written = done;
    blk[pl]->refs = 0;
  }
  c->live.reserve(n);
  for (int i = 0; i < n; ++i) {
    Block* b = blk[parents[i]->block->placement];
    auto h = new_snapshot(c);
    *h = *parents[i];
    h->block = b;
    h->offset = off[i];
    b->refs += 1;
    children[i] = h.release();
    c->live.insert(children[i]);
  }
  return PCS_OK;
}

pcs_status pcs_fork(pcs_ctx* c, const pcs_snapshot* parent, pcs_snapshot** child, void* stream) {
  if (!c || !child) return fail(PCS_E_INVAL, "null argument");
  pcs_snapshot* p = const_cast<pcs_snapshot*>(parent);
  return pcs_fork_many(c, &p, 1, child, stream);
}

pcs_status pcs_restore(pcs_ctx* c, pcs_snapshot* const* snaps, int32_t n, const pcs_session* targets,
                       int32_t verify, void* stream_) {
  PCS_TRACE("pcs_restore");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  if (n < 0 || (n > 0 && (!snaps || !targets))) return fail(PCS_E_INVAL, "bad arguments");
  if (verify < 0 || verify > 2) return fail(PCS_E_INVAL, "verify must be 0, 1 or 2");
  if (n == 0) return PCS_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  Prepared pr;
  st = build_restore(c, snaps, n, targets, verify, &pr, true);
  if (st) return st;
  for (int s = 0; s < n; ++s) {
    if (s > 0 && snaps[s]->block == snaps[s - 1]->block) continue;  // one wait per run of a block
    st = wait_written(snaps[s]->block, stream);
    if (st) return st;
  }
  uint8_t* ws = nullptr;
  st = ws_acquire(c, pr.L.total, stream, &ws);
  if (st) return st;
  PCS_CUDA(plan_send(c, ws, pr.L.nodes, pr.plan, stream));
  // verify == 1: count failures of this call in words[1] and wait for them;
  // verify == 2: accumulate them in words[2] for the next pcs_sync.
  uint32_t* words = c->call_words;
  if (verify == 1) PCS_CUDA(cudaMemsetAsync(words + 1, 0, 4, stream));
  PCS_CUDA(launch_prepared(c, pr, ws, words, stream));
  for (int s = 0; s < n; ++s) {
    if (s > 0 && snaps[s]->block == snaps[s - 1]->block) continue;
    st = note_use(c, snaps[s]->block, stream);
    if (st) return st;
  }
  st = ws_release(c, stream);
  if (st) return st;
  if (verify == 1) {
    uint32_t bad = 0;
    PCS_CUDA(cudaMemcpyAsync(&bad, words + 1, 4, cudaMemcpyDeviceToHost, stream));
    PCS_CUDA(cudaStreamSynchronize(stream));
    if (bad) return fail(PCS_E_CORRUPT, "%u of %d restored sessions failed verification", bad, n);
  }
  return PCS_OK;
}

// ---- Prepared calls ---------------------------------------------------------

pcs_status pcs_plan_checkpoint(pcs_ctx* c, const pcs_session* sessions, int32_t n,
                               uint32_t placement, pcs_snapshot** out, pcs_plan** plan,
                               void* stream_) {
  PCS_TRACE("pcs_plan_checkpoint");
  if (!c || !plan) return fail(PCS_E_INVAL, "bad arguments");
  *plan = nullptr;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  if (n <= 0 || !sessions || !out) return fail(PCS_E_INVAL, "bad session list");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  auto p = std::make_unique<pcs_plan>();
  Block* blk = nullptr;
  std::vector<std::unique_ptr<pcs_snapshot>> handles;
  st = build_checkpoint(c, sessions, n, placement, stream, &p->pr, &blk, &handles);
  if (st) return st;
  st = plan_upload(p.get());
  cudaError_t e = st ? cudaSuccess : launch_prepared(c, p->pr, plan_ws(p.get()), plan_words(p.get()), stream);
  if (st || e != cudaSuccess) {
    if (p->dev) cudaFree(p->dev);
    arena_of(c, placement)->free(blk);
    return st ? st : cuda_fail(e, "checkpoint launch");
  }
  blk->written = record_event(c->events, stream);
  blk->refs = n + 1;  // the snapshots and the plan
  p->blocks.push_back(blk);
  c->live.reserve(n);
  for (int s = 0; s < n; ++s) {
    out[s] = handles[s].release();
    c->live.insert(out[s]);
  }
  *plan = p.release();
  c->plans.insert(*plan);
  return PCS_OK;
}

pcs_status pcs_plan_restore(pcs_ctx* c, pcs_snapshot* const* snaps, int32_t n,
                            const pcs_session* targets, int32_t verify, pcs_plan** plan) {
  PCS_TRACE("pcs_plan_restore");
  if (!c || !plan) return fail(PCS_E_INVAL, "bad arguments");
  *plan = nullptr;
  if (n <= 0 || !snaps || !targets) return fail(PCS_E_INVAL, "bad arguments");
  if (verify != 0 && verify != 2)
    return fail(PCS_E_INVAL, "a prepared restore verifies with 0 or 2 (reported at pcs_sync)");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  auto p = std::make_unique<pcs_plan>();
  st = build_restore(c, snaps, n, targets, verify, &p->pr);
  if (st) return st;
  st = plan_upload(p.get());
  if (st) {
    if (p->dev) cudaFree(p->dev);
    return st;
  }
  for (int s = 0; s < n; ++s) {
    Block* b = snaps[s]->block;
    if (std::find(p->blocks.begin(), p->blocks.end(), b) == p->blocks.end()) {
      ++b->refs;
      p->blocks.push_back(b);
    }
  }
  *plan = p.release();
  c->plans.insert(*plan);
  return PCS_OK;
}

pcs_status pcs_plan_run(pcs_ctx* c, pcs_plan* p, void* stream_) {
  PCS_TRACE("pcs_plan_run");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::lock_guard<std::mutex> lk(c->mu);
  if (!p || !c->plans.count(p)) return fail(PCS_E_HANDLE, "not a live plan of this context");
  pcs_status st = set_device(c);
  if (st) return st;
  const bool ckpt = p->pr.mode == kModePack;
  for (Block* b : p->blocks) {
    if (!ckpt) {
      st = wait_written(b, stream);  // the records' latest checkpoint
      if (st) return st;
      continue;
    }
    // Rewriting records: after every queued reader of them, on any stream.
    for (auto& u : b->uses)
      if (u.first != stream && u.second && !u.second->done())
        PCS_CUDA(cudaStreamWaitEvent(stream, u.second->ev, 0));
  }
  PCS_CUDA(launch_prepared(c, p->pr, plan_ws(p), plan_words(p), stream));
  for (Block* b : p->blocks) {
    if (ckpt) {
      b->written = record_event(c->events, stream);
      if (!b->written) return fail(PCS_E_CUDA, "cudaEventRecord failed");
    } else {
      st = note_use(c, b, stream);
      if (st) return st;
    }
  }
  return PCS_OK;
}

pcs_status pcs_plan_destroy(pcs_ctx* c, pcs_plan* p) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (!p) return PCS_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  if (!c->plans.count(p)) return fail(PCS_E_HANDLE, "not a live plan of this context");
  pcs_status st = set_device(c);
  if (st) return st;
  c->plans.erase(p);
  destroy_plan(c, p);
  return PCS_OK;
}

pcs_status pcs_delete(pcs_ctx* c, pcs_snapshot* h) {
  PCS_TRACE("pcs_delete");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  if (!check_handle(c, h)) return fail(PCS_E_HANDLE, "unknown snapshot handle");
  c->live.erase(h);
  release_block(c, h->block);
  drop_snapshot(c, h);
  return PCS_OK;
}

pcs_status pcs_delete_many(pcs_ctx* c, pcs_snapshot* const* snaps, int32_t n) {
  PCS_TRACE("pcs_delete_many");
  if (!c || n < 0 || (n > 0 && !snaps)) return fail(PCS_E_INVAL, "bad arguments");
  std::lock_guard<std::mutex> lk(c->mu);
  for (int i = 0; i < n; ++i)
    if (!check_handle(c, snaps[i])) return fail(PCS_E_HANDLE, "snapshot %d: unknown handle", i);
  for (int i = 0; i < n; ++i) {
    pcs_snapshot* h = snaps[i];
    if (!c->live.erase(h)) return fail(PCS_E_HANDLE, "snapshot %d: listed twice", i);
    release_block(c, h->block);
    drop_snapshot(c, h);
  }
  return PCS_OK;
}

static pcs_status read_record(pcs_ctx* c, pcs_snapshot* h, uint64_t off, uint64_t bytes, void* dst) {
  if (h->block->written) PCS_CUDA(cudaEventSynchronize(h->block->written->ev));
  PCS_CUDA(cudaMemcpy(dst, h->record() + off, bytes, cudaMemcpyDefault));
  (void)c;
  return PCS_OK;
}

pcs_status pcs_snapshot_get_info(pcs_ctx* c, const pcs_snapshot* snap, pcs_snapshot_info* out) {
  if (!c || !out) return fail(PCS_E_INVAL, "null argument");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_snapshot* h = check_handle(c, snap);
  if (!h) return fail(PCS_E_HANDLE, "unknown snapshot handle");
  pcs_status st = set_device(c);
  if (st) return st;
  uint8_t hdr[64];
  st = read_record(c, h, 0, 64, hdr);
  if (st) return st;
  out->session_id = h->session_id;
  out->kind = h->kind;
  out->n_sections = static_cast<int32_t>(h->n_sections);
  out->placement = h->block->placement;
  out->total_bytes = h->total_bytes;
  std::memcpy(&out->session_fp, hdr + 24, 8);
  out->data = h->record();
  return PCS_OK;
}

pcs_status pcs_snapshot_get_section(pcs_ctx* c, const pcs_snapshot* snap, int32_t i,
                                pcs_section_info* out) {
  if (!c || !out) return fail(PCS_E_INVAL, "null argument");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_snapshot* h = check_handle(c, snap);
  if (!h) return fail(PCS_E_HANDLE, "unknown snapshot handle");
  if (i < 0 || i >= static_cast<int32_t>(h->n_sections))
    return fail(PCS_E_INVAL, "section %d out of range", i);
  pcs_status st = set_device(c);
  if (st) return st;
  Entry e;
  st = read_record(c, h, kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * i, sizeof e, &e);
  if (st) return st;
  out->type = e.type;
  out->dtype = e.dtype;
  out->layer = e.layer;
  out->layout = e.layout;
  out->offset = e.offset;
  out->bytes = e.bytes;
  out->fp = e.fp;
  out->dim0 = e.dim0;
  out->dim1 = e.dim1;
  out->aux = e.aux;
  return PCS_OK;
}

pcs_status pcs_snapshot_copy_out(pcs_ctx* c, const pcs_snapshot* snap, uint64_t offset,
                                 uint64_t bytes, void* dst, void* stream_) {
  PCS_TRACE("pcs_snapshot_copy_out");
  if (!c || (bytes > 0 && !dst)) return fail(PCS_E_INVAL, "null argument");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_snapshot* h = check_handle(c, snap);
  if (!h) return fail(PCS_E_HANDLE, "unknown snapshot handle");
  if (offset > h->total_bytes || bytes > h->total_bytes - offset)
    return fail(PCS_E_INVAL, "range outside the record");
  pcs_status st = set_device(c);
  if (st) return st;
  if (bytes == 0) return PCS_OK;
  st = wait_written(h->block, stream);
  if (st) return st;
  PCS_CUDA(cudaMemcpyAsync(dst, h->record() + offset, bytes, cudaMemcpyDefault, stream));
  return note_use(c, h->block, stream);
}

static pcs_status ensure_stage(pcs_ctx* c) {
  if (c->stage) return PCS_OK;
  if (cudaHostAlloc(&c->stage, kStageBytes, cudaHostAllocDefault) != cudaSuccess) {
    cudaGetLastError();
    c->stage = nullptr;
    return fail(PCS_E_NOMEM, "cannot allocate the pinned staging buffer");
  }
  c->stage_bytes = kStageBytes;
  return PCS_OK;
}

pcs_status pcs_snapshot_write_file(pcs_ctx* c, const pcs_snapshot* snap, const char* path) {
  PCS_TRACE("pcs_snapshot_write_file");
  if (!c || !path) return fail(PCS_E_INVAL, "null argument");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_snapshot* h = check_handle(c, snap);
  if (!h) return fail(PCS_E_HANDLE, "unknown snapshot handle");
  pcs_status st = set_device(c);
  if (st) return st;
  if (h->block->written) PCS_CUDA(cudaEventSynchronize(h->block->written->ev));
  st = ensure_stage(c);
  if (st) return st;
  std::string tmp = std::string(path) + ".tmp";
  FILE* f = std::fopen(tmp.c_str(), "wb");
  if (!f) return fail(PCS_E_IO, "cannot open %s: %s", tmp.c_str(), std::strerror(errno));
  for (uint64_t off = 0; off < h->total_bytes; off += c->stage_bytes) {
    const uint64_t nb = std::min(c->stage_bytes, h->total_bytes - off);
    cudaError_t e = cudaMemcpy(c->stage, h->record() + off, nb, cudaMemcpyDefault);
    if (e != cudaSuccess || std::fwrite(c->stage, 1, nb, f) != nb) {
      std::fclose(f);
      std::remove(tmp.c_str());
      if (e != cudaSuccess) return cuda_fail(e, "snapshot read-back");
      return fail(PCS_E_IO, "write to %s failed", tmp.c_str());
    }
  }
  if (std::fflush(f) != 0 || fsync(fileno(f)) != 0) {
    std::fclose(f);
    std::remove(tmp.c_str());
    return fail(PCS_E_IO, "flush of %s failed", tmp.c_str());
  }
  std::fclose(f);
  if (std::rename(tmp.c_str(), path) != 0) {
    std::remove(tmp.c_str());
    return fail(PCS_E_IO, "rename to %s failed: %s", path, std::strerror(errno));
  }
  return PCS_OK;
}

pcs_status pcs_snapshot_read_file(pcs_ctx* c, const char* path, uint32_t placement,
                                  pcs_snapshot** out) {
  PCS_TRACE("pcs_snapshot_read_file");
  if (!c || !path || !out) return fail(PCS_E_INVAL, "null argument");
  if (placement != PCS_PLACE_DEVICE && placement != PCS_PLACE_PINNED_HOST)
    return fail(PCS_E_INVAL, "unknown placement %u", placement);
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  FILE* f = std::fopen(path, "rb");
  if (!f) return fail(PCS_E_IO, "cannot open %s: %s", path, std::strerror(errno));
  auto close_fail = [&](pcs_status s) {
    std::fclose(f);
    return s;
  };
  if (std::fseek(f, 0, SEEK_END) != 0) return close_fail(fail(PCS_E_IO, "seek failed"));
  const long fsize = std::ftell(f);
  std::rewind(f);
  uint8_t hdr[64];
  if (fsize < 64 || std::fread(hdr, 1, 64, f) != 64)
    return close_fail(fail(PCS_E_CORRUPT, "%s: too short for a record header", path));
  uint32_t magic, vn, sid, kind;
  uint64_t total;
  std::memcpy(&magic, hdr, 4);
  std::memcpy(&vn, hdr + 4, 4);
  std::memcpy(&sid, hdr + 8, 4);
  std::memcpy(&kind, hdr + 12, 4);
  std::memcpy(&total, hdr + 16, 8);
  const uint32_t nsec = vn >> 16;
  if (magic != kMagic || (vn & 0xFFFFu) != kVersion)
    return close_fail(fail(PCS_E_CORRUPT, "%s: not a PCS1 record", path));
  const uint64_t pstart = round_up(kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * nsec, kRecordAlign);
  if (nsec < 1 || total != static_cast<uint64_t>(fsize) || total % kRecordAlign != 0 || pstart > total)
    return close_fail(fail(PCS_E_CORRUPT, "%s: header sizes do not match the file", path));
  std::vector<Entry> table(nsec);
  if (std::fread(table.data(), sizeof(Entry), nsec, f) != nsec)
    return close_fail(fail(PCS_E_CORRUPT, "%s: truncated section table", path));
  uint64_t expect = pstart;
  for (uint32_t i = 0; i < nsec; ++i) {
    const Entry& e = table[i];
    if (e.offset != expect || e.bytes > total - e.offset || e.layout > PCS_LAYOUT_RING)
      return close_fail(fail(PCS_E_CORRUPT, "%s: section %u has an impossible offset or size", path, i));
    expect = round_up(e.offset + e.bytes, kRecordAlign);
  }
  if (expect != total) return close_fail(fail(PCS_E_CORRUPT, "%s: record size mismatch", path));
  Block* blk = nullptr;
  st = arena_of(c, placement)->alloc(total, nullptr, &blk);
  if (st) return close_fail(st);
  // Anything that reused this range must be done before the host writes it.
  PCS_CUDA(cudaDeviceSynchronize());
  std::rewind(f);
  if (placement == PCS_PLACE_PINNED_HOST) {
    if (std::fread(blk->ptr, 1, total, f) != total) {
      arena_of(c, placement)->free(blk);
      return close_fail(fail(PCS_E_IO, "%s: read failed", path));
    }
  } else {
    st = ensure_stage(c);
    if (st) {
      arena_of(c, placement)->free(blk);
      return close_fail(st);
    }
    for (uint64_t off = 0; off < total; off += c->stage_bytes) {
      const uint64_t nb = std::min(c->stage_bytes, total - off);
      if (std::fread(c->stage, 1, nb, f) != nb ||
          cudaMemcpy(blk->ptr + off, c->stage, nb, cudaMemcpyHostToDevice) != cudaSuccess) {
        arena_of(c, placement)->free(blk);
        return close_fail(fail(PCS_E_IO, "%s: read failed", path));
      }
    }
  }
  std::fclose(f);
  blk->refs = 1;
  auto h = new_snapshot(c);
  h->block = blk;
  h->offset = 0;
  h->total_bytes = total;
  h->payload_start = pstart;
  h->session_id = sid;
  h->kind = kind;
  for (auto& e : table) e.fp = 0;
  h->n_sections = static_cast<uint32_t>(table.size());
  h->tables = std::make_shared<const std::vector<Entry>>(std::move(table));
  *out = h.release();
  c->live.insert(*out);
  return PCS_OK;
}

// ---- Copy-on-write page pool -------------------------------------------------

pcs_status pcs_pool_create(pcs_ctx* c, void* base, uint64_t page_bytes, int32_t n_pages,
                           pcs_pool** out) {
  if (!c || !out) return fail(PCS_E_INVAL, "bad arguments");
  *out = nullptr;
  if (n_pages <= 0) return fail(PCS_E_INVAL, "n_pages must be positive");
  if (!base) return fail(PCS_E_INVAL, "base is null");
  if (page_bytes == 0 || page_bytes % 16 != 0 || !aligned16(base))
    return fail(PCS_E_ALIGN, "page_bytes and base must be non-zero multiples of 16");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  auto pl = std::make_unique<pcs_pool>();
  const uint64_t n = static_cast<uint64_t>(n_pages);
  const uint64_t bytes = 8 * n + 256;
  PCS_CUDA(cudaMalloc(&pl->meta, bytes));
  auto* m = static_cast<uint8_t*>(pl->meta);
  pl->d.base = static_cast<uint8_t*>(base);
  pl->d.rc = reinterpret_cast<uint32_t*>(m);
  pl->d.free_ids = reinterpret_cast<int32_t*>(m + 4 * n);
  pl->d.top = reinterpret_cast<int32_t*>(m + 8 * n);
  pl->d.err = c->words;
  pl->d.page_bytes = page_bytes;
  pl->d.n_pages = n_pages;
  // All pages free; the stack hands out the lowest ids first.
  std::vector<int32_t> init(n + 1);
  for (uint64_t i = 0; i < n; ++i) init[i] = static_cast<int32_t>(n - 1 - i);
  init[n] = n_pages;
  cudaError_t e = cudaMemset(pl->d.rc, 0, 4 * n);
  if (e == cudaSuccess) e = cudaMemcpy(pl->d.free_ids, init.data(), 4 * (n + 1), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    cudaFree(pl->meta);
    return cuda_fail(e, "pcs_pool_create");
  }
  *out = pl.release();
  c->pools.insert(*out);
  return PCS_OK;
}

pcs_status pcs_pool_destroy(pcs_ctx* c, pcs_pool* pl) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (!pl) return PCS_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  if (!c->pools.count(pl)) return fail(PCS_E_HANDLE, "not a live pool of this context");
  pcs_status st = set_device(c);
  if (st) return st;
  c->pools.erase(pl);
  PCS_CUDA(cudaDeviceSynchronize());
  cudaFree(pl->meta);
  delete pl;
  return PCS_OK;
}

namespace {

pcs_status pool_check(pcs_ctx* c, pcs_pool* pl) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  if (!pl || !c->pools.count(pl)) return fail(PCS_E_HANDLE, "not a live pool of this context");
  return set_device(c);
}

}  // namespace

pcs_status pcs_pool_alloc(pcs_ctx* c, pcs_pool* pl, int32_t* ids, int32_t n, void* stream) {
  PCS_TRACE("pcs_pool_alloc");
  if (n < 0 || (n > 0 && !ids)) return fail(PCS_E_INVAL, "bad arguments");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = pool_check(c, pl);
  if (st) return st;
  if (n == 0) return PCS_OK;
  LaunchScope ls(c, kKPoolAlloc, static_cast<cudaStream_t>(stream));
  PCS_CUDA(launch_pool_alloc(pl->d, ids, n, static_cast<cudaStream_t>(stream)));
  return PCS_OK;
}

pcs_status pcs_pool_share(pcs_ctx* c, pcs_pool* pl, const int32_t* src, int32_t* dst, int32_t n,
                          void* stream) {
  PCS_TRACE("pcs_pool_share");
  if (n < 0 || (n > 0 && !src)) return fail(PCS_E_INVAL, "bad arguments");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = pool_check(c, pl);
  if (st) return st;
  if (n == 0) return PCS_OK;
  LaunchScope ls(c, kKPoolShare, static_cast<cudaStream_t>(stream));
  PCS_CUDA(launch_pool_share(pl->d, src, dst, n, static_cast<cudaStream_t>(stream)));
  return PCS_OK;
}

pcs_status pcs_pool_prepare_write(pcs_ctx* c, pcs_pool* pl, int32_t* table, int64_t n_table,
                                  const int32_t* entries, int32_t n, void* stream) {
  PCS_TRACE("pcs_pool_prepare_write");
  if (n < 0 || n_table < 0 || (n > 0 && !table)) return fail(PCS_E_INVAL, "bad arguments");
  if (!entries && n > n_table) return fail(PCS_E_INVAL, "n exceeds the table");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = pool_check(c, pl);
  if (st) return st;
  if (n == 0) return PCS_OK;
  LaunchScope ls(c, kKPoolCow, static_cast<cudaStream_t>(stream));
  PCS_CUDA(launch_pool_cow(pl->d, table, n_table, entries, n, c->sm_count,
                           static_cast<cudaStream_t>(stream)));
  return PCS_OK;
}

pcs_status pcs_pool_release(pcs_ctx* c, pcs_pool* pl, const int32_t* ids, int32_t n, void* stream) {
  PCS_TRACE("pcs_pool_release");
  if (n < 0 || (n > 0 && !ids)) return fail(PCS_E_INVAL, "bad arguments");
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = pool_check(c, pl);
  if (st) return st;
  if (n == 0) return PCS_OK;
  LaunchScope ls(c, kKPoolRelease, static_cast<cudaStream_t>(stream));
  PCS_CUDA(launch_pool_release(pl->d, ids, n, static_cast<cudaStream_t>(stream)));
  return PCS_OK;
}

pcs_status pcs_pool_query(pcs_ctx* c, pcs_pool* pl, int32_t* free_pages, uint32_t* counts,
                          int32_t* free_ids, void* stream) {
  if (!c) return fail(PCS_E_INVAL, "ctx is null");
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = pool_check(c, pl);
  if (st) return st;
  PCS_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int32_t top = 0;
  PCS_CUDA(cudaMemcpy(&top, pl->d.top, 4, cudaMemcpyDeviceToHost));
  if (free_pages) *free_pages = top;
  const uint64_t n = static_cast<uint64_t>(pl->d.n_pages);
  if (counts) PCS_CUDA(cudaMemcpy(counts, pl->d.rc, 4 * n, cudaMemcpyDeviceToHost));
  if (free_ids && top > 0)
    PCS_CUDA(cudaMemcpy(free_ids, pl->d.free_ids, 4ull * std::min<uint64_t>(top, n),
                        cudaMemcpyDeviceToHost));
  return PCS_OK;
}

// ---- Discovery: distance, reads, procedure -----------------------------------

pcs_status pcs_mismatch(pcs_ctx* c, const pcs_buf* a, const pcs_buf* b, int32_t n,
                        uint64_t* counts, void* stream_) {
  PCS_TRACE("pcs_mismatch");
  if (!c || n < 0 || (n > 0 && (!a || !b || !counts))) return fail(PCS_E_INVAL, "bad arguments");
  if (n == 0) return PCS_OK;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::vector<MmPair> pairs(n);
  std::vector<uint64_t> tb(n + 1), extra(n);
  uint64_t tiles = 0;
  for (int i = 0; i < n; ++i) {
    const uint64_t m = std::min(a[i].bytes, b[i].bytes);
    if (m > 0 && (!a[i].ptr || !b[i].ptr)) return fail(PCS_E_INVAL, "pair %d: null buffer", i);
    pairs[i].a = static_cast<const uint8_t*>(a[i].ptr);
    pairs[i].b = static_cast<const uint8_t*>(b[i].ptr);
    pairs[i].bytes = m;
    pairs[i].vec = aligned16(a[i].ptr) && aligned16(b[i].ptr);
    extra[i] = std::max(a[i].bytes, b[i].bytes) - m;
    tb[i] = tiles;
    tiles += (m + kMmUnit - 1) / kMmUnit;
  }
  tb[n] = tiles;
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  const uint64_t o_tb = round_up(sizeof(MmPair) * n, kRecordAlign);
  const uint64_t o_ex = round_up(o_tb + 8ull * (n + 1), kRecordAlign);
  const uint64_t total = o_ex + 8ull * n;
  uint8_t* ws = nullptr;
  st = ws_acquire(c, total, stream, &ws);
  if (st) return st;
  c->plan.assign(total, 0);
  put(c->plan, 0, pairs);
  put(c->plan, o_tb, tb);
  put(c->plan, o_ex, extra);
  PCS_CUDA(plan_copy(c, ws, total, stream));
  // Counts start at the bytes only one buffer has.
  PCS_CUDA(cudaMemcpyAsync(counts, ws + o_ex, 8ull * n, cudaMemcpyDeviceToDevice, stream));
  {
    LaunchScope ls(c, kKMismatch, stream);
    PCS_CUDA(launch_mismatch(reinterpret_cast<const MmPair*>(ws),
                             reinterpret_cast<const uint64_t*>(ws + o_tb), n, tiles, counts,
                             c->sm_count, stream));
  }
  return ws_release(c, stream);
}

pcs_status pcs_classify_reads(pcs_ctx* c, const pcs_buf* bufs, int32_t n, const uint64_t* addr,
                              const uint64_t* bytes, int64_t m, uint8_t* flags, void* stream_) {
  PCS_TRACE("pcs_classify_reads");
  if (!c || n < 0 || m < 0 || (n > 0 && (!bufs || !flags)) || (m > 0 && (!addr || !bytes)))
    return fail(PCS_E_INVAL, "bad arguments");
  if (n == 0) return PCS_OK;
  if (n > 0x7FFFFFFF - 1) return fail(PCS_E_INVAL, "too many buffers");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  std::vector<uint32_t> ord(n);
  for (int i = 0; i < n; ++i) ord[i] = static_cast<uint32_t>(i);
  auto start_of = [&](uint32_t i) { return reinterpret_cast<uint64_t>(bufs[i].ptr); };
  std::stable_sort(ord.begin(), ord.end(),
                   [&](uint32_t x, uint32_t y) { return start_of(x) < start_of(y); });
  std::vector<uint64_t> st_(n), en(n), mx(n);
  uint64_t run = 0;
  for (int k = 0; k < n; ++k) {
    const uint64_t b0 = start_of(ord[k]);
    const uint64_t len = bufs[ord[k]].bytes;
    st_[k] = b0;
    en[k] = b0 + len < b0 ? ~0ull : b0 + len;
    run = std::max(run, en[k]);
    mx[k] = run;
  }
  std::lock_guard<std::mutex> lk(c->mu);
  pcs_status st = set_device(c);
  if (st) return st;
  const uint64_t o_en = round_up(8ull * n, 256), o_mx = round_up(o_en + 8ull * n, 256);
  const uint64_t o_or = round_up(o_mx + 8ull * n, 256), total = o_or + 4ull * n;
  uint8_t* ws = nullptr;
  st = ws_acquire(c, total, stream, &ws);
  if (st) return st;
  c->plan.assign(total, 0);
  put(c->plan, 0, st_);
  put(c->plan, o_en, en);
  put(c->plan, o_mx, mx);
  put(c->plan, o_or, ord);
  PCS_CUDA(plan_copy(c, ws, total, stream));
  PCS_CUDA(cudaMemsetAsync(flags, 0, n, stream));
  ReadPlan rp{};
  rp.start = reinterpret_cast<const uint64_t*>(ws);
  rp.end = reinterpret_cast<const uint64_t*>(ws + o_en);
  rp.maxend = reinterpret_cast<const uint64_t*>(ws + o_mx);
  rp.orig = reinterpret_cast<const uint32_t*>(ws + o_or);
  rp.n = n;
  if (m > 0) {
    LaunchScope ls(c, kKClassifyReads, stream);
    PCS_CUDA(launch_classify_reads(rp, addr, bytes, m, flags, c->sm_count, stream));
  }
  return ws_release(c, stream);
}

pcs_status pcs_discover(int32_t k, pcs_probe_fn probe, void* user, uint64_t eps,
                        uint8_t* pcs_out, int32_t* probes_out, int32_t* consistent) {
  if (k < 0 || !probe || (k > 0 && !pcs_out)) return fail(PCS_E_INVAL, "bad arguments");
  int32_t probes = 0;
  std::vector<uint8_t> keep(std::max(k, 1));
  auto run = [&](const std::vector<uint8_t>& mask, uint64_t* d) -> pcs_status {
    ++probes;
    const int32_t rc = probe(user, mask.data(), d);
    if (rc != 0) return fail(PCS_E_INVAL, "probe %d returned %d", probes, rc);
    return PCS_OK;
  };
  // 1. necessity: leave one out.
  std::vector<uint8_t> chosen(std::max(k, 1), 0);
  for (int i = 0; i < k; ++i) {
    for (int j = 0; j < k; ++j) keep[j] = j != i;
    uint64_t d = 0;
    pcs_status st = run(keep, &d);
    if (st) return st;
    chosen[i] = d > eps;
  }
  // 2. sufficiency of the necessary set.
  uint64_t d = 0;
  pcs_status st = run(chosen, &d);
  if (st) return st;
  // 3. redundancy fallback: add the component that most reduces D.
  while (d > eps) {
    int best = -1;
    uint64_t best_d = 0;
    for (int j = 0; j < k; ++j) {
      if (chosen[j]) continue;
      keep = chosen;
      keep[j] = 1;
      uint64_t dj = 0;
      st = run(keep, &dj);
      if (st) return st;
      if (best < 0 || dj < best_d) {
        best = j;
        best_d = dj;
      }
    }
    if (best < 0) break;  // everything is in and D still exceeds eps
    chosen[best] = 1;
    d = best_d;
  }
  for (int i = 0; i < k; ++i) pcs_out[i] = chosen[i];
  if (probes_out) *probes_out = probes;
  if (consistent) *consistent = d <= eps;
  return PCS_OK;
}

pcs_status pcs_fingerprint_static(const pcs_buf* bufs, int32_t n, uint64_t* fp_out,
                                  void* stream) {
  static_assert(kStaticMaxBufs == PCS_STATIC_MAX_BUFFERS, "limit");
  static_assert(kStaticMaxNodes == PCS_STATIC_MAX_NODES, "limit");
  if (n < 0 || n > kStaticMaxBufs)
    return fail(PCS_E_INVAL, "pcs_fingerprint_static takes 0..%d buffers, got %d", kStaticMaxBufs, n);
  if (n == 0) return PCS_OK;
  if (!bufs || !fp_out) return fail(PCS_E_INVAL, "null argument");
  StaticPlan plan{};  // on the stack; passed to the kernels by value
  plan.n = n;
  uint64_t chunks = 0;
  for (int i = 0; i < n; ++i) {
    if (bufs[i].bytes > 0 && !bufs[i].ptr) return fail(PCS_E_INVAL, "buffer %d: null pointer", i);
    StaticBuf& b = plan.b[i];
    b.ptr = static_cast<const uint8_t*>(bufs[i].ptr);
    b.bytes = bufs[i].bytes;
    b.n_chunks = n_chunks_of(b.bytes);
    const uintptr_t a = reinterpret_cast<uintptr_t>(b.ptr);
    b.align = (a & 15u) == 0 ? 16u : ((a & 3u) == 0 ? 4u : 1u);
    chunks += b.n_chunks;
  }
  // Smallest warp task (2^g chunks) that keeps every warp busy and fits the
  // fixed node array.
  auto tasks_for = [&](int g) {
    uint64_t t = 0;
    for (int i = 0; i < n; ++i) t += (plan.b[i].n_chunks + (1ull << g) - 1) >> g;
    return t;
  };
  int g = 0;
  while (g < kMaxGroupLog2 && (tasks_for(g) > kStaticMaxNodes || (chunks >> (g + 1)) >= 8192)) ++g;
  const uint64_t tasks = tasks_for(g);
  if (tasks > kStaticMaxNodes)
    return fail(PCS_E_INVAL,
                "pcs_fingerprint_static: these buffers need %llu scratch nodes, the fixed limit "
                "is %u (about 8 GiB per call)",
                static_cast<unsigned long long>(tasks), kStaticMaxNodes);
  uint32_t t = 0;
  for (int i = 0; i < n; ++i) {
    plan.b[i].task_begin = t;
    plan.b[i].n_tasks = static_cast<uint32_t>((plan.b[i].n_chunks + (1ull << g) - 1) >> g);
    t += plan.b[i].n_tasks;
  }
  plan.n_tasks = t;
  plan.glog2 = g;
  uint64_t* nodes = nullptr;
  cudaError_t e = static_scratch(&nodes);
  if (e != cudaSuccess) return cuda_fail(e, "looking up the fixed scratch");
  e = launch_fingerprint_static(plan, nodes, fp_out, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "pcs_fingerprint_static launch");
  return PCS_OK;
}

}  // extern "C"
