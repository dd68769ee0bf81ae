// pcs_kernels.cu -- sm_103a kernels of the PCS hot path.
//
// k_stream<MODE>  one pass over 4 KiB chunks of many byte streams: a warp owns
//                 a task of 2^g chunks; lane l moves the 16-byte segments
//                 l + 32k of each chunk (every warp access is 512 contiguous
//                 bytes), optionally gathers / scatters them through a row or
//                 paged-ring layout, and folds them into the PCSFP64-v1 lane
//                 chain; a shuffle tree makes the chunk hash and then the
//                 task's aligned-group node (Sec. 4 FINGERPRINT, step 1).
// k_bulk<MODE>    the moving passes (pack, restore) of aligned streams: per-warp
//                 TMA pipelines of 8 KiB tiles through shared memory, the
//                 fingerprint of each tile fused into the copy
//                 (k_bulk_shared: the same for small launches, the last
//                 tiles handed out at run time).
// k_hash          the read-only fingerprint pass of aligned buffers: a warp per
//                 8 KiB tile, plain loads into registers, 20 warps per SM.
// k_finalize<MODE> trees the task nodes of each stream into its fingerprint and
//                 writes outputs: fps / classification flags, record headers
//                 and section tables (checkpoint, Sec. 3 "The contract", I4),
//                 or the verification verdict of a restore (I1).
// k_score         cos(query, key) per bank entry, fp32, fixed order (Sec. 5).
// k_topk          per-bank radix select of the k largest (score, -index),
//                 kept indices written in ascending order (Sec. 7.5).
//
// k_gfinish       the global threshold's later digit passes and its
//                 compaction, in one cooperative launch (Sec. 7.5 variant).
//
// Only k_gfinish has blocks that wait on one another, at grid barriers of a
// cooperative launch (all blocks resident); every wait here, there and on an
// mbarrier, gives up after about two seconds and sets the timeout bit.
// Index values read from device memory are bounds-checked; a bad one is
// reported through the error word and skipped.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "pcs_internal.h"

namespace pcs {
namespace {

constexpr uint64_t kP = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kSeed = 0x5043534650363401ull;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned kFull = 0xffffffffu;

// ---------------------------------------------------------------------------
// PCSFP64-v1 primitives
// ---------------------------------------------------------------------------

// SplitMix64 finaliser (Steele, Lea & Flood 2014).
__device__ __forceinline__ uint64_t fmix(uint64_t z) {
  z ^= z >> 30;
  z *= 0xBF58476D1CE4E5B9ull;
  z ^= z >> 27;
  z *= 0x94D049BB133111EBull;
  z ^= z >> 31;
  return z;
}

__device__ __forceinline__ uint64_t rotl64(uint64_t x, int r) {
  return (x << r) | (x >> (64 - r));
}

__device__ __forceinline__ uint64_t comb(uint64_t a, uint64_t b) {
  return fmix(a * kP + rotl64(b, 31));
}

// A hint to bring the 128-byte line holding `p` into this SM's L1.
__device__ __forceinline__ void prefetch_l1(const void* p) {
  asm volatile("prefetch.global.L1 [%0];" ::"l"(p));
}

// Programmatic dependent launch (sm_90 and later).  The streaming, finalising,
// scoring and top-k kernels are launched with programmatic stream
// serialisation (launch_after), so the GPU may schedule one while the kernel
// before it on the stream is still finishing.  Each calls this before it
// touches anything another kernel may write: wait until that kernel has
// completed and its writes are visible, then let the next kernel be
// scheduled.  Before this point a kernel reads only what the host wrote
// before the launch (work lists and section, session and bank
// descriptors), which no kernel writes.
__device__ __forceinline__ void grid_dependency() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Absorb one 16-byte segment (two little-endian words) into a lane chain.
__device__ __forceinline__ uint64_t absorb(uint64_t h, uint4 v) {
  const uint64_t w0 = static_cast<uint64_t>(v.x) | (static_cast<uint64_t>(v.y) << 32);
  const uint64_t w1 = static_cast<uint64_t>(v.z) | (static_cast<uint64_t>(v.w) << 32);
  h = (rotl64(h, 23) ^ w0) * kP;
  h = (rotl64(h, 23) ^ w1) * kP;
  return h;
}

// Fixed-order pairwise tree over the values of lanes [0, n), n <= 32; an odd
// last item is carried up.  The root ends in lane 0.
__device__ __forceinline__ uint64_t warp_tree(uint64_t v, int n, int lane) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t o = __shfl_down_sync(kFull, v, d);
    if ((lane & (2 * d - 1)) == 0 && lane + d < n) v = comb(v, o);
  }
  return v;
}

// Tree over a[0..n) (global or shared), reduced in place by aligned groups
// of 32; every lane returns the root.  Called by one whole warp.
__device__ uint64_t warp_tree_inplace(uint64_t* a, uint32_t n, int lane) {
  while (n > 1) {
    const uint32_t groups = (n + 31) / 32;
    for (uint32_t g = 0; g < groups; ++g) {
      const uint32_t i = 32 * g + lane;
      const uint64_t v = i < n ? a[i] : 0;
      const uint32_t m = min(32u, n - 32 * g);
      const uint64_t r = warp_tree(v, static_cast<int>(m), lane);
      __syncwarp();
      if (lane == 0) a[g] = r;
      __syncwarp();
    }
    n = groups;
  }
  return a[0];
}

// The same tree for n <= 1024, nothing written; called by one whole warp,
// every lane returns the root.  Up to 32 items: one warp tree.  Beyond,
// in blocks of 256 items: lane l reads items 8l .. 8l+7 of the block and
// reduces them in its registers (the tree's first three levels over that
// aligned group of eight, an odd last item carried up), the warp then
// reduces the 32 group roots (five more levels), and the roots of up to four
// blocks end the tree.  Aligned groups of 2^m items reduce to the nodes of
// the global pairwise tree, so the root is the same; all 32 lanes combine
// at once, where trees of 32-item groups leave half the lanes idle at each
// level (a 256-item tree took 1,790 warp instructions that way).
__device__ uint64_t warp_tree_regs(const uint64_t* a, uint32_t n, int lane) {
  if (n <= 32) {
    const uint64_t v = lane < static_cast<int>(n) ? a[lane] : 0;
    return __shfl_sync(kFull, warp_tree(v, static_cast<int>(n), lane), 0);
  }
  const uint32_t blocks = (n + 255) / 256;
  uint64_t block_root = 0;  // root of block b, kept in lane b
  for (uint32_t b = 0; b < blocks; ++b) {
    const uint32_t base = 256 * b;
    const uint32_t nb = min(256u, n - base);
    const int m = max(0, min(8, static_cast<int>(nb) - 8 * lane));  // this lane's items
    uint64_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = i < m ? a[base + 8 * lane + i] : 0;
#pragma unroll
    for (int w = 1; w < 8; w <<= 1)
#pragma unroll
      for (int i = 0; i + w < 8; i += 2 * w)
        if (i + w < m) v[i] = comb(v[i], v[i + w]);
    const uint64_t r = __shfl_sync(kFull, warp_tree(v[0], static_cast<int>((nb + 7) / 8), lane), 0);
    if (lane == static_cast<int>(b)) block_root = r;
  }
  const uint64_t root = blocks > 1 ? warp_tree(block_root, static_cast<int>(blocks), lane) : block_root;
  return __shfl_sync(kFull, root, 0);
}

// Tree of a 2-chunk tile, both chunks at once.  Lane l holds a0 = lane value
// l of chunk 0 and a1 = lane value l of chunk 1.  Level 1 puts chunk q's pair
// (2i, 2i+1) in lane 16q + i; from then on the pair of every level is in lanes
// (2L, 2L+1), so each level is one comb across the warp.  After five levels
// lane q holds chunk q's hash; with nc == 2 one more level gives the tile's
// node comb(x0, x1) (the pairwise tree over its chunks).  Result in lane 0.
__device__ __forceinline__ uint64_t tile_tree2(uint64_t a0, uint64_t a1, int nc, int lane) {
  const int i = lane & 15;
  const uint64_t l0 = __shfl_sync(kFull, a0, 2 * i), r0 = __shfl_sync(kFull, a0, 2 * i + 1);
  const uint64_t l1 = __shfl_sync(kFull, a1, 2 * i), r1 = __shfl_sync(kFull, a1, 2 * i + 1);
  uint64_t v = lane < 16 ? comb(l0, r0) : comb(l1, r1);
  const int levels = nc == 2 ? 5 : 4;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    if (k < levels) {
      const uint64_t l = __shfl_sync(kFull, v, (2 * lane) & 31);
      const uint64_t r = __shfl_sync(kFull, v, (2 * lane + 1) & 31);
      v = comb(l, r);
    }
  }
  return v;
}

// ---------------------------------------------------------------------------
// Memory helpers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint4 ld_stream(const uint8_t* p) {
  return __ldcs(reinterpret_cast<const uint4*>(p));
}

__device__ __forceinline__ void st_stream(uint8_t* p, uint4 v) {
  __stcs(reinterpret_cast<uint4*>(p), v);
}

// Bytes [0, n) of a segment (n <= 16) at an address that may not be 16-byte
// aligned; whole 32-bit words when `a4` (4-byte aligned).  The rest read as 0.
__device__ __forceinline__ uint4 ld_small(const uint8_t* p, int n, bool a4) {
  uint32_t w[4] = {0, 0, 0, 0};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (a4 && 4 * j + 4 <= n) {
      w[j] = *reinterpret_cast<const uint32_t*>(p + 4 * j);
    } else {
#pragma unroll
      for (int b = 0; b < 4; ++b)
        if (4 * j + b < n) w[j] |= static_cast<uint32_t>(p[4 * j + b]) << (8 * b);
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void st_small(uint8_t* p, uint4 v, int n, bool a4) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (a4 && 4 * j + 4 <= n) {
      *reinterpret_cast<uint32_t*>(p + 4 * j) = w[j];
    } else {
#pragma unroll
      for (int b = 0; b < 4; ++b)
        if (4 * j + b < n) p[4 * j + b] = static_cast<uint8_t>(w[j] >> (8 * b));
    }
  }
}

// Zero the bytes of a segment at or past `n` (n in [1, 16)).
__device__ __forceinline__ uint4 mask_tail(uint4 v, int n) {
  uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int keep = n - 4 * j;  // bytes of word j to keep
    if (keep <= 0) w[j] = 0;
    else if (keep < 4) w[j] &= (1u << (8 * keep)) - 1u;
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ uint64_t div_rows(uint64_t x, uint64_t d, int shift) {
  return shift >= 0 ? (x >> shift) : (x / d);
}

// Address of logical byte `off` (a multiple of 16) on the layout side of a
// ROWS / RING stream, or null if its row / page id is out of range.
__device__ __forceinline__ uint8_t* row_addr(const SecDesc& s, uint64_t off, uint32_t* err) {
  const uint64_t r = div_rows(off, s.row_bytes, s.rb_shift);
  const uint64_t w = off - r * s.row_bytes;
  uint64_t id, row;
  if (s.layout == kRows) {
    id = static_cast<uint32_t>(__ldg(s.index + r));
    row = id;
  } else {
    // RING: logical row r sits in ring slot (start + r) mod window.
    uint64_t slot = s.ring_start + r;
    if (slot >= s.window) slot -= s.window;
    const uint64_t pg = div_rows(slot, s.page_rows, s.pr_shift);
    id = static_cast<uint32_t>(__ldg(s.index + pg));
    row = id * s.page_rows + (slot - pg * s.page_rows);
  }
  if (id >= s.base_rows) {
    atomicOr(err, kDevErrIndex);
    return nullptr;
  }
  return s.lbase + row * s.row_bytes + w;
}

// ---------------------------------------------------------------------------
// Streaming kernel
// ---------------------------------------------------------------------------

constexpr int kSegs = 8;  // 16-byte segments per lane per chunk

template <int MODE>
struct ModeTraits {
  static constexpr bool kHash = MODE == kModeHash || MODE == kModePack || MODE == kModeRestoreV;
  static constexpr bool kLoadLayout = MODE == kModeHash || MODE == kModePack;
  static constexpr bool kStore = MODE != kModeHash;
};

// Load segment `off` of a stream from its read side.
template <int MODE>
__device__ __forceinline__ uint4 load_seg(const SecDesc& s, uint64_t off, uint32_t* err) {
  const uint4 z = make_uint4(0, 0, 0, 0);
  if (off >= s.bytes) return z;
  if (ModeTraits<MODE>::kLoadLayout) {
    if (s.layout == kContig) {
      const uint64_t left = s.bytes - off;
      if (left >= 16 && s.align == 16) return ld_stream(s.lbase + off);
      return ld_small(s.lbase + off, left < 16 ? static_cast<int>(left) : 16, s.align >= 4);
    }
    const uint8_t* p = row_addr(s, off, err);
    return p ? ld_stream(p) : z;
  } else {
    // Payload inside a record: padded to 256 bytes, so a whole segment is
    // readable; bytes past the logical end are masked to zero.
    uint4 v = ld_stream(s.payload + off);
    const uint64_t left = s.bytes - off;
    if (left < 16) v = mask_tail(v, static_cast<int>(left));
    return v;
  }
}

// Store segment `off` to a stream's write side.
template <int MODE>
__device__ __forceinline__ void store_seg(const SecDesc& s, uint64_t off, uint4 v, uint32_t* err) {
  if (MODE == kModePack) {
    // Record payload: write through the 256-byte padding (zeros past L).
    const uint64_t padded = (s.bytes + kRecordAlign - 1) / kRecordAlign * kRecordAlign;
    if (off < padded) st_stream(s.payload + off, v);
  } else if (MODE == kModeRestore || MODE == kModeRestoreV) {
    if (off >= s.bytes) return;
    if (s.layout == kContig) {
      const uint64_t left = s.bytes - off;
      if (left >= 16 && s.align == 16) st_stream(s.lbase + off, v);
      else st_small(s.lbase + off, v, left < 16 ? static_cast<int>(left) : 16, s.align >= 4);
      return;
    }
    uint8_t* p = row_addr(s, off, err);
    if (p) st_stream(p, v);
  }
}

// Section of warp task `task` in a work list: the last j with begin[j] <=
// task (begin rises), searched from item `lo` on (begin[lo] <= task; lo = 0
// searches the whole list, begin[0] = 0).  Called by a whole warp with a
// warp-uniform task: each round the lanes probe 32 evenly spaced entries of
// the range still open and keep the part after the last probe <= task, so
// that 12,544 items take three dependent loads instead of fourteen.
__device__ __forceinline__ int find_item(const uint32_t* __restrict__ begin, int lo, int n_items,
                                        uint32_t task, int lane) {
  int span = n_items - lo;  // the answer lies in [lo, lo + span)
  while (span > 1) {
    const int step = (span + 31) >> 5;
    const int i = lo + lane * step;
    const bool le = i < lo + span && __ldg(begin + i) <= task;
    const unsigned m = __ballot_sync(kFull, le);  // lane 0 probes lo: never empty
    const int last = 31 - __clz(m);
    lo += last * step;
    span = min(step, span - last * step);
  }
  return lo;
}

// The warp tasks of one streaming pass (body of k_stream and k_small).
template <int MODE>
__device__ __forceinline__ void run_stream_tasks(const SecDesc* __restrict__ secs, const WorkList& wl,
                                                 int glog2, uint64_t* __restrict__ nodes,
                                                 uint32_t* err, SecDesc* sdesc) {
  using T = ModeTraits<MODE>;
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const uint32_t nw = gridDim.x * kWarps;
  int cur = -1;
  for (uint32_t task = blockIdx.x * kWarps + wib; task < wl.n_tasks; task += nw) {
    const int j = find_item(wl.begin, 0, wl.n_items, task, lane);
    if (j != cur) {
      __syncwarp();
      const SecDesc* src = &secs[__ldg(wl.ids + j)];
      if (lane < static_cast<int>(sizeof(SecDesc) / 16))
        reinterpret_cast<uint4*>(&sdesc[wib])[lane] = __ldg(reinterpret_cast<const uint4*>(src) + lane);
      __syncwarp();
      cur = j;
    }
    const SecDesc& s = sdesc[wib];
    const uint32_t local = task - __ldg(wl.begin + j);
    const uint64_t c0 = static_cast<uint64_t>(local) << glog2;
    const uint64_t c1 = min(c0 + (1ull << glog2), static_cast<unsigned long long>(s.n_chunks));
    uint64_t mine = 0;  // lane j keeps the hash of chunk c0 + j
    for (uint64_t c = c0; c < c1; c += 2) {
      const bool two = c + 1 < c1;
      const uint64_t base = c * kChunkBytes + 16u * lane;
      uint4 va[kSegs], vb[kSegs];
#pragma unroll
      for (int k = 0; k < kSegs; ++k) va[k] = load_seg<MODE>(s, base + 512u * k, err);
      if (two) {
#pragma unroll
        for (int k = 0; k < kSegs; ++k) vb[k] = load_seg<MODE>(s, base + kChunkBytes + 512u * k, err);
      }
      if (T::kStore) {
#pragma unroll
        for (int k = 0; k < kSegs; ++k) store_seg<MODE>(s, base + 512u * k, va[k], err);
        if (two) {
#pragma unroll
          for (int k = 0; k < kSegs; ++k) store_seg<MODE>(s, base + kChunkBytes + 512u * k, vb[k], err);
        }
      }
      if (T::kHash) {
        uint64_t ha = fmix(kSeed ^ (c * 32u + lane));
#pragma unroll
        for (int k = 0; k < kSegs; ++k) ha = absorb(ha, va[k]);
        ha = __shfl_sync(kFull, warp_tree(fmix(ha), 32, lane), 0);
        const int jj = static_cast<int>(c - c0);
        if (lane == jj) mine = ha;
        if (two) {
          uint64_t hb = fmix(kSeed ^ ((c + 1) * 32u + lane));
#pragma unroll
          for (int k = 0; k < kSegs; ++k) hb = absorb(hb, vb[k]);
          hb = __shfl_sync(kFull, warp_tree(fmix(hb), 32, lane), 0);
          if (lane == jj + 1) mine = hb;
        }
      }
    }
    if (T::kHash) {
      const uint64_t root = warp_tree(mine, static_cast<int>(c1 - c0), lane);
      if (lane == 0) nodes[s.task_begin + local] = root;
    }
  }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 2)
    k_stream(const SecDesc* __restrict__ secs, WorkList wl, int glog2,
             uint64_t* __restrict__ nodes, uint32_t* err) {
  grid_dependency();
  __shared__ SecDesc sdesc[kWarps];
  run_stream_tasks<MODE>(secs, wl, glog2, nodes, err, sdesc);
}

// ---------------------------------------------------------------------------
// TMA-staged streaming kernel
//
// Every warp runs its own pipeline over a contiguous range of tiles; a tile
// is 2 chunks (8 KiB) of one stream in payload order.  A warp owns
// kWarpStages shared-memory stages: it stages tile i + kWarpStages while it
// works on tile i.  Staging is one cp.async.bulk copy per run of rows that
// are contiguous in memory (or one copy of the contiguous payload), all
// completing on the stage's mbarrier; working on a tile = hash its chunks
// from shared memory, issue the bulk store of the tile (to the payload, or
// one per row run of the layout side), and wait until the store has read
// the stage.  Warps never wait on each other.  Every wait is bounded; a wait
// that gives up records kDevErrTimeout and the warp stops.
// ---------------------------------------------------------------------------

constexpr int kTileChunks = kBulkTileChunks;
constexpr uint32_t kTileBytes = kTileChunks * kChunkBytes;

// Shape of the TMA kernel (the moving modes: pack, restore, verified
// restore): warps per block and stages per warp, 3 tiles per warp in flight.
// The read-only hash pass has a kernel of its own (k_hash, below).
template <int MODE>
struct BulkShape {
  static_assert(MODE != kModeHash, "the hash-only pass runs in k_hash");
  static constexpr int kWarps = 8;
  static constexpr int kStages = 3;
  static constexpr int kThreads = 32 * kWarps;
};
// Copies one contiguous 8 KiB load of a hashing pass is split into (1 KiB
// each).  Measured, 4,096 and 16,384 Markov sessions of 192 KiB: pack 0.308
// -> 0.276 ms and 1.105 -> 1.001 ms, verified restore 0.304 -> 0.268 ms and
// 1.108 -> 0.993 ms (2, 4 and 16 pieces gained less).  Plain
// restores keep one copy (a fork of 256 KV records lost 1.3 % with pieces),
// and so do loads of a restore into rows (split, the KV step's verified
// restore took twice as long).
constexpr int kContigPieces = 8;
static_assert(kTileBytes / kContigPieces % 16 == 0 && kContigPieces <= 32, "pieces");
// Work sharing of the TMA kernel.  With static ranges alone, warps given
// equal tile counts finish up to 10-25 % apart (a per-warp %globaltimer
// probe: 4,096 Markov sessions 226-263 us, median 236; 64 banks 69-92 us,
// median 79).  A launch of fewer than kDynMaxTilesPerWarp tiles per warp
// runs k_bulk_shared: 1 / kDynShare of its tiles (the last ones) are handed
// out at run time, in chunks of up to kDynChunkMax tiles, about
// kDynGrabsPerWarp per warp.  Measured (alternating builds, one box): the
// 64-bank step 0.273 -> 0.261 ms; at 84 tiles per warp (4,096 Markov
// sessions) no change; at 2,587 (the 256-session KV step) sharing 1/4 or 1/8
// made the step 0.7-1.5 % slower, so large launches keep static ranges.
constexpr uint32_t kDynMaxTilesPerWarp = 64;
constexpr uint32_t kDynShare = 8;
constexpr uint32_t kDynGrabsPerWarp = 8;
constexpr uint32_t kDynChunkMax = 32;
constexpr int kTileRows = 32;  // rows >= 512 bytes touching an 8 KiB tile: at most 17
constexpr long long kWaitCycles = 4000000000ll;  // give up a wait after ~2 s of SM clock
static_assert(kTileBytes / kBulkMinRowBytes + 1 <= kTileRows, "tile rows");

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(20000u)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase of `bar` with the given parity to complete.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
  return true;
}

__device__ __forceinline__ void bulk_g2s(void* sdst, const void* gsrc, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(sdst)),
      "l"(gsrc), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void bulk_s2g(void* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst),
               "r"(smem_u32(ssrc)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// What a stage holds (written by the warp when it stages the tile).
struct WarpStage {
  SecDesc d;                // the tile's stream
  uint32_t sec;             // its index (0xFFFFFFFF: none yet)
  uint64_t p0, p1;          // payload bytes of the tile: [p0, p1)
  uint64_t r0;              // first row touching the tile (ROWS / RING)
  uint32_t node;            // node slot of the tile
  uint32_t n_rows;          // rows touching [p0, min(p1, L))
  uint8_t* rowp[kTileRows]; // layout-side address of each row (null = out of range)
};

template <int W, int S>
struct BulkShared {
  alignas(128) uint8_t buf[W][S][kTileBytes];
  alignas(8) uint64_t bar[W][S];
  WarpStage st[W][S];
};

// Layout-side address of row r of a ROWS / RING stream (null if out of range).
__device__ __forceinline__ uint8_t* row_ptr(const SecDesc& s, uint64_t r, uint32_t* err) {
  uint64_t id, row;
  if (s.layout == kRows) {
    id = static_cast<uint32_t>(__ldg(s.index + r));
    row = id;
  } else {
    uint64_t slot = s.ring_start + r;
    if (slot >= s.window) slot -= s.window;
    const uint64_t pg = div_rows(slot, s.page_rows, s.pr_shift);
    id = static_cast<uint32_t>(__ldg(s.index + pg));
    row = id * s.page_rows + (slot - pg * s.page_rows);
  }
  if (id >= s.base_rows) {
    atomicOr(err, kDevErrIndex);
    return nullptr;
  }
  return s.lbase + row * s.row_bytes;
}

// End of the bytes of tile [p0, p1) that bulk copies stage: the layout side
// up to its last whole 16-byte segment; the payload (padded to 256 bytes in
// the record) up to its 16-byte-rounded end.
template <int MODE>
__device__ __forceinline__ uint64_t staged_end(const SecDesc& s, uint64_t p1) {
  const uint64_t end =
      ModeTraits<MODE>::kLoadLayout ? (s.bytes & ~15ull) : ((s.bytes + 15) & ~15ull);
  return p1 < end ? p1 : end;
}

// Bytes of [p0, pe) that row i of a stage covers.
__device__ __forceinline__ uint32_t row_share(const WarpStage& m, uint64_t rb, int i, uint64_t pe) {
  const uint64_t lo = (m.r0 + i) * rb, hi = lo + rb;
  const uint64_t a = lo > m.p0 ? lo : m.p0, b = hi < pe ? hi : pe;
  return b > a ? static_cast<uint32_t>(b - a) : 0u;
}

// Bulk copies between a stage's buffer and the layout side, one per run of
// rows contiguous in memory, covering payload bytes [m.p0, pe).  Lane i owns
// row i (address rp; null = skipped).  Returns the bytes this lane copied.
template <bool kLoad>
__device__ __forceinline__ uint32_t issue_runs(const WarpStage& m, uint8_t* rp, uint64_t pe,
                                               uint8_t* tile, uint64_t* bar, int lane) {
  const uint64_t rb = m.d.row_bytes;
  const int n = static_cast<int>(m.n_rows);
  const uintptr_t u = reinterpret_cast<uintptr_t>(rp);
  const uintptr_t prev = __shfl_up_sync(kFull, u, 1);
  const bool start = lane < n && (lane == 0 || u == 0 || prev == 0 || u != prev + rb);
  const unsigned starts = __ballot_sync(kFull, start);
  if (!start || rp == nullptr) return 0;
  const unsigned later = lane < 31 ? (starts >> (lane + 1)) : 0u;
  const int next = later ? lane + __ffs(later) : n;
  const uint64_t row_lo = (m.r0 + lane) * rb, row_hi = (m.r0 + next) * rb;
  const uint64_t a = row_lo > m.p0 ? row_lo : m.p0;
  const uint64_t b = row_hi < pe ? row_hi : pe;
  if (a >= b) return 0;
  uint8_t* g = rp + (a - row_lo);
  uint8_t* sp = tile + (a - m.p0);
  if (kLoad) bulk_g2s(sp, g, static_cast<uint32_t>(b - a), bar);
  else bulk_s2g(g, sp, static_cast<uint32_t>(b - a));
  return static_cast<uint32_t>(b - a);
}

// Copy the descriptor of section `sec` into a stage (a whole warp; nothing
// is read when the stage already holds it).
__device__ __forceinline__ void stage_desc(const SecDesc* __restrict__ secs, uint32_t sec,
                                           WarpStage& st, int lane) {
  if (st.sec != sec) {  // warp-uniform
    __syncwarp();
    if (lane < static_cast<int>(sizeof(SecDesc) / 16))
      reinterpret_cast<uint4*>(&st.d)[lane] = __ldg(reinterpret_cast<const uint4*>(secs + sec) + lane);
    if (lane == 0) st.sec = sec;
  }
  __syncwarp();
}

// Stage tile t (of work list item `item`) into stage `st` / barrier `bar`.
template <int MODE>
__device__ __forceinline__ void stage_tile(const SecDesc* __restrict__ secs, const WorkList& wl,
                                           int item, uint32_t t, WarpStage& st, uint8_t* tile,
                                           uint64_t* bar, uint32_t* err, int lane) {
  using T = ModeTraits<MODE>;
  const uint32_t sec = __ldg(wl.ids + item);
  const uint32_t loc = t - __ldg(wl.begin + item);
  stage_desc(secs, sec, st, lane);
  const SecDesc& s = st.d;
  const uint64_t L = s.bytes;
  const uint64_t p0 = static_cast<uint64_t>(loc) * kTileBytes;
  const uint64_t cend = s.n_chunks * kChunkBytes;
  const uint64_t p1 = p0 + kTileBytes < cend ? p0 + kTileBytes : cend;
  const uint64_t pe = staged_end<MODE>(s, p1);
  uint64_t r0 = 0;
  uint32_t n_rows = 0;
  uint8_t* rp = nullptr;
  if (s.layout != kContig) {
    r0 = div_rows(p0, s.row_bytes, s.rb_shift);
    const uint64_t lim = L < p1 ? L : p1;
    if (lim > p0) n_rows = static_cast<uint32_t>(div_rows(lim - 1, s.row_bytes, s.rb_shift) + 1 - r0);
    if (lane < static_cast<int>(n_rows)) rp = row_ptr(s, r0 + lane, err);
    st.rowp[lane] = rp;
  }
  if (lane == 0) {
    st.p0 = p0;
    st.p1 = p1;
    st.r0 = r0;
    st.node = s.task_begin + loc;
    st.n_rows = n_rows;
  }
  __syncwarp();
  if (!T::kLoadLayout || s.layout == kContig) {
    // One contiguous piece: the record payload, or a contiguous buffer.  A
    // hashing pass whose layout side is contiguous (a pack from a
    // contiguous buffer, a verified restore into one) loads it as
    // kContigPieces copies issued by as many lanes.
    const uint32_t bytes = pe > p0 ? static_cast<uint32_t>(pe - p0) : 0u;
    const int pieces = (T::kHash && s.layout == kContig) ? kContigPieces : 1;
    if (lane == 0) mbar_arrive_expect_tx(bar, bytes);
    __syncwarp();
    if (lane < pieces && bytes) {
      const uint32_t piece = ((bytes + pieces - 1) / pieces + 15u) & ~15u;
      const uint32_t lo = static_cast<uint32_t>(lane) * piece;
      const uint32_t hi = lo + piece < bytes ? lo + piece : bytes;
      if (hi > lo) bulk_g2s(tile + lo, (T::kLoadLayout ? s.lbase : s.payload) + p0 + lo, hi - lo, bar);
    }
    return;
  }
  // Rows: zero the share of rows whose id was out of range, arm the barrier
  // with the bytes the copies will bring, then one bulk copy per run.
  uint32_t mine = 0;
  if (lane < static_cast<int>(n_rows)) {
    const uint32_t share = row_share(st, s.row_bytes, lane, pe);
    if (rp == nullptr) {
      const uint64_t lo = (r0 + lane) * s.row_bytes;
      const uint64_t a = lo > p0 ? lo : p0;
      for (uint32_t o = 0; o < share; o += 16)
        *reinterpret_cast<uint4*>(tile + (a - p0) + o) = make_uint4(0, 0, 0, 0);
      fence_async_smem();
    } else {
      mine = share;
    }
  }
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) mine += __shfl_xor_sync(kFull, mine, d);
  if (lane == 0) mbar_arrive_expect_tx(bar, mine);
  __syncwarp();
  issue_runs<true>(st, rp, pe, tile, bar, lane);
}

// One staged tile whose loads have landed: complete it, issue its stores
// (one bulk group), fold its chunks into the fingerprint and write its node.
// Returns whether stores were issued.  Called by a whole warp.
template <int MODE>
__device__ __forceinline__ bool bulk_tile(const WarpStage& m, uint8_t* tile,
                                          uint64_t* __restrict__ nodes, int lane) {
  using T = ModeTraits<MODE>;
  const uint4 zero = make_uint4(0, 0, 0, 0);
  const SecDesc& s = m.d;
  const uint64_t L = s.bytes, p0 = m.p0, p1 = m.p1;
  const uint64_t pe = staged_end<MODE>(s, p1);
  // Complete the tile: [pe, p1) holds the stream's unaligned tail (layout
  // side) and zeros past its end.
  for (uint64_t o = pe + 16u * lane; o < p1; o += 512u) {
    uint4 v = zero;
    if (T::kLoadLayout && o < L) {
      const uint64_t left = L - o;
      v = ld_small(s.lbase + o, left < 16 ? static_cast<int>(left) : 16, true);
    }
    *reinterpret_cast<uint4*>(tile + (o - p0)) = v;
  }
  if (!T::kLoadLayout && (L & 15u) && L >= p0 && L < p1 && lane == 0) {
    // Restore: payload bytes past the logical end read as zero.
    const uint64_t o = L & ~15ull;
    uint4* q = reinterpret_cast<uint4*>(tile + (o - p0));
    *q = mask_tail(*q, static_cast<int>(L - o));
  }
  fence_async_smem();
  __syncwarp();
  bool issued = false;
  if (MODE == kModePack) {
    // Contiguous payload, through the record's 256-byte padding.
    const uint64_t padded = (L + kRecordAlign - 1) / kRecordAlign * kRecordAlign;
    const uint64_t se = p1 < padded ? p1 : padded;
    if (lane == 0 && se > p0) {
      bulk_s2g(s.payload + p0, tile, static_cast<uint32_t>(se - p0));
      bulk_commit();
      issued = true;
    }
  } else if (MODE == kModeRestore || MODE == kModeRestoreV) {
    const uint64_t lim = L < p1 ? L : p1;
    if (s.layout == kContig) {
      const uint64_t vend = lim & ~15ull;  // whole segments by bulk copy
      if (lane == 0 && vend > p0) {
        bulk_s2g(s.lbase + p0, tile, static_cast<uint32_t>(vend - p0));
        bulk_commit();
        issued = true;
      }
      for (uint64_t o = (vend > p0 ? vend : p0) + lane; o < lim; o += 32) s.lbase[o] = tile[o - p0];
    } else {
      uint8_t* rp = m.rowp[lane];
      if (issue_runs<false>(m, rp, lim, tile, nullptr, lane)) {
        bulk_commit();
        issued = true;
      }
    }
  }
  if (T::kHash) {
    // The tile's chunks, interleaved lane chains, read from shared memory.
    const uint64_t c0 = p0 / kChunkBytes;
    const int nc = static_cast<int>((p1 - p0) / kChunkBytes);
    uint64_t h[kTileChunks];
#pragma unroll
    for (int q = 0; q < kTileChunks; ++q) h[q] = fmix(kSeed ^ ((c0 + q) * 32u + lane));
#pragma unroll
    for (int k = 0; k < kSegs; ++k) {
#pragma unroll
      for (int q = 0; q < kTileChunks; ++q) {
        const uint4 v = q < nc ? *reinterpret_cast<const uint4*>(tile + q * kChunkBytes + 512 * k + 16 * lane)
                               : zero;
        h[q] = absorb(h[q], v);
      }
    }
    // Moving passes are bound by DRAM; one tree per chunk paces the warps
    // so that loads and stores interleave best (measured: the shared tree
    // of tile_tree2 makes pack and restore slower).
    uint64_t mine = 0;
#pragma unroll
    for (int q = 0; q < kTileChunks; ++q) {
      const uint64_t x = __shfl_sync(kFull, warp_tree(fmix(h[q]), 32, lane), 0);
      if (lane == q) mine = x;
    }
    const uint64_t root = warp_tree(mine, nc, lane);
    if (lane == 0) nodes[m.node] = root;
  }
  return issued;
}

// The TMA kernel with static work: each warp moves a contiguous, balanced
// range of the launch's tiles, kWarpStages in flight.
template <int MODE>
__global__ void __launch_bounds__(BulkShape<MODE>::kThreads, 1)
    k_bulk(const SecDesc* __restrict__ secs, WorkList wl, uint64_t* __restrict__ nodes,
           uint32_t* err) {
  constexpr int kBulkWarps = BulkShape<MODE>::kWarps;
  constexpr int kWarpStages = BulkShape<MODE>::kStages;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  auto& sh = *reinterpret_cast<BulkShared<kBulkWarps, kWarpStages>*>(smem_raw);
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  if (lane < kWarpStages) {
    mbar_init(&sh.bar[warp][lane], 1);
    sh.st[warp][lane].sec = 0xFFFFFFFFu;
  }
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncwarp();

  // This warp's tiles: a contiguous, balanced range [t0, t1).
  const uint64_t T_all = wl.n_tasks;
  const uint64_t gw = static_cast<uint64_t>(blockIdx.x) * kBulkWarps + warp;
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kBulkWarps;
  const uint32_t t0 = static_cast<uint32_t>(T_all * gw / nw);
  const uint32_t t1 = static_cast<uint32_t>(T_all * (gw + 1) / nw);
  if (t0 >= t1) return;
  // The work list and the descriptors are the host's, written before the
  // launch: the first tile's item and section are found while the kernel
  // ahead on the stream drains.
  int item = find_item(wl.begin, 0, wl.n_items, t0, lane);  // item of the next tile to stage
  stage_desc(secs, __ldg(wl.ids + item), sh.st[warp][0], lane);
  grid_dependency();
  auto item_of = [&](uint32_t t) {
    while (item + 1 < wl.n_items && __ldg(wl.begin + item + 1) <= t) ++item;
    return item;
  };
  const int pre = static_cast<int>(t1 - t0 < static_cast<uint32_t>(kWarpStages) ? t1 - t0 : kWarpStages);
  for (int k = 0; k < pre; ++k)
    stage_tile<MODE>(secs, wl, item_of(t0 + k), t0 + k, sh.st[warp][k], sh.buf[warp][k],
                     &sh.bar[warp][k], err, lane);
  bool any_issued = false;
  for (uint32_t i = 0; t0 + i < t1; ++i) {
    const int sidx = static_cast<int>(i % kWarpStages);
    const uint32_t use = i / kWarpStages;
    uint64_t* bar = &sh.bar[warp][sidx];
    uint8_t* tile = sh.buf[warp][sidx];
    WarpStage& m = sh.st[warp][sidx];
    bool ok = true;
    if (lane == 0) ok = mbar_wait(bar, use & 1);
    ok = __shfl_sync(kFull, ok, 0);
    if (!ok) {
      if (lane == 0) atomicOr(err, kDevErrTimeout);
      break;
    }
    if (bulk_tile<MODE>(m, tile, nodes, lane)) {
      bulk_wait_read();
      any_issued = true;
    }
    __syncwarp();
    // Reuse the stage for tile i + kWarpStages.
    const uint32_t tn = t0 + i + kWarpStages;
    if (tn < t1) stage_tile<MODE>(secs, wl, item_of(tn), tn, m, tile, bar, err, lane);
  }
  if (any_issued) bulk_wait_all();
}

// The TMA kernel with shared work, for launches of fewer than
// kDynMaxTilesPerWarp tiles per warp: each warp first moves a contiguous,
// balanced range of the first T_static tiles, then chunks of the rest
// [T_static, T_all) handed out by an atomic counter (sched[0]) to whichever
// warp asks first, so that warps that drew slower memory do not hold up the
// end of the launch.  sched[0..1] are zero on entry; the last warp to finish
// sets them back to zero.
template <int MODE>
__global__ void __launch_bounds__(BulkShape<MODE>::kThreads, 1)
    k_bulk_shared(const SecDesc* __restrict__ secs, WorkList wl, uint64_t* __restrict__ nodes,
                  uint32_t* err, uint32_t* sched) {
  constexpr int kBulkWarps = BulkShape<MODE>::kWarps;
  constexpr int kWarpStages = BulkShape<MODE>::kStages;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  auto& sh = *reinterpret_cast<BulkShared<kBulkWarps, kWarpStages>*>(smem_raw);
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  if (lane < kWarpStages) {
    mbar_init(&sh.bar[warp][lane], 1);
    sh.st[warp][lane].sec = 0xFFFFFFFFu;
  }
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncwarp();

  const uint32_t T_all = wl.n_tasks;
  const uint64_t gw = static_cast<uint64_t>(blockIdx.x) * kBulkWarps + warp;
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kBulkWarps;
  const uint32_t T_dyn = T_all / kDynShare;
  const uint32_t T_static = T_all - T_dyn;
  const uint64_t per = T_dyn / (nw * kDynGrabsPerWarp);
  const uint32_t chunk = static_cast<uint32_t>(per < 1 ? 1 : (per > kDynChunkMax ? kDynChunkMax : per));
  const uint32_t t0 = static_cast<uint32_t>(T_static * gw / nw);
  const uint32_t t1 = static_cast<uint32_t>(T_static * (gw + 1) / nw);
  uint32_t next = t0, chunk_end = t1;  // tiles [next, chunk_end) are this warp's
  int item = find_item(wl.begin, 0, wl.n_items, t0, lane);  // item of the last tile taken
  // The work list and the descriptors are the host's: the first static
  // tile's section is read before waiting for the kernel ahead.  The
  // counters in `sched` are touched only after the wait.
  if (t0 < t1) stage_desc(secs, __ldg(wl.ids + item), sh.st[warp][0], lane);
  grid_dependency();
  // The next chunk, reserved ahead of need (where the warp would wait on a
  // stage anyway) so that neither the atomic nor the search of its item
  // delays a refill.
  bool reserved = false, drained = false;
  uint32_t res_next = 0, res_end = 0;
  int res_item = 0;
  auto reserve = [&]() {
    if (reserved || drained) return;
    uint32_t g = 0;
    if (lane == 0) g = atomicAdd(sched, chunk);
    g = __shfl_sync(kFull, g, 0);
    if (g >= T_dyn) {
      drained = true;
      return;
    }
    res_next = T_static + g;
    res_end = T_static + (g + chunk < T_dyn ? g + chunk : T_dyn);
    res_item = item + 1 < wl.n_items && __ldg(wl.begin + item + 1) <= res_next
                   ? find_item(wl.begin, item, wl.n_items, res_next, lane)
                   : item;
    reserved = true;
  };
  // The next tile of this warp (and `item`, its item); false once none is left.
  auto take = [&](uint32_t* t) -> bool {
    if (next >= chunk_end) {
      reserve();
      if (!reserved) return false;
      next = res_next;
      chunk_end = res_end;
      item = res_item;
      reserved = false;
    }
    *t = next++;
    while (item + 1 < wl.n_items && __ldg(wl.begin + item + 1) <= *t) ++item;
    return true;
  };
  int staged = 0;
  for (int k = 0; k < kWarpStages; ++k) {
    uint32_t t;
    if (!take(&t)) break;
    stage_tile<MODE>(secs, wl, item, t, sh.st[warp][k], sh.buf[warp][k], &sh.bar[warp][k], err,
                     lane);
    ++staged;
  }
  bool any_issued = false;
  for (int i = 0; i < staged; ++i) {
    const int sidx = i % kWarpStages;
    const uint32_t use = static_cast<uint32_t>(i) / kWarpStages;
    uint64_t* bar = &sh.bar[warp][sidx];
    uint8_t* tile = sh.buf[warp][sidx];
    WarpStage& m = sh.st[warp][sidx];
    if (next + 1 >= chunk_end) reserve();  // the refill after next needs a new chunk
    bool ok = true;
    if (lane == 0) ok = mbar_wait(bar, use & 1);
    ok = __shfl_sync(kFull, ok, 0);
    if (!ok) {
      if (lane == 0) atomicOr(err, kDevErrTimeout);
      break;
    }
    if (bulk_tile<MODE>(m, tile, nodes, lane)) {
      bulk_wait_read();
      any_issued = true;
    }
    __syncwarp();
    // Reuse the stage for this warp's next tile.
    uint32_t tn;
    if (take(&tn)) {
      stage_tile<MODE>(secs, wl, item, tn, m, tile, bar, err, lane);
      ++staged;
    }
  }
  if (any_issued) bulk_wait_all();
  // The last warp out leaves the counters at zero for the next launch.
  if (lane == 0) {
    __threadfence();
    if (atomicAdd(sched + 1, 1u) == static_cast<uint32_t>(nw) - 1) {
      atomicExch(sched, 0u);
      atomicExch(sched + 1, 0u);
    }
  }
}

// ---------------------------------------------------------------------------
// Read-only fingerprint pass (hash mode of the streams the TMA kernel would
// take: 16-byte aligned contiguous device buffers)
//
// Every warp walks a contiguous range of 8 KiB tiles; per tile each lane
// issues its sixteen 16-byte loads (segments lane + 32k of both chunks) into
// registers, then runs the two lane chains interleaved and one shared tree
// (tile_tree2).  No shared memory: 20 warps per SM fit in the register file
// (88 registers), and their loads hide each other's hashing.  Measured on
// the 200-buffer classify sweep: 6.68 TB/s, against 6.27 TB/s for the TMA
// pipeline with two 8 KiB stages per warp (which shared memory capped at 12
// warps) and 6.99 TB/s for a plain-load byte compare of the same pairs;
// 16 warps 6.49, 24 warps (spilling) 6.08, two tiles in flight per warp
// (166 registers, 12 warps) 5.42.
// ---------------------------------------------------------------------------

constexpr int kHashWarps = 20;
constexpr int kHashThreads = 32 * kHashWarps;

__global__ void __launch_bounds__(kHashThreads, 1)
    k_hash(const SecDesc* __restrict__ secs, WorkList wl, uint64_t* __restrict__ nodes) {
  grid_dependency();
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  // This warp's tiles: a contiguous, balanced range [t0, t1).
  const uint64_t T_all = wl.n_tasks;
  const uint64_t gw = static_cast<uint64_t>(blockIdx.x) * kHashWarps + warp;
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kHashWarps;
  const uint32_t t0 = static_cast<uint32_t>(T_all * gw / nw);
  const uint32_t t1 = static_cast<uint32_t>(T_all * (gw + 1) / nw);
  if (t0 >= t1) return;
  int item = find_item(wl.begin, 0, wl.n_items, t0, lane);
  for (uint32_t t = t0; t < t1; ++t) {
    while (item + 1 < wl.n_items && __ldg(wl.begin + item + 1) <= t) ++item;
    const SecDesc* s = secs + __ldg(wl.ids + item);
    const uint8_t* base = reinterpret_cast<const uint8_t*>(
        __ldg(reinterpret_cast<const unsigned long long*>(&s->lbase)));
    const uint64_t L = __ldg(reinterpret_cast<const unsigned long long*>(&s->bytes));
    const uint64_t nch = __ldg(reinterpret_cast<const unsigned long long*>(&s->n_chunks));
    const uint32_t loc = t - __ldg(wl.begin + item);
    const uint64_t p0 = static_cast<uint64_t>(loc) * kTileBytes;
    const uint64_t c0 = p0 / kChunkBytes;
    // Bytes at or past L read as zero (the chunk's padding).
    uint4 v[2 * kSegs];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
#pragma unroll
      for (int k = 0; k < kSegs; ++k) {
        const uint64_t off = p0 + q * kChunkBytes + 512u * k + 16u * lane;
        uint4 x = make_uint4(0, 0, 0, 0);
        if (off + 16 <= L) x = ld_stream(base + off);
        else if (off < L) x = ld_small(base + off, static_cast<int>(L - off), true);
        v[q * kSegs + k] = x;
      }
    }
    uint64_t ha = fmix(kSeed ^ (c0 * 32u + lane));
    uint64_t hb = fmix(kSeed ^ ((c0 + 1) * 32u + lane));
#pragma unroll
    for (int k = 0; k < kSegs; ++k) {
      ha = absorb(ha, v[k]);
      hb = absorb(hb, v[kSegs + k]);
    }
    static_assert(kTileChunks == 2, "tile_tree2 reduces two chunks");
    const uint64_t root = tile_tree2(fmix(ha), fmix(hb), nch - c0 >= 2 ? 2 : 1, lane);
    if (lane == 0) nodes[__ldg(&s->task_begin) + loc] = root;
  }
}

// ---------------------------------------------------------------------------
// Finalisation: stream fps, record headers, verification
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint64_t stream_fp(const SecDesc& s, uint64_t* nodes, int lane) {
  const uint64_t root = s.fin_count <= kFinRegNodes ? warp_tree_regs(nodes + s.fin_begin, s.fin_count, lane)
                                             : warp_tree_inplace(nodes + s.fin_begin, s.fin_count, lane);
  return fmix(root ^ (s.bytes * kP));
}

// One warp per aligned group of 32 nodes of one stream (one reduction level).
__global__ void __launch_bounds__(kThreads)
    k_reduce_nodes(const NodeLevel* __restrict__ lv, int n_secs, uint64_t* nodes, uint32_t base,
                   uint32_t n_groups) {
  grid_dependency();
  const int lane = threadIdx.x & 31;
  const uint32_t nw = gridDim.x * kWarps;
  for (uint32_t g = blockIdx.x * kWarps + (threadIdx.x >> 5); g < n_groups; g += nw) {
    int lo = 0, hi = n_secs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(&lv[mid].dst) - base <= g) lo = mid;
      else hi = mid - 1;
    }
    const NodeLevel L = lv[lo];
    const uint32_t local = g - (L.dst - base);
    const uint32_t n = min(32u, L.count - 32u * local);
    const uint64_t v = lane < static_cast<int>(n) ? nodes[L.src + 32u * local + lane] : 0;
    const uint64_t r = warp_tree(v, static_cast<int>(n), lane);
    if (lane == 0) nodes[L.dst + local] = r;
  }
}

// Fingerprints of independent buffers (pcs_fingerprint / pcs_classify):
// warps w0, w0 + nw, ... take buffer after buffer.
__device__ __forceinline__ void finalize_hash_warps(const SecDesc* __restrict__ secs, int n_secs,
                                                    uint64_t* nodes, uint64_t* fp_out,
                                                    const uint64_t* fp_before, uint8_t* flags,
                                                    int w0, int nw) {
  const int lane = threadIdx.x & 31;
  for (int i = w0; i < n_secs; i += nw) {
    const SecDesc s = secs[i];
    const uint64_t fp = stream_fp(s, nodes, lane);
    if (lane == 0) {
      if (fp_out) fp_out[i] = fp;
      if (fp_before) flags[i] = fp != fp_before[i] ? 1 : 0;
    }
  }
}

__global__ void __launch_bounds__(kThreads)
    k_finalize_hash(const SecDesc* __restrict__ secs, int n_secs, uint64_t* nodes,
                    uint64_t* fp_out, const uint64_t* fp_before, uint8_t* flags) {
  grid_dependency();
  finalize_hash_warps(secs, n_secs, nodes, fp_out, fp_before, flags,
                      blockIdx.x * kWarps + (threadIdx.x >> 5), gridDim.x * kWarps);
}

constexpr uint32_t kMaxSmemFps = 2048;  // level-1 nodes of up to 65535 fps

// Session fp = fmix(tree(fps) ^ n): fps read with a stride of `stride`
// u64 words (the fp field of consecutive 64-byte entries).  Warp-wide.
__device__ uint64_t session_fp(const uint64_t* fps, uint32_t stride, uint32_t n, uint64_t* smem,
                               int lane) {
  const uint32_t groups = (n + 31) / 32;
  for (uint32_t g = 0; g < groups; ++g) {
    const uint32_t i = 32 * g + lane;
    const uint64_t v = i < n ? fps[static_cast<uint64_t>(i) * stride] : 0;
    const uint64_t r = warp_tree(v, static_cast<int>(min(32u, n - 32 * g)), lane);
    if (lane == 0) smem[g] = r;
  }
  __syncwarp();
  const uint64_t root = warp_tree_inplace(smem, groups, lane);
  return fmix(root ^ static_cast<uint64_t>(n));
}

// Checkpoint: fps into the section table, then header and session fp.
// Restore with verification: compare recomputed fps with the record.
// The whole block handles sessions b0, b0 + stride, ...
template <int MODE>
__device__ void finalize_sessions_block(const SecDesc* __restrict__ secs,
                                        const SessDesc* __restrict__ sess, int n_sess,
                                        const Entry* __restrict__ entries, uint64_t* nodes,
                                        uint8_t* corrupt, uint32_t* bad, int b0, int stride,
                                        uint64_t* smem, uint32_t* s_bad) {
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const uint32_t nwarps = blockDim.x >> 5;
  for (int b = b0; b < n_sess; b += stride) {
    const SessDesc S = sess[b];
    Entry* table = reinterpret_cast<Entry*>(S.record + kHeaderBytes);
    if (threadIdx.x == 0) *s_bad = 0;
    __syncthreads();
    for (uint32_t j = wib; j < S.n_sections; j += nwarps) {
      const SecDesc s = secs[S.sec_begin + j];
      uint4 ew = make_uint4(0, 0, 0, 0);  // lanes 0..3: the entry, read before the tree
      if (MODE == kModePack && lane < 4)
        ew = reinterpret_cast<const uint4*>(&entries[S.sec_begin + j])[lane];
      const uint64_t fp = stream_fp(s, nodes, lane);
      if (MODE == kModePack) {
        // Lanes 0..3 write the 64-byte entry as four 16-byte words; the fp
        // (bytes 32..39) is the first half of lane 2's word.
        if (lane == 2) {
          ew.x = static_cast<uint32_t>(fp);
          ew.y = static_cast<uint32_t>(fp >> 32);
        }
        if (lane < 4) reinterpret_cast<uint4*>(&table[j])[lane] = ew;
      } else {
        if (lane == 0 && table[j].fp != fp) atomicOr(s_bad, 1u);
      }
    }
    __syncthreads();
    if (wib == 0) {
      const uint64_t* fps = &table[0].fp;
      const uint64_t sfp = session_fp(fps, kEntryBytes / 8, S.n_sections, smem, lane);
      if (lane == 0) {
        if (MODE == kModePack) {
          uint4* h = reinterpret_cast<uint4*>(S.record);
          h[0] = make_uint4(kMagic, kVersion | (S.n_sections << 16), S.session_id, S.kind);
          h[1] = make_uint4(static_cast<uint32_t>(S.total_bytes),
                            static_cast<uint32_t>(S.total_bytes >> 32), static_cast<uint32_t>(sfp),
                            static_cast<uint32_t>(sfp >> 32));
          h[2] = make_uint4(0, 0, 0, 0);
          h[3] = make_uint4(0, 0, 0, 0);
        } else {
          const uint64_t stored = *reinterpret_cast<const uint64_t*>(S.record + 24);
          const bool broken = *s_bad != 0 || stored != sfp;
          if (corrupt) corrupt[b] = broken ? 1 : 0;
          if (broken) atomicAdd(bad, 1u);
        }
      }
    }
    if (MODE == kModePack) {
      // Zero the gap between the end of the table and the first payload.
      const uint64_t from = kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * S.n_sections;
      for (uint64_t o = from + 16u * threadIdx.x; o < S.payload_start; o += 16u * blockDim.x)
        *reinterpret_cast<uint4*>(S.record + o) = make_uint4(0, 0, 0, 0);
    }
    __syncthreads();
  }
}

// Any block size up to 512 threads (a warp per section in turn).
template <int MODE>
__global__ void __launch_bounds__(512)
    k_finalize_sessions(const SecDesc* __restrict__ secs, const SessDesc* __restrict__ sess,
                        int n_sess, const Entry* __restrict__ entries, uint64_t* nodes,
                        uint8_t* corrupt, uint32_t* bad) {
  __shared__ uint64_t smem[kMaxSmemFps];
  __shared__ uint32_t s_bad;
  // The host's descriptors of the block's first session (each warp's first
  // section and, for a checkpoint, its table entry) are brought into L1
  // while the kernel ahead on the stream drains.
  if (static_cast<int>(blockIdx.x) < n_sess) {
    const SessDesc* S0 = sess + blockIdx.x;
    const uint32_t j = threadIdx.x >> 5;
    if (j < __ldg(&S0->n_sections) && (threadIdx.x & 31) == 0) {
      const uint32_t i = __ldg(&S0->sec_begin) + j;
      prefetch_l1(secs + i);
      prefetch_l1(reinterpret_cast<const uint8_t*>(secs + i) + sizeof(SecDesc) - 1);
      if (MODE == kModePack) prefetch_l1(entries + i);
    }
  }
  grid_dependency();
  finalize_sessions_block<MODE>(secs, sess, n_sess, entries, nodes, corrupt, bad, blockIdx.x,
                                gridDim.x, smem, &s_bad);
}

// Sessions of at most 32 sections: one warp per session (lane j keeps
// section j's fp), the same outputs as finalize_sessions_block.
template <int MODE>
__global__ void __launch_bounds__(kThreads)
    k_finalize_sessions_warp(const SecDesc* __restrict__ secs, const SessDesc* __restrict__ sess,
                             int n_sess, const Entry* __restrict__ entries, uint64_t* nodes,
                             uint8_t* corrupt, uint32_t* bad) {
  const int lane = threadIdx.x & 31;
  const int nw = gridDim.x * kWarps;
  // Lane j reads section j's node range and length, all sections at once.
  // These are the host's descriptors: the warp's first session reads them
  // while the kernel ahead on the stream drains.
  SessDesc S;
  uint32_t fin_begin = 0, fin_count = 0;
  uint64_t sec_bytes = 0;
  auto load_session = [&](int b) {
    S = sess[b];
    fin_begin = fin_count = 0;
    sec_bytes = 0;
    if (lane < static_cast<int>(S.n_sections)) {
      const SecDesc* sj = secs + S.sec_begin + lane;
      fin_begin = __ldg(&sj->fin_begin);
      fin_count = __ldg(&sj->fin_count);
      sec_bytes = __ldg(reinterpret_cast<const unsigned long long*>(&sj->bytes));
    }
  };
  const int b_first = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (b_first < n_sess) load_session(b_first);
  grid_dependency();
  for (int b = b_first; b < n_sess; b += nw) {
    if (b != b_first) load_session(b);
    Entry* table = reinterpret_cast<Entry*>(S.record + kHeaderBytes);
    const int ns = static_cast<int>(S.n_sections);
    // A restore's stored fps (lane j: section j's), read once; each
    // section's tree then starts from its node loads, and a checkpoint's
    // entry is read before the tree.
    uint64_t stored = 0;
    if (MODE != kModePack && lane < ns) stored = table[lane].fp;
    uint64_t mine = 0;
    bool bad_sec = false;
    for (int j = 0; j < ns; ++j) {
      uint4 ew = make_uint4(0, 0, 0, 0);  // pack: lanes 0..3 hold the entry, read before the tree
      if (MODE == kModePack && lane < 4)
        ew = reinterpret_cast<const uint4*>(&entries[S.sec_begin + j])[lane];
      const uint32_t nb = __shfl_sync(kFull, fin_begin, j);
      const uint32_t nc = __shfl_sync(kFull, fin_count, j);
      const uint64_t by = __shfl_sync(kFull, sec_bytes, j);
      const uint64_t root = nc <= kFinRegNodes ? warp_tree_regs(nodes + nb, nc, lane)
                                               : warp_tree_inplace(nodes + nb, nc, lane);
      const uint64_t fp = fmix(root ^ (by * kP));
      if (MODE == kModePack) {
        // The fp (bytes 32..39 of the entry) is the first half of lane 2's word.
        if (lane == 2) {
          ew.x = static_cast<uint32_t>(fp);
          ew.y = static_cast<uint32_t>(fp >> 32);
        }
        if (lane < 4) reinterpret_cast<uint4*>(&table[j])[lane] = ew;
        if (lane == j) mine = fp;
      } else {
        if (lane == j) {
          mine = stored;
          bad_sec = stored != fp;
        }
      }
    }
    // Session fp = fmix(tree(fps) ^ n), the fps being the table's.
    const uint64_t sfp = fmix(warp_tree(mine, ns, lane) ^ static_cast<uint64_t>(ns));
    const bool any_bad = __any_sync(kFull, bad_sec);
    if (lane == 0) {
      if (MODE == kModePack) {
        uint4* h = reinterpret_cast<uint4*>(S.record);
        h[0] = make_uint4(kMagic, kVersion | (S.n_sections << 16), S.session_id, S.kind);
        h[1] = make_uint4(static_cast<uint32_t>(S.total_bytes),
                          static_cast<uint32_t>(S.total_bytes >> 32), static_cast<uint32_t>(sfp),
                          static_cast<uint32_t>(sfp >> 32));
        h[2] = make_uint4(0, 0, 0, 0);
        h[3] = make_uint4(0, 0, 0, 0);
      } else {
        const uint64_t stored = *reinterpret_cast<const uint64_t*>(S.record + 24);
        const bool broken = any_bad || stored != sfp;
        if (corrupt) corrupt[b] = broken ? 1 : 0;
        if (broken) atomicAdd(bad, 1u);
      }
    }
    if (MODE == kModePack) {
      // Zero the gap between the end of the table and the first payload.
      const uint64_t from = kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * S.n_sections;
      for (uint64_t o = from + 16u * lane; o < S.payload_start; o += 16u * 32)
        *reinterpret_cast<uint4*>(S.record + o) = make_uint4(0, 0, 0, 0);
    }
  }
}

// Small calls in one launch: the streaming pass, then the finalisation by
// the last block to finish (an atomic ticket; no block waits for another).
// `ticket` is zero on entry and reset by the last block.
template <int MODE>
__global__ void __launch_bounds__(kThreads, 2)
    k_small(const SecDesc* __restrict__ secs, WorkList wl, int glog2, uint64_t* nodes,
            uint32_t* err, uint32_t* ticket, int n_items, const SessDesc* __restrict__ sess,
            const Entry* __restrict__ entries, uint64_t* fp_out, const uint64_t* fp_before,
            uint8_t* flags, uint32_t* bad) {
  grid_dependency();
  __shared__ SecDesc sdesc[kWarps];
  __shared__ uint64_t smem[64];  // up to 2048 sections per session
  __shared__ uint32_t s_bad;
  __shared__ bool s_last;
  run_stream_tasks<MODE>(secs, wl, glog2, nodes, err, sdesc);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (MODE == kModeHash) {
    finalize_hash_warps(secs, n_items, nodes, fp_out, fp_before, flags, threadIdx.x >> 5, kWarps);
  } else {
    finalize_sessions_block<MODE>(secs, sess, n_items, entries, nodes, nullptr, bad, 0, 1, smem,
                                  &s_bad);
  }
  if (threadIdx.x == 0) *ticket = 0;
}

// ---------------------------------------------------------------------------
// Relevance score and top-k
// ---------------------------------------------------------------------------

// Order-preserving map float -> uint32 (-0 ranks as +0, NaN lowest).
__device__ __forceinline__ uint32_t ord32(float s) {
  if (isnan(s)) return 0u;
  if (s == 0.f) s = 0.f;
  const uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Digits of the 64-bit ranking key of the global threshold, most significant
// first: 11, 11 and 10 bits of ord32(score), then the same of the position.
__device__ __forceinline__ int gdigit_bits(int pass) { return pass % 3 == 2 ? 10 : 11; }
__device__ __forceinline__ int gdigit_shift(int pass) {
  return pass == 0 ? 53 : pass == 1 ? 42 : pass == 2 ? 32 : pass == 3 ? 21 : pass == 4 ? 10 : 0;
}

// The digit choice of one pass, by one warp, from the summed histograms
// (staged in shared memory): scanning digits from the top, the first whose
// bytes overrun the budget left is fixed into the prefix; if it holds a
// single key, or it was the last digit, that key is the first that does not
// fit and the threshold is set.
template <bool UNIFORM>
__device__ void gselect_pick(GState* st, int pass, uint64_t ubytes, const uint32_t* ch,
                             const unsigned long long* wh) {
  const int lane = threadIdx.x & 31;
  const int bits = gdigit_bits(pass), shift = gdigit_shift(pass);
  const int top = (1 << bits) - 1, per = (1 << bits) / 32;  // lane l: bins top-per*l ...
  auto weight = [&](int bin) -> uint64_t {
    return UNIFORM ? static_cast<uint64_t>(ch[bin]) * ubytes : static_cast<uint64_t>(wh[bin]);
  };
  uint64_t local = 0;
  for (int j = 0; j < per; ++j) local += weight(top - per * lane - j);
  uint64_t incl = local;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  const uint64_t R = __ldcg(&st->remaining);
  const unsigned hit = __ballot_sync(kFull, incl > R);
  if (hit == 0) {  // every candidate fits (only when the whole population does)
    if (lane == 0) {
      st->threshold = 0;
      st->done = 1;
    }
    return;
  }
  if (lane != __ffs(hit) - 1) return;
  const uint64_t prefix = __ldcg(&st->prefix), mask = __ldcg(&st->mask);
  uint64_t cum = incl - local;
  for (int j = 0; j < per; ++j) {
    const int bin = top - per * lane - j;
    const uint64_t w = weight(bin);
    if (cum + w > R) {
      const uint64_t np = prefix | (static_cast<uint64_t>(bin) << shift);
      const uint64_t nm = mask | (static_cast<uint64_t>(top) << shift);
      st->prefix = np;
      st->mask = nm;
      st->remaining = R - cum;
      if (ch[bin] == 1u || shift == 0) {
        st->threshold = np | ~nm;
        st->done = 1;
      }
      return;
    }
    cum += w;
  }
}

// End of a histogram pass, by every block: add the block's bins (ch, wh in
// shared memory) to the global ones; the last block to finish (atomic
// ticket) stages the sums in the same shared arrays, picks the digit and
// clears the global bins for the next pass.
template <bool UNIFORM>
__device__ void gpass_finish(GState* st, int pass, uint64_t ubytes, uint32_t* ch,
                             unsigned long long* wh, bool* s_last, bool pick = true) {
  const int nb = 1 << gdigit_bits(pass);
  __syncthreads();
  for (int i = threadIdx.x; i < nb; i += blockDim.x) {
    if (ch[i]) atomicAdd(&st->chist[i], ch[i]);
    if (!UNIFORM && wh[i]) atomicAdd(reinterpret_cast<unsigned long long*>(&st->whist[i]), wh[i]);
  }
  if (!pick) return;  // a part of a split population: the host sums and picks
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *s_last = atomicAdd(&st->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!*s_last) return;
  __threadfence();
  for (int i = threadIdx.x; i < nb; i += blockDim.x) {
    ch[i] = __ldcg(&st->chist[i]);
    if (!UNIFORM) wh[i] = __ldcg(reinterpret_cast<const unsigned long long*>(&st->whist[i]));
    st->chist[i] = 0;
    st->whist[i] = 0;
  }
  __syncthreads();
  if (threadIdx.x < 32) gselect_pick<UNIFORM>(st, pass, ubytes, ch, wh);
  if (threadIdx.x == 0) st->ticket = 0;
}

__device__ __forceinline__ float elem(uint32_t bits16, bool bf16) {
  return bf16 ? __uint_as_float(bits16 << 16)
              : __half2float(__ushort_as_half(static_cast<unsigned short>(bits16)));
}

// Accumulate the key terms (q.k and k.k) of the 8 elements of one 16-byte
// segment, ascending element order, with separately rounded products and
// sums.  (q.q is the same for every key of a bank: accum8_query.)
__device__ __forceinline__ void accum8_key(uint4 q, uint4 k, bool bf16, float& sd, float& sk) {
  const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
  const uint32_t kw[4] = {k.x, k.y, k.z, k.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t qb = (qw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
    const uint32_t kb = (kw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
    const float qe = elem(qb, bf16), ke = elem(kb, bf16);
    sd = __fadd_rn(sd, __fmul_rn(qe, ke));
    sk = __fadd_rn(sk, __fmul_rn(ke, ke));
  }
}

// The query's own term, accumulated in the same lane order.
__device__ __forceinline__ void accum8_query(uint4 q, bool bf16, float& sq) {
  const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float qe = elem((qw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu, bf16);
    sq = __fadd_rn(sq, __fmul_rn(qe, qe));
  }
}

__device__ __forceinline__ float lane_tree_sum(float v) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) v = __fadd_rn(v, __shfl_down_sync(kFull, v, d));
  return v;
}

constexpr int kScoreIlp = 4;  // entries a warp scores at once (a multiple of 4)

// Element i (0..7) of a 16-byte segment as fp32 (exact conversion).
template <int DT>  // 1 = bf16, 0 = fp16
__device__ __forceinline__ float seg_elem(const uint4& v, int i) {
  const uint32_t w = (i >> 1) == 0 ? v.x : (i >> 1) == 1 ? v.y : (i >> 1) == 2 ? v.z : v.w;
  if (DT == 1) return __uint_as_float((i & 1) ? (w & 0xFFFF0000u) : (w << 16));
  return __half2float(__ushort_as_half(static_cast<unsigned short>((i & 1) ? (w >> 16) : (w & 0xFFFFu))));
}

// Each warp scores a contiguous, balanced range of entries, kScoreIlp at a
// time, following a cursor over the banks (one search per warp).  SPL = 16-byte
// key segments per lane (D <= 256 * SPL); DT = key type (1 bf16, 0 fp16).
// The bank's query is held in registers as fp32, with |q| computed once per
// bank in the same fixed order; every key load of the kScoreIlp entries is
// issued before any arithmetic.
template <int SPL, int DT, int HM>
__device__ __forceinline__ void score_range(const BankDesc* __restrict__ banks, int n_banks,
                                            uint64_t n_entries, float* __restrict__ scores,
                                            bool hist, uint32_t* s_cnt, unsigned long long* s_w) {
  const int lane = threadIdx.x & 31;
  const uint64_t gw = static_cast<uint64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kWarps;
  const uint64_t e_begin = n_entries * gw / nw, e_end = n_entries * (gw + 1) / nw;
  if (e_begin >= e_end) return;
  // The last bank starting at or before e_begin, searched by the whole warp
  // (32 probes a round, as in find_item).
  int b = 0;
  {
    int span = n_banks;
    while (span > 1) {
      const int step = (span + 31) >> 5;
      const int i = b + lane * step;
      const bool le = i < b + span && __ldg(&banks[i].entry_begin) <= e_begin;
      const unsigned m = __ballot_sync(kFull, le);  // lane 0 probes b: never empty
      const int last = 31 - __clz(m);
      b += last * step;
      span = min(step, span - last * step);
    }
  }
  int qbank = -1, segs = 0;
  float qnorm = 0.f;
  float qf[SPL][8];
#pragma unroll
  for (int j = 0; j < SPL; ++j)
#pragma unroll
    for (int i = 0; i < 8; ++i) qf[j][i] = 0.f;
  for (uint64_t e0 = e_begin; e0 < e_end; e0 += kScoreIlp) {
    // Entries of this round must share one bank to use the cached query;
    // a round stops early at a bank boundary.
    while (b + 1 < n_banks && __ldg(&banks[b + 1].entry_begin) <= e0) ++b;
    const BankDesc& B = banks[b];
    if (b != qbank) {  // warp-uniform: load the query, compute |q|
      segs = B.D / 8;
      const uint4* qrow = reinterpret_cast<const uint4*>(B.query);
      float sq = 0.f;
#pragma unroll
      for (int j = 0; j < SPL; ++j) {
        const int t = lane + 32 * j;
        const uint4 qv = t < segs ? __ldg(qrow + t) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          qf[j][i] = seg_elem<DT>(qv, i);
          if (t < segs) sq = __fadd_rn(sq, __fmul_rn(qf[j][i], qf[j][i]));
        }
      }
      // The tree's full sum is lane 0's; every lane finalises an entry below.
      qnorm = __shfl_sync(kFull, __fsqrt_rn(lane_tree_sum(sq)), 0);
      qbank = b;
    }
    const uint64_t bank_end = b + 1 < n_banks ? __ldg(&banks[b + 1].entry_begin) : n_entries;
    const uint64_t lim = min(static_cast<unsigned long long>(e_end), static_cast<unsigned long long>(bank_end));
    const int cnt = static_cast<int>(min(static_cast<uint64_t>(kScoreIlp), lim - e0));
    const uint8_t* kbase = reinterpret_cast<const uint8_t*>(B.keys) +
                           (e0 - B.entry_begin) * static_cast<uint64_t>(B.D) * 2;
    uint4 kv[kScoreIlp][SPL];
#pragma unroll
    for (int q = 0; q < kScoreIlp; ++q)
#pragma unroll
      for (int j = 0; j < SPL; ++j) {
        const int t = lane + 32 * j;
        kv[q][j] = (q < cnt && t < segs) ? ld_stream(kbase + static_cast<uint64_t>(q) * B.D * 2 + 16 * t)
                                         : make_uint4(0, 0, 0, 0);
      }
    // v[2q] = q.k and v[2q+1] = k.k of entry q, per lane: both chains step
    // together in paired fp32 operations (each half rounded on its own, as
    // the separate multiply and add).
    static_assert(kScoreIlp % 4 == 0, "the transposed tree reduces groups of 4 entries x 2 sums");
    float v[2 * kScoreIlp];
#pragma unroll
    for (int q = 0; q < kScoreIlp; ++q) {
      float2 acc = make_float2(0.f, 0.f);
#pragma unroll
      for (int j = 0; j < SPL; ++j) {
        if (lane + 32 * j < segs) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float ke = seg_elem<DT>(kv[q][j], i);
            acc = __fadd2_rn(acc, __fmul2_rn(make_float2(qf[j][i], ke), make_float2(ke, ke)));
          }
        }
      }
      v[2 * q] = acc.x;
      v[2 * q + 1] = acc.y;
    }
    // The lane tree (s[l] += s[l + d], d = 1 .. 16) of the eight sums of
    // each group of four entries at once: at d = 1, 2, 4 each lane keeps half
    // of its values and adds its partner's copy of them, so lane l ends with
    // sum 4*(l&1) + 2*(l>>1&1) + (l>>2&1); d = 8, 16 finish it.  Addition is
    // commutative, so every partial sum is the one the plain tree forms.
    const bool b0 = lane & 1, b1 = lane & 2, b2 = lane & 4;
#pragma unroll
    for (int g = 0; g < kScoreIlp / 4; ++g) {
      const float* vg = v + 8 * g;
      float w4[4], w2[2];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float give = b0 ? vg[i] : vg[4 + i];
        w4[i] = __fadd_rn(b0 ? vg[4 + i] : vg[i], __shfl_xor_sync(kFull, give, 1));
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const float give = b1 ? w4[i] : w4[2 + i];
        w2[i] = __fadd_rn(b1 ? w4[2 + i] : w4[i], __shfl_xor_sync(kFull, give, 2));
      }
      float w1 = __fadd_rn(b2 ? w2[1] : w2[0], __shfl_xor_sync(kFull, b2 ? w2[0] : w2[1], 4));
      w1 = __fadd_rn(w1, __shfl_xor_sync(kFull, w1, 8));
      w1 = __fadd_rn(w1, __shfl_xor_sync(kFull, w1, 16));
      // Lanes 0..3 hold q.k of entry 4g + 2*(l&1) + (l>>1&1); lane l + 4 its k.k.
      const float kk = __shfl_down_sync(kFull, w1, 4);
      const int q = 4 * g + 2 * (lane & 1) + ((lane >> 1) & 1);
      if (lane < 4 && q < cnt) {
        const float den = __fmul_rn(qnorm, __fsqrt_rn(kk));
        const float sc = den == 0.f ? 0.f : __fdiv_rn(w1, den);
        scores[e0 + q] = sc;
        if (HM && hist) {
          const uint32_t d = ord32(sc) >> 21;  // key bits 63..53
          atomicAdd(&s_cnt[d], 1u);
          if (HM == 2) atomicAdd(&s_w[d], static_cast<unsigned long long>(B.entry_bytes));
        }
      }
    }
    e0 = e0 + cnt - kScoreIlp;  // the loop adds kScoreIlp: next round starts at e0 + cnt
  }
}

// HM (global threshold): 0 none; 1 / 2 also histogram the top 11 key bits of
// every score (2: weighted by the bank's entry bytes) and pick the first digit.
template <int SPL, int DT, int HM>
__global__ void __launch_bounds__(kThreads)
    k_score_fixed(const BankDesc* __restrict__ banks, int n_banks, uint64_t n_entries,
                  float* __restrict__ scores, GHist gh) {
  grid_dependency();
  __shared__ uint32_t s_cnt[HM ? kGBins : 1];
  __shared__ unsigned long long s_w[HM == 2 ? kGBins : 1];
  __shared__ bool s_last;
  const bool hist = HM && !__ldcg(&gh.st->done);  // the same for every block
  if (hist) {
    for (int i = threadIdx.x; i < kGBins; i += kThreads) {
      s_cnt[i] = 0;
      if (HM == 2) s_w[i] = 0;
    }
    __syncthreads();
  }
  score_range<SPL, DT, HM>(banks, n_banks, n_entries, scores, hist, s_cnt, s_w);
  if (hist) gpass_finish<HM == 1>(gh.st, 0, gh.uniform_bytes, s_cnt, s_w, &s_last);
}


// Any key width or a mix of key types: the query is re-read per entry.
__global__ void __launch_bounds__(kThreads)
    k_score_any(const BankDesc* __restrict__ banks, int n_banks, uint64_t n_entries,
                float* __restrict__ scores) {
  grid_dependency();
  const int lane = threadIdx.x & 31;
  const uint64_t gw = static_cast<uint64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kWarps;
  const uint64_t e_begin = n_entries * gw / nw, e_end = n_entries * (gw + 1) / nw;
  if (e_begin >= e_end) return;
  int b = 0;
  {
    int lo = 0, hi = n_banks - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(&banks[mid].entry_begin) <= e_begin) lo = mid;
      else hi = mid - 1;
    }
    b = lo;
  }
  int qbank = -1;
  float qnorm = 0.f;
  for (uint64_t e = e_begin; e < e_end; ++e) {
    while (b + 1 < n_banks && __ldg(&banks[b + 1].entry_begin) <= e) ++b;
    const BankDesc& B = banks[b];
    const bool bf16 = B.is_bf16 != 0;
    const uint4* qrow = reinterpret_cast<const uint4*>(B.query);
    if (b != qbank) {
      float sq = 0.f;
      for (int t = lane; t < B.D / 8; t += 32) accum8_query(__ldg(qrow + t), bf16, sq);
      qnorm = __fsqrt_rn(lane_tree_sum(sq));
      qbank = b;
    }
    const uint8_t* krow = reinterpret_cast<const uint8_t*>(B.keys) +
                          (e - B.entry_begin) * static_cast<uint64_t>(B.D) * 2;
    float sd = 0.f, sk = 0.f;
    for (int t = lane; t < B.D / 8; t += 32)
      accum8_key(__ldg(qrow + t), ld_stream(krow + 16 * t), bf16, sd, sk);
    const float d = lane_tree_sum(sd);
    const float kk = lane_tree_sum(sk);
    if (lane == 0) {
      const float den = __fmul_rn(qnorm, __fsqrt_rn(kk));
      scores[e] = den == 0.f ? 0.f : __fdiv_rn(d, den);
    }
  }
}


// Exclusive block scan of a 0/1 flag; returns the rank, *total = sum.
__device__ __forceinline__ uint32_t block_rank(bool f, uint32_t* warp_cnt, uint32_t* total) {
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const unsigned m = __ballot_sync(kFull, f);
  const uint32_t in_warp = __popc(m & ((1u << lane) - 1u));
  if (lane == 0) warp_cnt[wib] = __popc(m);
  __syncthreads();
  uint32_t before = 0, sum = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const uint32_t c = warp_cnt[w];
    if (w < wib) before += c;
    sum += c;
  }
  __syncthreads();
  *total = sum;
  return before + in_warp;
}

// Exclusive block scan of one uint32 per thread; *total = block sum.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* warp_sum,
                                                    uint32_t* total) {
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  if (lane == 31) warp_sum[wib] = incl;
  __syncthreads();
  uint32_t before = 0, sum = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const uint32_t c = warp_sum[w];
    if (w < wib) before += c;
    sum += c;
  }
  __syncthreads();
  *total = sum;
  return before + incl - v;
}

// The digit of one radix-select pass (warp 0, histogram in shared memory):
// scanning bins from the top, the first whose running count reaches the
// rank still wanted is fixed into the prefix.
__device__ __forceinline__ void topk_pick(const uint32_t* hist, int shift, uint32_t* s_prefix,
                                          uint32_t* s_mask, uint32_t* s_remaining) {
  const int lane = threadIdx.x & 31;
  // Lane l covers bins 255-8l .. 248-8l (descending).
  uint32_t local = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) local += hist[255 - 8 * lane - j];
  uint32_t incl = local;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  const uint32_t remaining = *s_remaining;
  const unsigned hit = __ballot_sync(kFull, incl >= remaining);
  const int first = __ffs(hit) - 1;  // remaining <= count, so hit != 0
  if (lane == first) {
    uint32_t cum = incl - local;
    for (int j = 0; j < 8; ++j) {
      const int bin = 255 - 8 * lane - j;
      if (cum + hist[bin] >= remaining) {
        *s_prefix |= static_cast<uint32_t>(bin) << shift;
        *s_mask |= 0xFFu << shift;
        *s_remaining = remaining - cum;
        break;
      }
      cum += hist[bin];
    }
  }
}

constexpr int kTopkPer = 16;                    // entries a thread holds
constexpr int kTopkReg = kThreads * kTopkPer;   // banks up to this size stay in registers

// One bank of at most kTopkReg entries, 0 < k < n: thread t holds the keys of
// entries [16 t, 16 t + 16) for all four passes; the kept entries (every key
// above the threshold, then the first ones equal to it) are ranked with two
// block scans and written in ascending index order.
__device__ void topk_bank_reg(const float* __restrict__ sc, int n, int k, int32_t* __restrict__ out,
                              uint32_t* hist, uint32_t* warp_sum, uint32_t* s_prefix,
                              uint32_t* s_mask, uint32_t* s_remaining) {
  const int base = threadIdx.x * kTopkPer;
  uint32_t u[kTopkPer];
#pragma unroll
  for (int j = 0; j < kTopkPer; ++j) u[j] = base + j < n ? ord32(__ldg(sc + base + j)) : 0u;
  if (threadIdx.x == 0) {
    *s_prefix = 0;
    *s_mask = 0;
    *s_remaining = static_cast<uint32_t>(k);
  }
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = threadIdx.x; i < 256; i += kThreads) hist[i] = 0;
    __syncthreads();
    const uint32_t prefix = *s_prefix, mask = *s_mask;
#pragma unroll
    for (int j = 0; j < kTopkPer; ++j)
      if (base + j < n && (u[j] & mask) == prefix) atomicAdd(&hist[(u[j] >> shift) & 255u], 1u);
    __syncthreads();
    if (threadIdx.x < 32) topk_pick(hist, shift, s_prefix, s_mask, s_remaining);
    __syncthreads();
  }
  const uint32_t t = *s_prefix, take_eq = *s_remaining;
  uint32_t gt = 0, eq = 0;
#pragma unroll
  for (int j = 0; j < kTopkPer; ++j) {
    if (base + j < n) {
      gt |= static_cast<uint32_t>(u[j] > t) << j;
      eq |= static_cast<uint32_t>(u[j] == t) << j;
    }
  }
  uint32_t total;
  uint32_t r = block_excl_scan(__popc(eq), warp_sum, &total);  // equal keys before this thread's
  uint32_t keep = gt;
  for (uint32_t m = eq; m; m &= m - 1) {
    if (r >= take_eq) break;
    keep |= m & (~m + 1u);
    ++r;
  }
  uint32_t pos = block_excl_scan(__popc(keep), warp_sum, &total);
  for (uint32_t m = keep; m; m &= m - 1) out[pos++] = base + __ffs(m) - 1;
  __syncthreads();
}

__global__ void __launch_bounds__(kThreads)
    k_topk(const BankDesc* __restrict__ banks, int n_banks, const float* __restrict__ scores,
           int32_t* __restrict__ kept_idx) {
  grid_dependency();
  __shared__ uint32_t hist[256];
  __shared__ uint32_t warp_cnt[kWarps];
  __shared__ uint32_t s_prefix, s_mask, s_remaining;
  const int wib = threadIdx.x >> 5;
  for (int b = blockIdx.x; b < n_banks; b += gridDim.x) {
    const BankDesc B = banks[b];
    const int n = B.n, k = B.k;
    const float* sc = scores + B.entry_begin;
    int32_t* out = kept_idx + B.kept_begin;
    if (k >= n) {
      for (int i = threadIdx.x; i < n; i += kThreads) out[i] = i;
      continue;
    }
    if (k <= 0) continue;
    if (n <= kTopkReg) {
      topk_bank_reg(sc, n, k, out, hist, warp_cnt, &s_prefix, &s_mask, &s_remaining);
      continue;
    }
    if (threadIdx.x == 0) {
      s_prefix = 0;
      s_mask = 0;
      s_remaining = static_cast<uint32_t>(k);
    }
    __syncthreads();
    // Radix select, most significant byte first: the k-th largest ord32.
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = threadIdx.x; i < 256; i += kThreads) hist[i] = 0;
      __syncthreads();
      const uint32_t prefix = s_prefix, mask = s_mask;
      for (int i = threadIdx.x; i < n; i += kThreads) {
        const uint32_t u = ord32(sc[i]);
        if ((u & mask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (wib == 0) topk_pick(hist, shift, &s_prefix, &s_mask, &s_remaining);
      __syncthreads();
    }
    // Keep every entry above the threshold and the first `remaining` equal
    // to it, in ascending index order.
    const uint32_t t = s_prefix, take_eq = s_remaining;
    uint32_t eq_seen = 0, written = 0;
    for (int start = 0; start < n; start += kThreads) {
      const int i = start + threadIdx.x;
      const uint32_t u = i < n ? ord32(sc[i]) : 0u;
      const bool gt = i < n && u > t;
      const bool eq = i < n && u == t;
      uint32_t eq_total, kept_total;
      const uint32_t eq_rank = block_rank(eq, warp_cnt, &eq_total);
      const bool keep = gt || (eq && eq_seen + eq_rank < take_eq);
      const uint32_t pos = block_rank(keep, warp_cnt, &kept_total);
      if (keep && written + pos < static_cast<uint32_t>(k)) out[written + pos] = i;
      eq_seen += eq_total;
      written += kept_total;
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// One relevance threshold across all banks under a byte budget
//
// The entry at bank-major position i ranks by
//   key(i) = ord32(score_i) << 32 | (0xFFFFFFFF - i)
// (score descending, then bank, then index ascending; unique keys).  The kept
// set is the longest prefix of the descending key order whose entry bytes
// fit the budget: every key above the key of the first entry that does not
// fit.  That key is found most significant digit first, each pass summing
// the bytes (not the count) of the candidate keys per digit and picking the
// digit where the budget runs out.  The first pass rides on the score kernel
// (its last block, by atomic ticket, picks); k_gfinish runs the rest.
// k_gselect bins one pass of a part of a population split over processes;
// the host sums the parts' bins and picks.
// ---------------------------------------------------------------------------

// The bank holding entry i: the last bank in [lo, hi] whose first entry is
// <= i (empty banks share their successor's first entry and come before it).
__device__ __forceinline__ int gbank(const uint64_t* __restrict__ ebeg, int lo, int hi,
                                     uint64_t i) {
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(ebeg + mid) <= i) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

template <bool UNIFORM>
__global__ void __launch_bounds__(kThreads) k_gselect(GPlan p, int pass) {
  __shared__ uint32_t ch[kGBins];
  __shared__ unsigned long long wh[UNIFORM ? 1 : kGBins];
  __shared__ bool s_last;
  GState* st = p.st;
  if (__ldcg(&st->done)) return;  // the same for every block of the launch
  const int shift = gdigit_shift(pass);
  const uint32_t nb = 1u << gdigit_bits(pass);
  const uint64_t prefix = __ldcg(&st->prefix), mask = __ldcg(&st->mask);
  for (uint32_t i = threadIdx.x; i < nb; i += kThreads) {
    ch[i] = 0;
    if (!UNIFORM) wh[i] = 0;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  for (int t = blockIdx.x; t < p.tiles; t += gridDim.x) {
    const uint64_t start = static_cast<uint64_t>(t) * kGTile;
    const uint64_t end = start + kGTile < p.entries ? start + kGTile : p.entries;
    int b = p.tile_bank[t];
    const int hi = p.tile_bank[t + 1];
    // Every load of the tile in flight before any is used.
    constexpr int kPer = kGTile / kThreads;
    float sv[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const uint64_t i = start + static_cast<uint64_t>(j) * kThreads + threadIdx.x;
      sv[j] = i < end ? __ldg(p.scores + i) : 0.f;
    }
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const uint64_t i = start + static_cast<uint64_t>(j) * kThreads + threadIdx.x;
      uint32_t d = kGBins;  // not a candidate
      if (i < end) {
        const uint64_t key =
            (static_cast<uint64_t>(ord32(sv[j])) << 32) | (0xFFFFFFFFull - (p.pos_base + i));
        if ((key & mask) == prefix) d = static_cast<uint32_t>(key >> shift) & (nb - 1);
      }
      if (UNIFORM) {
        // Lanes with the same digit add once (the hot digits are few).
        const unsigned same = __match_any_sync(kFull, d);
        if (d < kGBins && lane == __ffs(same) - 1) atomicAdd(&ch[d], __popc(same));
      } else if (d < kGBins) {
        b = gbank(p.ebeg, b, hi, i);
        atomicAdd(&ch[d], 1u);
        atomicAdd(&wh[d], static_cast<unsigned long long>(__ldg(p.ebytes + b)));
      }
    }
  }
  gpass_finish<UNIFORM>(st, pass, p.uniform_bytes, ch, wh, &s_last, !p.local);
}


// ---------------------------------------------------------------------------
// The rest of the global threshold in one cooperative launch (k_gfinish):
// the digit passes after the first and the compaction.  Its blocks are all
// resident at once and meet at grid barriers; the last block to arrive makes
// the digit choice from the summed bins before it releases the others.
//
//   pass 0 (only when the score kernel could not take it): bins of the top
//     digit of every key;
//   the first full scan: keys above the digits fixed so far are kept for
//     sure and counted per tile; keys inside them (the candidates) are
//     binned by the next digit and stored in their 512-entry unit's slots;
//   later passes bin the candidates only;
//   once the threshold is known, the kept candidates join their tiles'
//   counts; each block sums the counts before its contiguous tile range and
//   writes the kept indices and bank offsets of its tiles in order.
// ---------------------------------------------------------------------------

// One block's copy of the select state.
struct GLocal {
  uint64_t prefix, mask, remaining, threshold;
  uint32_t done;
};

__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Bounded wait (one thread) until *p >= k, read with acquire semantics;
// false if about kWaitCycles of SM clock passed first.
__device__ __forceinline__ bool wait_flag_geq(const uint32_t* p, uint32_t k) {
  const long long t0 = clock64();
  while (ld_acquire(p) < k) {
    if (clock64() - t0 > kWaitCycles) return false;
    __nanosleep(20);
  }
  return true;
}

// Bounded grid barrier number k (1, 2, ...) of a cooperative launch.  The
// arrival count only grows (barrier k is full at k x blocks); the last block
// to arrive runs `last` (every thread of it), then publishes k.  A block that
// waits past kWaitCycles sets the timeout bit and returns false; the others
// then give up at their next barrier.
template <typename F>
__device__ bool grid_barrier(GState* st, uint32_t* err, uint32_t k, bool* s_flag, F&& last) {
  __syncthreads();
  if (threadIdx.x == 0) *s_flag = atom_add_acq_rel(&st->bar_count, 1u) == k * gridDim.x - 1;
  __syncthreads();
  if (*s_flag) {  // the last block: everybody else's writes are visible
    last();
    __syncthreads();
    if (threadIdx.x == 0) st_release(&st->bar_gen, k);
    return true;  // *s_flag stays set until the next barrier rewrites it
  }
  __syncthreads();  // every thread has read *s_flag
  if (threadIdx.x == 0) {
    const bool ok = wait_flag_geq(&st->bar_gen, k);
    if (!ok) atomicOr(err, kDevErrTimeout);
    *s_flag = ok;
  }
  __syncthreads();
  return *s_flag;
}

// Inclusive block scan of one uint64 per thread.
__device__ __forceinline__ uint64_t block_incl_scan64(uint64_t v, uint64_t* warp_sum) {
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  uint64_t incl = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  if (lane == 31) warp_sum[wib] = incl;
  __syncthreads();
  uint64_t before = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w)
    if (w < wib) before += warp_sum[w];
  __syncthreads();
  return before + incl;
}

// The digit choice of a pass from the summed bins, by the whole block:
// thread t holds the bins top - per*t - j (j < per), highest digits first;
// the first thread whose running bytes overrun the budget left finds the
// digit, as in gselect_pick.
template <bool UNIFORM>
__device__ void gpick_block(GLocal* s, int pass, uint64_t ubytes, const uint32_t* gc,
                            const unsigned long long* gw, uint64_t* scan64) {
  const int bits = gdigit_bits(pass), shift = gdigit_shift(pass);
  const int nb = 1 << bits, top = nb - 1, per = nb / kThreads;
  uint32_t cn[kGBins / kThreads];
  uint64_t wt[kGBins / kThreads];
  uint64_t local = 0;
#pragma unroll
  for (int j = 0; j < kGBins / kThreads; ++j) {
    cn[j] = 0;
    wt[j] = 0;
    if (j < per) {
      const int bin = top - per * static_cast<int>(threadIdx.x) - j;
      cn[j] = __ldcg(gc + bin);
      wt[j] = UNIFORM ? static_cast<uint64_t>(cn[j]) * ubytes
                      : static_cast<uint64_t>(__ldcg(gw + bin));
      local += wt[j];
    }
  }
  const uint64_t incl = block_incl_scan64(local, scan64);
  const uint64_t R = s->remaining;
  const int fit = __syncthreads_count(incl <= R);
  if (fit == kThreads) {  // every candidate fits (only when the whole population does)
    if (threadIdx.x == 0) {
      s->threshold = 0;
      s->done = 1;
    }
  } else if (static_cast<int>(threadIdx.x) == fit) {
    uint64_t cum = incl - local;
#pragma unroll
    for (int j = 0; j < kGBins / kThreads; ++j) {
      if (j < per && cum + wt[j] > R) {
        const int bin = top - per * static_cast<int>(threadIdx.x) - j;
        const uint64_t np = s->prefix | (static_cast<uint64_t>(bin) << shift);
        const uint64_t nm = s->mask | (static_cast<uint64_t>(top) << shift);
        s->prefix = np;
        s->mask = nm;
        s->remaining = R - cum;
        if (cn[j] == 1u || shift == 0) {
          s->threshold = np | ~nm;
          s->done = 1;
        }
        break;
      }
      cum += wt[j];
    }
  }
  __syncthreads();
}

// The bins of pass `pass`: the state's own for the first pass this launch
// bins (zero at launch), a scratch set (zeroed here) for the later ones.
__device__ __forceinline__ uint32_t* gbins_c(const GPlan& p, int pass, int first) {
  return pass == first ? p.st->chist : p.hb[pass].c;
}
__device__ __forceinline__ unsigned long long* gbins_w(const GPlan& p, int pass, int first) {
  return reinterpret_cast<unsigned long long*>(pass == first ? p.st->whist : p.hb[pass].w);
}

// Add a block's bins to the summed ones.
template <bool UNIFORM>
__device__ __forceinline__ void gbins_add(const uint32_t* ch, const unsigned long long* wh, int nb,
                                          uint32_t* gc, unsigned long long* gw) {
  __syncthreads();
  for (int i = threadIdx.x; i < nb; i += kThreads) {
    if (ch[i]) atomicAdd(gc + i, ch[i]);
    if (!UNIFORM && wh[i]) atomicAdd(gw + i, wh[i]);
  }
}

// Bin digit d (kGBins: not a candidate) with the given weight.  Uniform
// weights: every lane of the warp calls it and lanes with the same digit add
// once (the hot digits are few).
template <bool UNIFORM>
__device__ __forceinline__ void gbin(uint32_t* ch, unsigned long long* wh, uint32_t d,
                                     uint64_t bytes) {
  if (UNIFORM) {
    const unsigned same = __match_any_sync(kFull, d);
    if (d < kGBins && (threadIdx.x & 31) == __ffs(same) - 1) atomicAdd(&ch[d], __popc(same));
  } else if (d < kGBins) {
    atomicAdd(&ch[d], 1u);
    atomicAdd(&wh[d], static_cast<unsigned long long>(bytes));
  }
}

// Entries of tile t handled by this thread: warp w takes the 512 entries
// from t * kGTile + 512 w (its unit), lane l the 16 entries from 16 l of them.
constexpr int kGPer = kGTile / kThreads;
constexpr int kGUnit = 32 * kGPer;
static_assert(kGPer == 16, "tile layout: 16 entries per thread");

__device__ __forceinline__ uint64_t glane0(int t) {
  return static_cast<uint64_t>(t) * kGTile + (threadIdx.x >> 5) * kGUnit + (threadIdx.x & 31) * kGPer;
}

// The 16 scores from entry i0 (zero past `end`): four 16-byte loads when the
// run is whole and the scores are 16-byte aligned.
__device__ __forceinline__ void gload(const GPlan& p, uint64_t i0, uint64_t end, float (&sc)[kGPer]) {
  if (p.vec && i0 + kGPer <= end) {
    const float4* v = reinterpret_cast<const float4*>(p.scores + i0);
#pragma unroll
    for (int q = 0; q < kGPer / 4; ++q) {
      const float4 x = __ldg(v + q);
      sc[4 * q] = x.x;
      sc[4 * q + 1] = x.y;
      sc[4 * q + 2] = x.z;
      sc[4 * q + 3] = x.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < kGPer; ++j) sc[j] = i0 + j < end ? __ldg(p.scores + i0 + j) : 0.f;
  }
}

__device__ __forceinline__ uint64_t gkey_of(float sc, uint64_t pos) {
  return (static_cast<uint64_t>(ord32(sc)) << 32) | (0xFFFFFFFFull - pos);
}

// Exclusive warp scan of one uint32 per lane; *total = warp sum.
__device__ __forceinline__ uint32_t warp_excl_scan(uint32_t v, uint32_t* total) {
  const int lane = threadIdx.x & 31;
  uint32_t incl = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t o = __shfl_up_sync(kFull, incl, d);
    if (lane >= d) incl += o;
  }
  *total = __shfl_sync(kFull, incl, 31);
  return incl - v;
}

// The bank of entry i of a tile whose entries lie in banks lo .. hi, with
// its first entry and the next bank's.  Every lane of the warp calls it.
// When the tile touches at most 31 banks, lane k holds the first entry of
// bank lo + k and the search runs over the warp's registers.
__device__ __forceinline__ int gbank_tile(const GPlan& p, int lo, int hi, uint64_t i,
                                          uint64_t* first, uint64_t* next) {
  const int lane = threadIdx.x & 31;
  if (hi - lo <= 30) {  // the same for the whole warp
    const uint64_t eb = __ldg(p.ebeg + lo + min(lane, hi - lo + 1));
    int k = 0;  // the last k <= hi - lo with first entry <= i
#pragma unroll
    for (int step = 16; step > 0; step >>= 1) {
      const int c = k + step;
      const uint64_t v = __shfl_sync(kFull, eb, c < 31 ? c : 31);
      if (c <= hi - lo && v <= i) k = c;
    }
    *first = __shfl_sync(kFull, eb, k);
    *next = __shfl_sync(kFull, eb, k + 1);
    return lo + k;
  }
  const int b = gbank(p.ebeg, lo, hi, i);
  *first = __ldg(p.ebeg + b);
  *next = __ldg(p.ebeg + b + 1);
  return b;
}

template <bool UNIFORM>
__global__ void __launch_bounds__(kThreads, 4) k_gfinish(GPlan p, int first_pass) {
  __shared__ uint32_t ch[kGBins];
  __shared__ unsigned long long wh[UNIFORM ? 1 : kGBins];
  __shared__ GLocal s;
  __shared__ uint64_t scan64[kWarps];
  __shared__ uint32_t scan32[kWarps];
  __shared__ bool s_ok;
  GState* st = p.st;
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const uint64_t nthreads = static_cast<uint64_t>(gridDim.x) * kThreads;
  const uint64_t gtid = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x;
  const uint32_t units = static_cast<uint32_t>(p.tiles) * kWarps;
  const uint32_t gwarp = blockIdx.x * kWarps + wib, nwarps = gridDim.x * kWarps;
  if (threadIdx.x == 0) {
    s.prefix = __ldcg(&st->prefix);
    s.mask = __ldcg(&st->mask);
    s.remaining = __ldcg(&st->remaining);
    s.threshold = __ldcg(&st->threshold);
    s.done = __ldcg(&st->done);
  }
  // Scratch bins of the passes after the first binned here; nothing adds to
  // them before the first barrier.
  for (uint64_t i = gtid; i < static_cast<uint64_t>(kGPasses) * kGBins; i += nthreads) {
    const int ps = static_cast<int>(i / kGBins);
    if (ps > first_pass) {
      p.hb[ps].c[i % kGBins] = 0;
      p.hb[ps].w[i % kGBins] = 0;
    }
  }
  auto zero_bins = [&]() {
    for (int i = threadIdx.x; i < kGBins; i += kThreads) {
      ch[i] = 0;
      if (!UNIFORM) wh[i] = 0;
    }
    __syncthreads();
  };
  // The digit choice of a pass, by the last block to reach the barrier after
  // it; every block then reads the new state.
  auto pick = [&](int ps) {
    gpick_block<UNIFORM>(&s, ps, p.uniform_bytes, gbins_c(p, ps, first_pass),
                         gbins_w(p, ps, first_pass), scan64);
    if (threadIdx.x == 0) {
      st->prefix = s.prefix;
      st->mask = s.mask;
      st->remaining = s.remaining;
      st->threshold = s.threshold;
      st->done = s.done;
    }
  };
  auto load_state = [&]() {
    if (threadIdx.x == 0) {
      s.prefix = __ldcg(&st->prefix);
      s.mask = __ldcg(&st->mask);
      s.remaining = __ldcg(&st->remaining);
      s.threshold = __ldcg(&st->threshold);
      s.done = __ldcg(&st->done);
    }
    __syncthreads();
  };
  // Each warp's units in turn (unit u: the candidates of entries
  // [512 u, 512 u + 512)), the next unit's count fetched ahead.
  auto for_units = [&](auto&& body) {
    uint32_t u = gwarp;
    uint32_t nc = u < units ? __ldcg(p.ucand + u) : 0u;
    while (u < units) {
      const uint32_t un = u + nwarps;
      const uint32_t nn = un < units ? __ldcg(p.ucand + un) : 0u;
      if (nc) body(u, nc);
      u = un;
      nc = nn;
    }
  };
  uint32_t nbar = 0;  // barriers passed
  __syncthreads();
  int pass = first_pass;

  // Pass 0: the top digit of every key.
  if (pass == 0 && !s.done) {
    zero_bins();
    for (int t = blockIdx.x; t < p.tiles; t += gridDim.x) {
      const uint64_t end = min(static_cast<uint64_t>(t + 1) * kGTile, p.entries);
      const uint64_t i0 = glane0(t);
      float sc[kGPer];
      gload(p, i0, end, sc);
      int b = 0, hi = 0;
      if (!UNIFORM && i0 < end) {
        hi = p.tile_bank[t + 1];
        b = gbank(p.ebeg, p.tile_bank[t], hi, i0);
      }
#pragma unroll
      for (int j = 0; j < kGPer; ++j) {
        const uint64_t i = i0 + j;
        uint64_t bytes = 0;
        if (!UNIFORM && i < end) {
          while (b < hi && __ldg(p.ebeg + b + 1) <= i) ++b;
          bytes = __ldg(p.ebytes + b);
        }
        gbin<UNIFORM>(ch, wh, i < end ? ord32(sc[j]) >> 21 : kGBins, bytes);
      }
    }
    gbins_add<UNIFORM>(ch, wh, kGBins, gbins_c(p, 0, first_pass), gbins_w(p, 0, first_pass));
    if (!grid_barrier(st, p.err, ++nbar, &s_ok, [&] { pick(0); })) return;
    load_state();
    pass = 1;
  }

  // The first full scan: kept-for-sure counts per tile; candidates (keys
  // inside the digits fixed so far) binned by the next digit and stored in
  // their unit's slots.
  const bool cand_scan = !s.done;
  if (cand_scan) zero_bins();
  {
    const int shift = gdigit_shift(pass);
    const uint32_t dmask = (1u << gdigit_bits(pass)) - 1u;
    const uint64_t prefix = s.prefix, mask = s.mask;
    const uint64_t above = s.done ? s.threshold : (prefix | ~mask);
    for (int t = blockIdx.x; t < p.tiles; t += gridDim.x) {
      const uint64_t end = min(static_cast<uint64_t>(t + 1) * kGTile, p.entries);
      const uint64_t i0 = glane0(t);
      float sc[kGPer];
      gload(p, i0, end, sc);
      uint32_t sure = 0, cm = 0;
#pragma unroll
      for (int j = 0; j < kGPer; ++j) {
        if (i0 + j < end) {
          const uint64_t key = gkey_of(sc[j], p.pos_base + i0 + j);
          if (key > above) ++sure;
          else if (cand_scan && (key & mask) == prefix) cm |= 1u << j;
        }
      }
      uint32_t nc, sure_w;
      const uint32_t at0 = warp_excl_scan(__popc(cm), &nc);
      warp_excl_scan(sure, &sure_w);
      if (cm) {  // few lanes: bin the candidates and store them in the unit's slots
        const uint64_t slot = (static_cast<uint64_t>(t) * kWarps + wib) * kGUnit + at0;
        int b = 0, hi = 0;
        if (!UNIFORM) {
          hi = p.tile_bank[t + 1];
          b = gbank(p.ebeg, p.tile_bank[t], hi, i0);
        }
        uint32_t k = 0;
#pragma unroll
        for (int j = 0; j < kGPer; ++j) {
          if (cm & (1u << j)) {
            const uint64_t i = i0 + j;
            const uint64_t key = gkey_of(sc[j], p.pos_base + i);
            const uint32_t d = static_cast<uint32_t>(key >> shift) & dmask;
            p.ckey[slot + k] = key;
            atomicAdd(&ch[d], 1u);
            if (!UNIFORM) {
              while (b < hi && __ldg(p.ebeg + b + 1) <= i) ++b;
              p.cbank[slot + k] = static_cast<uint32_t>(b);
              atomicAdd(&wh[d], static_cast<unsigned long long>(__ldg(p.ebytes + b)));
            }
            ++k;
          }
        }
      }
      if (lane == 0) {
        p.ucand[static_cast<uint64_t>(t) * kWarps + wib] = nc;
        scan32[wib] = sure_w;
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t sum = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) sum += scan32[w];
        p.tile_cnt[t] = sum;
      }
      __syncthreads();
    }
  }
  if (cand_scan) {
    gbins_add<UNIFORM>(ch, wh, 1 << gdigit_bits(pass), gbins_c(p, pass, first_pass),
                       gbins_w(p, pass, first_pass));
    if (!grid_barrier(st, p.err, ++nbar, &s_ok, [&] { pick(pass); })) return;
    load_state();
    ++pass;
  }

  // Later passes over the candidates only.
  while (!s.done && pass < kGPasses) {
    zero_bins();
    const int shift = gdigit_shift(pass);
    const uint32_t dmask = (1u << gdigit_bits(pass)) - 1u;
    const uint64_t prefix = s.prefix, mask = s.mask;
    for_units([&](uint32_t u, uint32_t nc) {
      const uint64_t slot = static_cast<uint64_t>(u) * kGUnit;
      for (uint32_t k = lane; k < nc; k += 32) {
        const uint64_t key = __ldcg(p.ckey + slot + k);
        if ((key & mask) == prefix) {
          const uint32_t d = static_cast<uint32_t>(key >> shift) & dmask;
          atomicAdd(&ch[d], 1u);
          if (!UNIFORM)
            atomicAdd(&wh[d], static_cast<unsigned long long>(
                                  __ldg(p.ebytes + __ldcg(p.cbank + slot + k))));
        }
      }
    });
    gbins_add<UNIFORM>(ch, wh, 1 << gdigit_bits(pass), gbins_c(p, pass, first_pass),
                       gbins_w(p, pass, first_pass));
    if (!grid_barrier(st, p.err, ++nbar, &s_ok, [&] { pick(pass); })) return;
    load_state();
    ++pass;
  }
  const uint64_t T = s.threshold;

  // Kept candidates join their tiles' counts.
  if (cand_scan) {
    for_units([&](uint32_t u, uint32_t nc) {
      const uint64_t slot = static_cast<uint64_t>(u) * kGUnit;
      uint32_t kept = 0;
      for (uint32_t k = lane; k < nc; k += 32) kept += __ldcg(p.ckey + slot + k) > T;
#pragma unroll
      for (int d = 16; d > 0; d >>= 1) kept += __shfl_xor_sync(kFull, kept, d);
      if (lane == 0 && kept) atomicAdd(p.tile_cnt + u / kWarps, kept);
    });
  }
  if (!grid_barrier(st, p.err, ++nbar, &s_ok, [] {})) return;

  // Write: block b takes tiles [t0, t1) and starts at the kept count before t0.
  const int t0 = static_cast<int>(static_cast<int64_t>(p.tiles) * blockIdx.x / gridDim.x);
  const int t1 = static_cast<int>(static_cast<int64_t>(p.tiles) * (blockIdx.x + 1) / gridDim.x);
  uint32_t before = 0;
  {
    uint32_t part = 0;
    for (int t = threadIdx.x; t < t0; t += kThreads) part += __ldcg(p.tile_cnt + t);
    uint32_t total;
    block_excl_scan(part, scan32, &total);
    before = total;
  }
  if (blockIdx.x == 0) {  // the total and the offsets of trailing empty banks
    uint32_t part = 0;
    for (int t = threadIdx.x; t < p.tiles; t += kThreads) part += __ldcg(p.tile_cnt + t);
    uint32_t total;
    block_excl_scan(part, scan32, &total);
    if (threadIdx.x == 0) {
      st->total_kept = total;
      st->threshold = T;
      p.kept_off[p.n_banks] = static_cast<int32_t>(total);
      for (int b = p.n_banks - 1; b >= 0 && p.ebeg[b] == p.entries; --b)
        p.kept_off[b] = static_cast<int32_t>(total);
    }
  }
  for (int t = t0; t < t1; ++t) {
    const uint64_t end = min(static_cast<uint64_t>(t + 1) * kGTile, p.entries);
    const uint64_t i0 = glane0(t);
    uint32_t keep = 0;  // bit j: entry i0 + j is kept
    {
      float sc[kGPer];
      gload(p, i0, end, sc);
#pragma unroll
      for (int j = 0; j < kGPer; ++j)
        if (i0 + j < end && gkey_of(sc[j], p.pos_base + i0 + j) > T) keep |= 1u << j;
    }
    uint32_t wtot;
    const uint32_t lane_before = warp_excl_scan(__popc(keep), &wtot);
    if (lane == 0) scan32[wib] = wtot;
    __syncthreads();
    uint32_t rank = before + lane_before, all = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const uint32_t v = scan32[w];
      if (w < wib) rank += v;
      all += v;
    }
    __syncthreads();
    // The lane's bank cursor: bank b holds entries [first, next).
    const int hi = p.tile_bank[t + 1];
    uint64_t first, next;
    int b = gbank_tile(p, p.tile_bank[t], hi, i0, &first, &next);
    if (i0 < end) {
#pragma unroll
      for (int j = 0; j < kGPer; ++j) {
        const uint64_t i = i0 + j;
        if (i < end) {
          while (b < hi && next <= i) {
            ++b;
            first = next;
            next = __ldg(p.ebeg + b + 1);
          }
          if (i == first) {
            p.kept_off[b] = static_cast<int32_t>(rank);
            for (int e = b - 1; e >= 0 && __ldg(p.ebeg + e) == i; --e)
              p.kept_off[e] = static_cast<int32_t>(rank);
          }
          if (keep & (1u << j)) p.kept_idx[rank++] = static_cast<int32_t>(i - first);
        }
      }
    }
    before += all;
  }
}

// ---------------------------------------------------------------------------
// Copy-on-write page pool
//
// A page's count is the number of table slots that hold it.  A fork shares
// pages (count + 1, no bytes move); before a slot's page is written, the copy
// leg gives the slot a private copy if anybody else still holds the page.
// Of several holders writing in one launch, the last one to give up its hold
// finds the count at 1 and keeps the page, so exactly holders - 1 copies are
// made and no page is lost.  Ids are checked against the pool; -1 is an empty
// slot and is skipped.
// ---------------------------------------------------------------------------

__device__ __forceinline__ bool pool_id_ok(const PoolDev& P, int32_t p) {
  if (p < 0) return false;
  if (p >= P.n_pages) {
    atomicOr(P.err, kDevErrIndex);
    return false;
  }
  return true;
}

// Pops aggregated per warp: one atomic on the stack top for the warp's lanes.
__global__ void __launch_bounds__(kThreads) k_pool_alloc(PoolDev P, int32_t* ids, int32_t n) {
  const int32_t j = blockIdx.x * kThreads + threadIdx.x;
  const int lane = threadIdx.x & 31;
  const unsigned want = __ballot_sync(kFull, j < n);
  if (j >= n) return;
  const int cnt = __popc(want), r = __popc(want & ((1u << lane) - 1u));
  const int leader = __ffs(want) - 1;
  int32_t old = 0;
  if (lane == leader) {
    old = atomicSub(P.top, cnt);
    const int32_t ok = old <= 0 ? 0 : (old < cnt ? old : cnt);
    if (ok < cnt) {
      atomicAdd(P.top, cnt - ok);
      atomicOr(P.err, kDevErrNoPage);
    }
  }
  old = __shfl_sync(want, old, leader);
  const int32_t i = old - 1 - r;
  if (i >= 0) {
    const int32_t q = P.free_ids[i];
    P.rc[q] = 1;
    ids[j] = q;
  } else {
    ids[j] = -1;
  }
}

__global__ void __launch_bounds__(kThreads)
    k_pool_share(PoolDev P, const int32_t* src, int32_t* dst, int32_t n) {
  const int32_t j = blockIdx.x * kThreads + threadIdx.x;
  if (j >= n) return;
  const int32_t p = src[j];
  if (dst) dst[j] = p;
  if (!pool_id_ok(P, p)) return;
  if (atomicAdd(&P.rc[p], 1u) == 0u) {
    atomicSub(&P.rc[p], 1u);
    atomicOr(P.err, kDevErrRefcount);
  }
}

__global__ void __launch_bounds__(kThreads)
    k_pool_release(PoolDev P, const int32_t* ids, int32_t n) {
  const int32_t j = blockIdx.x * kThreads + threadIdx.x;
  const unsigned live = __ballot_sync(kFull, j < n);  // lanes that reach the push
  if (j >= n) return;
  const int32_t p = ids[j];
  bool freed = false;
  if (pool_id_ok(P, p)) {
    const uint32_t old = atomicSub(&P.rc[p], 1u);
    if (old == 1u) {
      freed = true;
    } else if (old == 0u) {
      atomicAdd(&P.rc[p], 1u);
      atomicOr(P.err, kDevErrRefcount);
    }
  }
  // Pushes aggregated per warp: one atomic on the stack top.
  const unsigned push = __ballot_sync(live, freed);
  if (!push) return;
  const int lane = threadIdx.x & 31;
  const int leader = __ffs(push) - 1;
  int32_t i0 = 0;
  if (lane == leader) i0 = atomicAdd(P.top, __popc(push));
  i0 = __shfl_sync(live, i0, leader);
  if (freed) {
    const int32_t i = i0 + __popc(push & ((1u << lane) - 1u));
    if (i < P.n_pages) {
      P.free_ids[i] = p;
    } else {  // counts were inconsistent: never write past the stack
      atomicSub(P.top, 1);
      atomicOr(P.err, kDevErrRefcount);
    }
  }
}

// One warp per table slot, eight slots per block round: lane 0 of each warp
// settles its slot's hold; the slots that need a page take them off the free
// stack with one atomic for the block (pages taken past an empty stack are
// given back and reported); then every warp copies its page, kCowDepth
// 16-byte loads in flight per lane.
constexpr int kCowDepth = 8;

__global__ void __launch_bounds__(kThreads)
    k_pool_cow(PoolDev P, int32_t* table, int64_t n_table, const int32_t* entries, int32_t n) {
  __shared__ uint32_t s_need;  // bit w: warp w needs a fresh page
  __shared__ int32_t s_base;   // stack top before this round's pops
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  for (int64_t j0 = static_cast<int64_t>(blockIdx.x) * kWarps; j0 < n;
       j0 += static_cast<int64_t>(gridDim.x) * kWarps) {
    const int64_t j = j0 + wib;
    int32_t p = -1;
    int64_t e = 0;
    bool need = false;
    if (threadIdx.x == 0) s_need = 0;
    __syncthreads();
    if (lane == 0 && j < n) {
      e = entries ? static_cast<int64_t>(entries[j]) : j;
      if (e < 0 || e >= n_table) {
        atomicOr(P.err, kDevErrIndex);
      } else {
        p = table[e];
        if (pool_id_ok(P, p)) {
          const uint32_t old = atomicSub(&P.rc[p], 1u);
          if (old == 1u) {
            atomicAdd(&P.rc[p], 1u);  // held here alone: keep it
          } else if (old == 0u) {
            atomicAdd(&P.rc[p], 1u);
            atomicOr(P.err, kDevErrRefcount);
          } else {
            need = true;
            atomicOr(&s_need, 1u << wib);
          }
        }
      }
    }
    __syncthreads();
    const uint32_t mask = s_need;
    if (threadIdx.x == 0 && mask) {
      const int cnt = __popc(mask);
      const int32_t old = atomicSub(P.top, cnt);
      const int32_t ok = old <= 0 ? 0 : (old < cnt ? old : cnt);
      if (ok < cnt) {
        atomicAdd(P.top, cnt - ok);
        atomicOr(P.err, kDevErrNoPage);
      }
      s_base = old;
    }
    __syncthreads();
    int32_t q = -1;
    if (lane == 0 && need) {
      const int32_t i = s_base - 1 - __popc(mask & ((1u << wib) - 1u));
      if (i >= 0) {
        q = P.free_ids[i];
        P.rc[q] = 1;
      } else {
        atomicAdd(&P.rc[p], 1u);  // no page: keep the shared hold
      }
    }
    q = __shfl_sync(kFull, q, 0);
    if (q >= 0) {
      p = __shfl_sync(kFull, p, 0);
      const uint4* src =
          reinterpret_cast<const uint4*>(P.base + static_cast<uint64_t>(p) * P.page_bytes);
      uint4* dst = reinterpret_cast<uint4*>(P.base + static_cast<uint64_t>(q) * P.page_bytes);
      const uint64_t words = P.page_bytes / 16;
      for (uint64_t k0 = lane; k0 < words; k0 += 32 * kCowDepth) {
        uint4 v[kCowDepth];
#pragma unroll
        for (int u = 0; u < kCowDepth; ++u) {
          const uint64_t k = k0 + 32u * u;
          if (k < words) v[u] = __ldcs(src + k);
        }
#pragma unroll
        for (int u = 0; u < kCowDepth; ++u) {
          const uint64_t k = k0 + 32u * u;
          if (k < words) dst[k] = v[u];
        }
      }
      if (lane == 0) table[e] = q;
    }
  }
}

// ---------------------------------------------------------------------------
// Byte-mismatch distance: the count of differing bytes of buffer pairs (the
// distance D of the discovery procedure at the byte level).  Every block
// takes 16 KiB tiles of the pairs in turn; 16-byte loads where both buffers
// are 16-byte aligned, byte loads otherwise.
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t bytes_ne(uint32_t x, uint32_t y) {
  return __popc(__vcmpne4(x, y)) >> 3;
}

// Every warp takes a contiguous range of 2 KiB units of the concatenated
// pairs, finds the pair of its first unit once and walks forward; its count
// is reduced across the warp and added to the pair when the pair changes.
__global__ void __launch_bounds__(kThreads, 4)
    k_mismatch(const MmPair* __restrict__ pairs, const uint64_t* __restrict__ unit_begin,
               int32_t n, uint64_t units, uint64_t* counts) {
  const int lane = threadIdx.x & 31;
  const uint64_t warps = static_cast<uint64_t>(gridDim.x) * kWarps;
  const uint64_t w = static_cast<uint64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const uint64_t per = (units + warps - 1) / warps;
  const uint64_t u0 = w * per;
  const uint64_t u1 = u0 + per < units ? u0 + per : units;
  if (u0 >= u1) return;
  int lo = 0, hi = n - 1;  // the last pair whose first unit is <= u0
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(unit_begin + mid) <= u0) lo = mid;
    else hi = mid - 1;
  }
  int pi = lo;
  MmPair P = pairs[pi];
  uint64_t pbeg = __ldg(unit_begin + pi), pend = __ldg(unit_begin + pi + 1);
  uint32_t c = 0;
  for (uint64_t u = u0; u < u1; ++u) {
    if (u >= pend) {
      const uint32_t tot = __reduce_add_sync(kFull, c);
      if (lane == 0 && tot)
        atomicAdd(reinterpret_cast<unsigned long long*>(counts + pi),
                  static_cast<unsigned long long>(tot));
      c = 0;
      do {
        ++pi;
        pend = __ldg(unit_begin + pi + 1);
      } while (u >= pend);
      P = pairs[pi];
      pbeg = __ldg(unit_begin + pi);
    }
    const uint64_t off = (u - pbeg) * kMmUnit;
    const uint32_t len = static_cast<uint32_t>(P.bytes - off < kMmUnit ? P.bytes - off : kMmUnit);
    if (P.vec) {
      const uint4* a = reinterpret_cast<const uint4*>(P.a + off);
      const uint4* b = reinterpret_cast<const uint4*>(P.b + off);
      const uint32_t words = len >> 4;
      uint4 va[4], vb[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t x = lane + 32u * k;
        if (x < words) {
          va[k] = __ldcs(a + x);
          vb[k] = __ldcs(b + x);
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t x = lane + 32u * k;
        if (x < words)
          c += bytes_ne(va[k].x, vb[k].x) + bytes_ne(va[k].y, vb[k].y) +
               bytes_ne(va[k].z, vb[k].z) + bytes_ne(va[k].w, vb[k].w);
      }
      for (uint32_t x = (words << 4) + lane; x < len; x += 32) c += P.a[off + x] != P.b[off + x];
    } else {
      for (uint32_t x = lane; x < len; x += 32) c += P.a[off + x] != P.b[off + x];
    }
  }
  const uint32_t tot = __reduce_add_sync(kFull, c);
  if (lane == 0 && tot)
    atomicAdd(reinterpret_cast<unsigned long long*>(counts + pi),
              static_cast<unsigned long long>(tot));
}

// ---------------------------------------------------------------------------
// Reads against buffers: a buffer is read iff a read of at least one byte
// overlaps it (state versus witness: restore reads state, not witness).
// One thread per read; the candidates are the buffers starting before the
// read ends and, among them, those from the first whose running maximum end
// passes the read's start.
// ---------------------------------------------------------------------------

// Threads stride over the reads; a block marks the buffers it saw in a
// shared bitmap and writes each flag once at the end (many reads hit few
// buffers, so stores to the flags would otherwise pile up on a few lines).
// With few buffers the sorted arrays are staged in shared memory too.
constexpr int kReadStage = 512;  // buffers staged in shared memory

__global__ void __launch_bounds__(kThreads)
    k_classify_reads(ReadPlan P, const uint64_t* __restrict__ addr,
                     const uint64_t* __restrict__ bytes, int64_t m, uint8_t* flags) {
  extern __shared__ __align__(16) uint8_t rd_smem[];
  uint32_t* const seen = reinterpret_cast<uint32_t*>(rd_smem);  // [words] bitmap
  const int words = (P.n + 31) / 32;
  const bool staged = P.n <= kReadStage;
  uint64_t* s_start = reinterpret_cast<uint64_t*>(seen + ((words + 1) & ~1));
  uint64_t* s_end = s_start + (staged ? P.n : 0);
  uint64_t* s_max = s_end + (staged ? P.n : 0);
  for (int w = threadIdx.x; w < words; w += kThreads) seen[w] = 0;
  if (staged)
    for (int i = threadIdx.x; i < P.n; i += kThreads) {
      s_start[i] = P.start[i];
      s_end[i] = P.end[i];
      s_max[i] = P.maxend[i];
    }
  __syncthreads();
  const uint64_t* st = staged ? s_start : P.start;
  const uint64_t* en = staged ? s_end : P.end;
  const uint64_t* mx = staged ? s_max : P.maxend;
  for (int64_t j = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; j < m;
       j += static_cast<int64_t>(gridDim.x) * kThreads) {
    const uint64_t a = addr[j], len = bytes[j];
    if (len == 0) continue;
    const uint64_t e = a + len < a ? ~0ull : a + len;
    int lo = 0, hi = P.n;  // hi: first buffer starting at or after e
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (st[mid] < e) lo = mid + 1;
      else hi = mid;
    }
    const int end_i = lo;
    lo = 0;
    hi = end_i;  // first buffer whose running maximum end exceeds a
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (mx[mid] > a) hi = mid;
      else lo = mid + 1;
    }
    for (int i = lo; i < end_i; ++i) {
      const uint32_t bit = 1u << (i & 31);
      // Most reads hit a buffer already marked: look before the atomic.
      if (en[i] > a && en[i] > st[i] && !(seen[i >> 5] & bit)) atomicOr(&seen[i >> 5], bit);
    }
  }
  __syncthreads();
  for (int w = threadIdx.x; w < words; w += kThreads) {
    uint32_t bits = seen[w];
    while (bits) {
      const int b = __ffs(bits) - 1;
      bits &= bits - 1;
      flags[P.orig[32 * w + b]] = 1;
    }
  }
}

// ---------------------------------------------------------------------------
// Self-test of the bounded waits: one thread waits, through the helpers the
// production kernels use and with their bound, for something that never
// happens -- the second arrival at an mbarrier that expects two (the TMA
// pipeline's wait) or a flag nothing writes (the grid barrier's poll) --
// then records the timeout in the context's error word and returns.
// ---------------------------------------------------------------------------

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__global__ void k_selftest_wait(int which, const uint32_t* never_set, uint32_t* err) {
  __shared__ uint64_t bar;
  if (threadIdx.x != 0) return;
  bool ok;
  if (which == 0) {
    mbar_init(&bar, 2);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    mbar_arrive(&bar);
    ok = mbar_wait(&bar, 0);
  } else {
    ok = wait_flag_geq(never_set, 1);
  }
  if (!ok) atomicOr(err, kDevErrTimeout);
}

// Launch `k` with programmatic stream serialisation: the GPU may schedule it
// while the kernel before it on `stream` finishes (its blocks wait in
// grid_dependency() until that kernel's writes are visible), instead of only
// after that kernel has retired.  After a copy, an event or another kind of
// stream operation the launch waits as usual.
template <typename... P, typename... A>
cudaError_t launch_after(void (*k)(P...), unsigned grid, unsigned block, size_t smem,
                         cudaStream_t stream, A... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, args...);
}

template <int MODE>
int occupancy() {
  int b = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_stream<MODE>, kThreads, 0);
  return b > 0 ? b : 1;
}

// Blocks of kThreads threads (no dynamic shared memory) of `kernel` that one
// SM holds at once, asked once per kernel.  A grid of SMs x this many blocks
// is one resident wave: a larger grid of equal blocks leaves its last wave
// part-full, with fewer loads in flight while it runs.
int resident_blocks(const void* kernel) {
  static std::mutex mu;
  static const void* keys[64];
  static int vals[64];
  static int n = 0;
  std::lock_guard<std::mutex> lk(mu);
  for (int i = 0; i < n; ++i)
    if (keys[i] == kernel) return vals[i];
  int b = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, kThreads, 0) != cudaSuccess || b < 1)
    b = 1;
  if (n < 64) {
    keys[n] = kernel;
    vals[n++] = b;
  }
  return b;
}

template <int MODE>
cudaError_t launch_bulk_mode(const SecDesc* secs, WorkList wl, uint64_t* nodes, uint32_t* err,
                             uint32_t* sched, int sm_count, cudaStream_t stream) {
  using Shape = BulkShape<MODE>;
  const size_t smem = sizeof(BulkShared<Shape::kWarps, Shape::kStages>);
  // One bit per device.  Contexts on other threads may set the attribute at
  // the same time; setting it twice is harmless.
  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(k_bulk<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k_bulk_shared<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured.fetch_or(bit, std::memory_order_release);
  }
  const uint64_t want = (static_cast<uint64_t>(wl.n_tasks) + Shape::kWarps - 1) / Shape::kWarps;
  const int blocks = static_cast<int>(want < static_cast<uint64_t>(sm_count) ? want : sm_count);
  if (wl.n_tasks < static_cast<uint64_t>(kDynMaxTilesPerWarp) * blocks * Shape::kWarps)
    return launch_after(k_bulk_shared<MODE>, blocks, Shape::kThreads, smem, stream, secs, wl, nodes,
                        err, sched);
  return launch_after(k_bulk<MODE>, blocks, Shape::kThreads, smem, stream, secs, wl, nodes, err);
}

}  // namespace

int stream_blocks_per_sm() { return occupancy<kModePack>(); }

cudaError_t launch_stream(int mode, const SecDesc* secs, WorkList wl, int group_log2,
                          uint64_t* nodes, uint32_t* dev_err, int sm_count, int blocks_per_sm,
                          cudaStream_t stream) {
  if (wl.n_tasks == 0) return cudaSuccess;
  const uint64_t want = (static_cast<uint64_t>(wl.n_tasks) + kWarps - 1) / kWarps;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * blocks_per_sm;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  switch (mode) {
    case kModeHash:
      return launch_after(k_stream<kModeHash>, blocks, kThreads, 0, stream, secs, wl, group_log2,
                          nodes, dev_err);
    case kModePack:
      return launch_after(k_stream<kModePack>, blocks, kThreads, 0, stream, secs, wl, group_log2,
                          nodes, dev_err);
    case kModeRestore:
      return launch_after(k_stream<kModeRestore>, blocks, kThreads, 0, stream, secs, wl,
                          group_log2, nodes, dev_err);
    case kModeRestoreV:
      return launch_after(k_stream<kModeRestoreV>, blocks, kThreads, 0, stream, secs, wl,
                          group_log2, nodes, dev_err);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_bulk(int mode, const SecDesc* secs, WorkList wl, uint64_t* nodes,
                        uint32_t* dev_err, uint32_t* sched, int sm_count, cudaStream_t stream) {
  if (wl.n_tasks == 0) return cudaSuccess;
  switch (mode) {
    case kModeHash: {
      const uint64_t want = (static_cast<uint64_t>(wl.n_tasks) + kHashWarps - 1) / kHashWarps;
      const int blocks = static_cast<int>(want < static_cast<uint64_t>(sm_count) ? want : sm_count);
      return launch_after(k_hash, blocks, kHashThreads, 0, stream, secs, wl, nodes);
    }
    case kModePack: return launch_bulk_mode<kModePack>(secs, wl, nodes, dev_err, sched, sm_count, stream);
    case kModeRestore:
      return launch_bulk_mode<kModeRestore>(secs, wl, nodes, dev_err, sched, sm_count, stream);
    case kModeRestoreV:
      return launch_bulk_mode<kModeRestoreV>(secs, wl, nodes, dev_err, sched, sm_count, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_small(int mode, const SecDesc* secs, WorkList wl, int group_log2,
                         uint64_t* nodes, uint32_t* dev_err, uint32_t* ticket, int n_items,
                         const SessDesc* sess, const Entry* entries, uint64_t* fp_out,
                         const uint64_t* fp_before, uint8_t* flags, uint32_t* bad, int sm_count,
                         int blocks_per_sm, cudaStream_t stream) {
  if (wl.n_tasks == 0) return cudaErrorInvalidValue;
  const uint64_t want = (static_cast<uint64_t>(wl.n_tasks) + kWarps - 1) / kWarps;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * blocks_per_sm;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  switch (mode) {
    case kModeHash:
      return launch_after(k_small<kModeHash>, blocks, kThreads, 0, stream, secs, wl, group_log2,
                          nodes, dev_err, ticket, n_items, sess, entries, fp_out, fp_before, flags,
                          bad);
    case kModePack:
      return launch_after(k_small<kModePack>, blocks, kThreads, 0, stream, secs, wl, group_log2,
                          nodes, dev_err, ticket, n_items, sess, entries, fp_out, fp_before, flags,
                          bad);
    case kModeRestoreV:
      return launch_after(k_small<kModeRestoreV>, blocks, kThreads, 0, stream, secs, wl,
                          group_log2, nodes, dev_err, ticket, n_items, sess, entries, fp_out,
                          fp_before, flags, bad);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_finalize(int mode, const SecDesc* secs, const SessDesc* sess, int n_sess,
                            const Entry* entries, uint64_t* nodes, uint64_t* fp_out,
                            const uint64_t* fp_before, uint8_t* flags, uint32_t* bad,
                            int max_secs, cudaStream_t stream) {
  if (n_sess <= 0) return cudaSuccess;
  if (mode != kModeHash && max_secs <= 32 && n_sess >= 256) {
    // Many sessions of few sections: a warp each, not a block each.  Fewer
    // sessions take a block each, a warp per section, so a session's
    // sections are treed side by side (the 64-bank step: 0.224 -> 0.220 ms).
    const int want = (n_sess + kWarps - 1) / kWarps;
    const int blocks = want < 65535 ? want : 65535;
    if (mode == kModePack)
      return launch_after(k_finalize_sessions_warp<kModePack>, blocks, kThreads, 0, stream, secs,
                          sess, n_sess, entries, nodes, flags, bad);
    if (mode == kModeRestoreV)
      return launch_after(k_finalize_sessions_warp<kModeRestoreV>, blocks, kThreads, 0, stream,
                          secs, sess, n_sess, entries, nodes, flags, bad);
    return cudaErrorInvalidValue;
  }
  if (mode == kModeHash) {
    const int blocks = (n_sess + kWarps - 1) / kWarps;
    return launch_after(k_finalize_hash, blocks < 4096 ? blocks : 4096, kThreads, 0, stream, secs,
                        n_sess, nodes, fp_out, fp_before, flags);
  }
  if (mode == kModePack || mode == kModeRestoreV) {
    // A block per session, a warp per section (up to 16 at once: two
    // blocks of 64-register threads fit an SM).
    const int warps = max_secs < 8 ? 8 : max_secs > 16 ? 16 : max_secs;
    const int blocks = n_sess < 65535 ? n_sess : 65535;
    if (mode == kModePack)
      return launch_after(k_finalize_sessions<kModePack>, blocks, 32 * warps, 0, stream, secs, sess,
                          n_sess, entries, nodes, flags, bad);
    return launch_after(k_finalize_sessions<kModeRestoreV>, blocks, 32 * warps, 0, stream, secs,
                        sess, n_sess, entries, nodes, flags, bad);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_reduce_nodes(const NodeLevel* lv, int n_secs, uint64_t* nodes, uint32_t base,
                                uint32_t n_groups, int sm_count, cudaStream_t stream) {
  if (n_groups == 0) return cudaSuccess;
  const uint64_t want = (static_cast<uint64_t>(n_groups) + kWarps - 1) / kWarps;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * 8;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  return launch_after(k_reduce_nodes, blocks, kThreads, 0, stream, lv, n_secs, nodes, base, n_groups);
}

cudaError_t launch_score(const BankDesc* banks, int n_banks, uint64_t n_entries, int max_dim,
                         int key_types, float* scores, int sm_count, cudaStream_t stream,
                         GHist gh, bool* fused) {
  if (fused) *fused = false;
  if (n_entries == 0) return cudaSuccess;
  // At least two rounds of kScoreIlp entries per warp; at most one resident
  // wave (large populations fill it).  Eight rounds per warp took the 64-bank
  // population's score (16,164 entries) 15.5 us under ncu.
  const uint64_t want = (n_entries + kWarps * kScoreIlp * 2 - 1) / (kWarps * kScoreIlp * 2);
  auto grid = [&](const void* k) {
    const uint64_t cap = static_cast<uint64_t>(sm_count) * resident_blocks(k);
    return static_cast<int>(want < cap ? want : cap);
  };
  // key_types: 0 = all fp16, 1 = all bf16, 2 = mixed.
  if (key_types == 2 || max_dim > 1024) {
    return launch_after(k_score_any, grid(reinterpret_cast<const void*>(k_score_any)), kThreads, 0,
                        stream, banks, n_banks, n_entries, scores);
  }
  const int spl = max_dim <= 256 ? 1 : max_dim <= 512 ? 2 : 4;
  const int hm = gh.st ? gh.mode : 0;
  cudaError_t e = cudaSuccess;
#define PCS_SCORE(S, D, H)                                                                      \
  e = launch_after(k_score_fixed<S, D, H>,                                                      \
                   grid(reinterpret_cast<const void*>(k_score_fixed<S, D, H>)), kThreads, 0, stream, \
                   banks, n_banks, n_entries, scores, gh)
#define PCS_SCORE_H(S, D) (hm == 0 ? PCS_SCORE(S, D, 0) : hm == 1 ? PCS_SCORE(S, D, 1) : PCS_SCORE(S, D, 2))
  if (key_types == 1) {
    if (spl == 1) PCS_SCORE_H(1, 1);
    else if (spl == 2) PCS_SCORE_H(2, 1);
    else PCS_SCORE_H(4, 1);
  } else {
    if (spl == 1) PCS_SCORE_H(1, 0);
    else if (spl == 2) PCS_SCORE_H(2, 0);
    else PCS_SCORE_H(4, 0);
  }
#undef PCS_SCORE_H
#undef PCS_SCORE
  if (fused) *fused = hm != 0 && e == cudaSuccess;
  return e;
}

cudaError_t launch_topk(const BankDesc* banks, int n_banks, const float* scores,
                        int32_t* kept_idx, cudaStream_t stream) {
  if (n_banks <= 0) return cudaSuccess;
  return launch_after(k_topk, n_banks < 65535 ? n_banks : 65535, kThreads, 0, stream, banks,
                      n_banks, scores, kept_idx);
}

static int gblocks(const GPlan& p, int sm_count, const void* kernel) {
  const int cap = sm_count * resident_blocks(kernel);
  return p.tiles < cap ? p.tiles : cap;
}

cudaError_t launch_gselect(const GPlan& p, int pass, int sm_count, cudaStream_t stream) {
  if (p.tiles <= 0) return cudaSuccess;
  if (p.uniform) {
    const int g = gblocks(p, sm_count, reinterpret_cast<const void*>(k_gselect<true>));
    k_gselect<true><<<g, kThreads, 0, stream>>>(p, pass);
  } else {
    const int g = gblocks(p, sm_count, reinterpret_cast<const void*>(k_gselect<false>));
    k_gselect<false><<<g, kThreads, 0, stream>>>(p, pass);
  }
  return cudaGetLastError();
}

static unsigned grid_for(int64_t n) { return static_cast<unsigned>((n + kThreads - 1) / kThreads); }

cudaError_t launch_pool_alloc(const PoolDev& p, int32_t* ids, int32_t n, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  k_pool_alloc<<<grid_for(n), kThreads, 0, stream>>>(p, ids, n);
  return cudaGetLastError();
}

cudaError_t launch_pool_share(const PoolDev& p, const int32_t* src, int32_t* dst, int32_t n,
                              cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  k_pool_share<<<grid_for(n), kThreads, 0, stream>>>(p, src, dst, n);
  return cudaGetLastError();
}

cudaError_t launch_pool_release(const PoolDev& p, const int32_t* ids, int32_t n,
                                cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  k_pool_release<<<grid_for(n), kThreads, 0, stream>>>(p, ids, n);
  return cudaGetLastError();
}

cudaError_t launch_pool_cow(const PoolDev& p, int32_t* table, int64_t n_table,
                            const int32_t* entries, int32_t n, int sm_count, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  const int64_t want = (static_cast<int64_t>(n) + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sm_count) *
                      resident_blocks(reinterpret_cast<const void*>(k_pool_cow));
  k_pool_cow<<<static_cast<unsigned>(want < cap ? want : cap), kThreads, 0, stream>>>(
      p, table, n_table, entries, n);
  return cudaGetLastError();
}

cudaError_t launch_mismatch(const MmPair* pairs, const uint64_t* unit_begin, int32_t n,
                            uint64_t units, uint64_t* counts, int sm_count, cudaStream_t stream) {
  if (units == 0 || n <= 0) return cudaSuccess;
  // One resident wave (four blocks per SM), at least eight units per warp.
  const uint64_t want = (units + 8 * kWarps - 1) / (8 * kWarps);
  const uint64_t cap = static_cast<uint64_t>(sm_count) * 4;
  k_mismatch<<<static_cast<unsigned>(want < cap ? want : cap), kThreads, 0, stream>>>(
      pairs, unit_begin, n, units, counts);
  return cudaGetLastError();
}

cudaError_t launch_classify_reads(const ReadPlan& p, const uint64_t* addr, const uint64_t* bytes,
                                  int64_t m, uint8_t* flags, int sm_count, cudaStream_t stream) {
  if (m <= 0 || p.n <= 0) return cudaSuccess;
  const size_t words = (static_cast<size_t>(p.n) + 31) / 32;
  size_t smem = ((words + 1) & ~static_cast<size_t>(1)) * 4;
  if (p.n <= kReadStage) smem += 24ull * p.n;
  if (smem > 48 * 1024) {  // more buffers than a block's bitmap can hold
    cudaError_t e = cudaFuncSetAttribute(k_classify_reads,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  const uint64_t want = (static_cast<uint64_t>(m) + kThreads - 1) / kThreads;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * 8;  // 32 registers: 8 blocks per SM
  k_classify_reads<<<static_cast<unsigned>(want < cap ? want : cap), kThreads, smem, stream>>>(
      p, addr, bytes, m, flags);
  return cudaGetLastError();
}

cudaError_t launch_gfinish(const GPlan& p, int first_pass, int sm_count, cudaStream_t stream) {
  if (p.tiles <= 0) return cudaSuccess;
  const void* k = p.uniform ? reinterpret_cast<const void*>(k_gfinish<true>)
                            : reinterpret_cast<const void*>(k_gfinish<false>);
  // Every block must be resident at once: at most one wave.
  const int cap = sm_count * resident_blocks(k);
  const int grid = p.tiles < cap ? p.tiles : cap;
  GPlan a = p;
  int fp = first_pass;
  void* args[] = {&a, &fp};
  return cudaLaunchCooperativeKernel(k, dim3(grid), dim3(kThreads), args, 0, stream);
}


cudaError_t launch_selftest_wait(int which, const uint32_t* never_set, uint32_t* err,
                                 cudaStream_t stream) {
  k_selftest_wait<<<1, 32, 0, stream>>>(which, never_set, err);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Fingerprints with no allocation
//
// For callers that cannot allocate device memory, pcs_fingerprint_static runs
// the fingerprint with its whole working set in one fixed array owned by this
// file: the tree nodes of one call.  The plan (at most kStaticMaxBufs buffers)
// travels as a kernel parameter.  The array is created with the module on
// every GPU that runs the call and stays there until the process exits; all
// calls share it, so calls that overlap on the GPU race on it.  No slot needs
// to start at zero: a call writes every node it later reads.
// ---------------------------------------------------------------------------

namespace {

static __device__ __align__(256) uint64_t g_static_nodes[kStaticMaxNodes];

__global__ void __launch_bounds__(kThreads)
    k_fp_static(const StaticPlan plan, uint64_t* __restrict__ nodes) {
  const int lane = threadIdx.x & 31;
  const uint32_t nw = gridDim.x * kWarps;
  const int g = plan.glog2;
  for (uint32_t task = blockIdx.x * kWarps + (threadIdx.x >> 5); task < plan.n_tasks; task += nw) {
    int j = 0;
    while (j + 1 < plan.n && plan.b[j + 1].task_begin <= task) ++j;
    const StaticBuf& b = plan.b[j];
    const uint32_t local = task - b.task_begin;
    const uint64_t c0 = static_cast<uint64_t>(local) << g;
    const uint64_t c1 = min(c0 + (1ull << g), static_cast<unsigned long long>(b.n_chunks));
    uint64_t mine = 0;  // lane j keeps the hash of chunk c0 + j
    for (uint64_t c = c0; c < c1; ++c) {
      uint64_t h = fmix(kSeed ^ (c * 32u + lane));
#pragma unroll
      for (int k = 0; k < kSegs; ++k) {
        const uint64_t off = c * kChunkBytes + 512u * k + 16u * lane;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (off < b.bytes) {
          const uint64_t left = b.bytes - off;
          if (left >= 16 && b.align == 16) v = ld_stream(b.ptr + off);
          else v = ld_small(b.ptr + off, left < 16 ? static_cast<int>(left) : 16, b.align >= 4);
        }
        h = absorb(h, v);
      }
      const uint64_t x = __shfl_sync(kFull, warp_tree(fmix(h), 32, lane), 0);
      if (lane == static_cast<int>(c - c0)) mine = x;
    }
    const uint64_t root = warp_tree(mine, static_cast<int>(c1 - c0), lane);
    if (lane == 0) nodes[b.task_begin + local] = root;
  }
}

__global__ void __launch_bounds__(kThreads)
    k_fp_static_final(const StaticPlan plan, uint64_t* nodes, uint64_t* __restrict__ fp_out) {
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (i >= plan.n) return;
  const StaticBuf& b = plan.b[i];
  const uint64_t root = warp_tree_inplace(nodes + b.task_begin, b.n_tasks, lane);
  if (lane == 0) fp_out[i] = fmix(root ^ (b.bytes * kP));
}

}  // namespace

cudaError_t static_scratch(uint64_t** nodes) {
  static std::mutex mu;
  static uint64_t* addr[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_nodes);
    if (e != cudaSuccess) return e;
    addr[dev] = static_cast<uint64_t*>(p);
  }
  *nodes = addr[dev];
  return cudaSuccess;
}

cudaError_t launch_fingerprint_static(const StaticPlan& plan, uint64_t* nodes, uint64_t* fp_out,
                                      cudaStream_t stream) {
  if (plan.n <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const uint64_t want = (static_cast<uint64_t>(plan.n_tasks) + kWarps - 1) / kWarps;
  const uint64_t cap = static_cast<uint64_t>(sms) * 4;
  const int blocks = static_cast<int>(want < cap ? (want ? want : 1) : cap);
  k_fp_static<<<blocks, kThreads, 0, stream>>>(plan, nodes);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_fp_static_final<<<(plan.n + kWarps - 1) / kWarps, kThreads, 0, stream>>>(plan, nodes, fp_out);
  return cudaGetLastError();
}

}  // namespace pcs
