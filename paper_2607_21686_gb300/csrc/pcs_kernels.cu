// pcs_kernels.cu -- sm_103a kernels of the PCS hot path.
//
// k_stream<MODE>  one pass over 4 KiB chunks of many byte streams: a warp owns
//                 a task of 2^g chunks; lane l moves the 16-byte segments
//                 l + 32k of each chunk (every warp access is 512 contiguous
//                 bytes), optionally gathers / scatters them through a row or
//                 paged-ring layout, and folds them into the PCSFP64-v1 lane
//                 chain; a shuffle tree makes the chunk hash and then the
//                 task's aligned-group node (Sec. 4 FINGERPRINT, step 1).
// k_finalize<MODE> trees the task nodes of each stream into its fingerprint and
//                 writes outputs: fps / classification flags, record headers
//                 and section tables (checkpoint, Sec. 3 "The contract", I4),
//                 or the verification verdict of a restore (I1).
// k_score         cos(query, key) per bank entry, fp32, fixed order (Sec. 5).
// k_topk          per-bank radix select of the k largest (score, -index),
//                 kept indices written in ascending order (Sec. 7.5).
// k_copy          fork: independent copy of a record (I3).
//
// No kernel waits on another block: every pass is a plain data-parallel
// sweep, so nothing here can spin.  Index values read from device memory are
// bounds-checked; a bad one is reported through the error word and skipped.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

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

template <int MODE>
__global__ void __launch_bounds__(kThreads, 2)
    k_stream(const SecDesc* __restrict__ secs, int n_secs, uint32_t n_tasks, int glog2,
             uint64_t* __restrict__ nodes, uint32_t* err) {
  using T = ModeTraits<MODE>;
  __shared__ SecDesc sdesc[kWarps];
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const uint32_t nw = gridDim.x * kWarps;
  int cur = -1;
  for (uint32_t task = blockIdx.x * kWarps + wib; task < n_tasks; task += nw) {
    // The stream owning this task: last i with task_begin <= task.
    int lo = 0, hi = n_secs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(&secs[mid].task_begin) <= task) lo = mid;
      else hi = mid - 1;
    }
    if (lo != cur) {
      __syncwarp();
      if (lane < static_cast<int>(sizeof(SecDesc) / 16))
        reinterpret_cast<uint4*>(&sdesc[wib])[lane] =
            __ldg(reinterpret_cast<const uint4*>(&secs[lo]) + lane);
      __syncwarp();
      cur = lo;
    }
    const SecDesc& s = sdesc[wib];
    const uint64_t c0 = static_cast<uint64_t>(task - s.task_begin) << glog2;
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
        uint64_t hb = fmix(kSeed ^ ((c + 1) * 32u + lane));
#pragma unroll
        for (int k = 0; k < kSegs; ++k) ha = absorb(ha, va[k]);
        if (two) {
#pragma unroll
          for (int k = 0; k < kSegs; ++k) hb = absorb(hb, vb[k]);
        }
        ha = warp_tree(fmix(ha), 32, lane);
        hb = warp_tree(fmix(hb), 32, lane);
        ha = __shfl_sync(kFull, ha, 0);
        hb = __shfl_sync(kFull, hb, 0);
        const int j = static_cast<int>(c - c0);
        if (lane == j) mine = ha;
        if (two && lane == j + 1) mine = hb;
      }
    }
    if (T::kHash) {
      const uint64_t root = warp_tree(mine, static_cast<int>(c1 - c0), lane);
      if (lane == 0) nodes[task] = root;
    }
  }
}

// ---------------------------------------------------------------------------
// Finalisation: stream fps, record headers, verification
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint64_t stream_fp(const SecDesc& s, uint64_t* nodes, int lane) {
  const uint64_t root = warp_tree_inplace(nodes + s.task_begin, s.n_tasks, lane);
  return fmix(root ^ (s.bytes * kP));
}

// Fingerprints of independent buffers (pcs_fingerprint / pcs_classify).
__global__ void __launch_bounds__(kThreads)
    k_finalize_hash(const SecDesc* __restrict__ secs, int n_secs, uint64_t* nodes,
                    uint64_t* fp_out, const uint64_t* fp_before, uint8_t* flags) {
  const int lane = threadIdx.x & 31;
  const int nw = gridDim.x * kWarps;
  for (int i = blockIdx.x * kWarps + (threadIdx.x >> 5); i < n_secs; i += nw) {
    const SecDesc s = secs[i];
    const uint64_t fp = stream_fp(s, nodes, lane);
    if (lane == 0) {
      if (fp_out) fp_out[i] = fp;
      if (fp_before) flags[i] = fp != fp_before[i] ? 1 : 0;
    }
  }
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
template <int MODE>
__global__ void __launch_bounds__(kThreads)
    k_finalize_sessions(const SecDesc* __restrict__ secs, const SessDesc* __restrict__ sess,
                        int n_sess, const Entry* __restrict__ entries, uint64_t* nodes,
                        uint8_t* corrupt, uint32_t* bad) {
  __shared__ uint64_t smem[kMaxSmemFps];
  __shared__ uint32_t s_bad;
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  for (int b = blockIdx.x; b < n_sess; b += gridDim.x) {
    const SessDesc S = sess[b];
    Entry* table = reinterpret_cast<Entry*>(S.record + kHeaderBytes);
    if (threadIdx.x == 0) s_bad = 0;
    __syncthreads();
    for (uint32_t j = wib; j < S.n_sections; j += kWarps) {
      const SecDesc s = secs[S.sec_begin + j];
      const uint64_t fp = stream_fp(s, nodes, lane);
      if (MODE == kModePack) {
        // Lanes 0..3 write the 64-byte entry as four 16-byte words.
        if (lane < 4) {
          Entry e = entries[S.sec_begin + j];
          e.fp = fp;
          reinterpret_cast<uint4*>(&table[j])[lane] = reinterpret_cast<const uint4*>(&e)[lane];
        }
      } else {
        if (lane == 0 && table[j].fp != fp) atomicOr(&s_bad, 1u);
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
          const bool broken = s_bad != 0 || stored != sfp;
          if (corrupt) corrupt[b] = broken ? 1 : 0;
          if (broken) atomicAdd(bad, 1u);
        }
      }
    }
    if (MODE == kModePack) {
      // Zero the gap between the end of the table and the first payload.
      const uint64_t from = kHeaderBytes + static_cast<uint64_t>(kEntryBytes) * S.n_sections;
      for (uint64_t o = from + 16u * threadIdx.x; o < S.payload_start; o += 16u * kThreads)
        *reinterpret_cast<uint4*>(S.record + o) = make_uint4(0, 0, 0, 0);
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Relevance score and top-k
// ---------------------------------------------------------------------------

__device__ __forceinline__ float elem(uint32_t bits16, bool bf16) {
  return bf16 ? __uint_as_float(bits16 << 16)
              : __half2float(__ushort_as_half(static_cast<unsigned short>(bits16)));
}

// Accumulate the 8 elements of one 16-byte segment, ascending element order,
// with separately rounded products and sums.
__device__ __forceinline__ void accum8(uint4 q, uint4 k, bool bf16, float& sd, float& sq,
                                       float& sk) {
  const uint32_t qw[4] = {q.x, q.y, q.z, q.w};
  const uint32_t kw[4] = {k.x, k.y, k.z, k.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t qb = (qw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
    const uint32_t kb = (kw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
    const float qe = elem(qb, bf16), ke = elem(kb, bf16);
    sd = __fadd_rn(sd, __fmul_rn(qe, ke));
    sq = __fadd_rn(sq, __fmul_rn(qe, qe));
    sk = __fadd_rn(sk, __fmul_rn(ke, ke));
  }
}

__device__ __forceinline__ float lane_tree_sum(float v) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) v = __fadd_rn(v, __shfl_down_sync(kFull, v, d));
  return v;
}

__global__ void __launch_bounds__(kThreads)
    k_score(const BankDesc* __restrict__ banks, int n_banks, uint64_t n_entries,
            float* __restrict__ scores) {
  const int lane = threadIdx.x & 31;
  const uint64_t nw = static_cast<uint64_t>(gridDim.x) * kWarps;
  int cur = -1;
  BankDesc B{};
  for (uint64_t e = static_cast<uint64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5); e < n_entries;
       e += nw) {
    int lo = 0, hi = n_banks - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(&banks[mid].entry_begin) <= e) lo = mid;
      else hi = mid - 1;
    }
    if (lo != cur) {
      B = banks[lo];
      cur = lo;
    }
    const uint64_t i = e - B.entry_begin;
    const bool bf16 = B.is_bf16 != 0;
    const int segs = B.D / 8;
    const uint8_t* krow = reinterpret_cast<const uint8_t*>(B.keys) + i * static_cast<uint64_t>(B.D) * 2;
    const uint8_t* qrow = reinterpret_cast<const uint8_t*>(B.query);
    float sd = 0.f, sq = 0.f, sk = 0.f;
    for (int t = lane; t < segs; t += 32) {
      const uint4 kv = ld_stream(krow + 16 * t);
      const uint4 qv = __ldg(reinterpret_cast<const uint4*>(qrow) + t);
      accum8(qv, kv, bf16, sd, sq, sk);
    }
    sd = lane_tree_sum(sd);
    sq = lane_tree_sum(sq);
    sk = lane_tree_sum(sk);
    if (lane == 0) {
      const float den = __fmul_rn(__fsqrt_rn(sq), __fsqrt_rn(sk));
      scores[e] = den == 0.f ? 0.f : __fdiv_rn(sd, den);
    }
  }
}

__device__ __forceinline__ uint32_t ord32(float s) {
  if (isnan(s)) return 0u;
  if (s == 0.f) s = 0.f;
  const uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
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

__global__ void __launch_bounds__(kThreads)
    k_topk(const BankDesc* __restrict__ banks, int n_banks, const float* __restrict__ scores,
           int32_t* __restrict__ kept_idx) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t warp_cnt[kWarps];
  __shared__ uint32_t s_prefix, s_mask, s_remaining;
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
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
      if (wib == 0) {
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
        const uint32_t remaining = s_remaining;
        const unsigned hit = __ballot_sync(kFull, incl >= remaining);
        const int first = __ffs(hit) - 1;  // remaining <= count, so hit != 0
        if (lane == first) {
          uint32_t cum = incl - local;
          for (int j = 0; j < 8; ++j) {
            const int bin = 255 - 8 * lane - j;
            if (cum + hist[bin] >= remaining) {
              s_prefix = prefix | (static_cast<uint32_t>(bin) << shift);
              s_mask = mask | (0xFFu << shift);
              s_remaining = remaining - cum;
              break;
            }
            cum += hist[bin];
          }
        }
      }
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
// Fork copy
// ---------------------------------------------------------------------------

__global__ void __launch_bounds__(kThreads)
    k_copy(const uint4* __restrict__ src, uint4* __restrict__ dst, uint64_t n16) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kThreads;
  uint64_t i = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x;
  for (; i + 3 * stride < n16; i += 4 * stride) {
    const uint4 a = __ldcs(src + i), b = __ldcs(src + i + stride);
    const uint4 c = __ldcs(src + i + 2 * stride), d = __ldcs(src + i + 3 * stride);
    __stcs(dst + i, a);
    __stcs(dst + i + stride, b);
    __stcs(dst + i + 2 * stride, c);
    __stcs(dst + i + 3 * stride, d);
  }
  for (; i < n16; i += stride) __stcs(dst + i, __ldcs(src + i));
}

template <int MODE>
int occupancy() {
  int b = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_stream<MODE>, kThreads, 0);
  return b > 0 ? b : 1;
}

}  // namespace

int stream_blocks_per_sm() { return occupancy<kModePack>(); }

cudaError_t launch_stream(int mode, const SecDesc* secs, int n_secs, uint32_t n_tasks,
                          int group_log2, uint64_t* nodes, uint32_t* dev_err, int sm_count,
                          int blocks_per_sm, cudaStream_t stream) {
  if (n_tasks == 0) return cudaSuccess;
  const uint64_t want = (static_cast<uint64_t>(n_tasks) + kWarps - 1) / kWarps;
  const int blocks = static_cast<int>(
      want < static_cast<uint64_t>(sm_count) * blocks_per_sm ? want
                                                            : static_cast<uint64_t>(sm_count) * blocks_per_sm);
  switch (mode) {
    case kModeHash:
      k_stream<kModeHash><<<blocks, kThreads, 0, stream>>>(secs, n_secs, n_tasks, group_log2, nodes, dev_err);
      break;
    case kModePack:
      k_stream<kModePack><<<blocks, kThreads, 0, stream>>>(secs, n_secs, n_tasks, group_log2, nodes, dev_err);
      break;
    case kModeRestore:
      k_stream<kModeRestore><<<blocks, kThreads, 0, stream>>>(secs, n_secs, n_tasks, group_log2, nodes, dev_err);
      break;
    case kModeRestoreV:
      k_stream<kModeRestoreV><<<blocks, kThreads, 0, stream>>>(secs, n_secs, n_tasks, group_log2, nodes, dev_err);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_finalize(int mode, const SecDesc* secs, const SessDesc* sess, int n_sess,
                            const Entry* entries, uint64_t* nodes, uint64_t* fp_out,
                            const uint64_t* fp_before, uint8_t* flags, uint32_t* bad,
                            cudaStream_t stream) {
  if (n_sess <= 0) return cudaSuccess;
  if (mode == kModeHash) {
    const int blocks = (n_sess + kWarps - 1) / kWarps;
    k_finalize_hash<<<blocks < 4096 ? blocks : 4096, kThreads, 0, stream>>>(secs, n_sess, nodes, fp_out,
                                                                            fp_before, flags);
  } else if (mode == kModePack) {
    k_finalize_sessions<kModePack><<<n_sess < 65535 ? n_sess : 65535, kThreads, 0, stream>>>(
        secs, sess, n_sess, entries, nodes, flags, bad);
  } else if (mode == kModeRestoreV) {
    k_finalize_sessions<kModeRestoreV><<<n_sess < 65535 ? n_sess : 65535, kThreads, 0, stream>>>(
        secs, sess, n_sess, entries, nodes, flags, bad);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_score(const BankDesc* banks, int n_banks, uint64_t n_entries,
                         const uint64_t* /*entry_begin_sorted*/, float* scores, int sm_count,
                         cudaStream_t stream) {
  if (n_entries == 0) return cudaSuccess;
  const uint64_t want = (n_entries + kWarps - 1) / kWarps;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * 8;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  k_score<<<blocks, kThreads, 0, stream>>>(banks, n_banks, n_entries, scores);
  return cudaGetLastError();
}

cudaError_t launch_topk(const BankDesc* banks, int n_banks, const float* scores,
                        int32_t* kept_idx, cudaStream_t stream) {
  if (n_banks <= 0) return cudaSuccess;
  k_topk<<<n_banks < 65535 ? n_banks : 65535, kThreads, 0, stream>>>(banks, n_banks, scores,
                                                                     kept_idx);
  return cudaGetLastError();
}

cudaError_t launch_copy(const void* src, void* dst, uint64_t bytes, int sm_count,
                        cudaStream_t stream) {
  const uint64_t n16 = bytes / 16;
  if (n16 == 0) return cudaSuccess;
  const uint64_t want = (n16 + kThreads - 1) / kThreads;
  const uint64_t cap = static_cast<uint64_t>(sm_count) * 8;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  k_copy<<<blocks, kThreads, 0, stream>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst), n16);
  return cudaGetLastError();
}

}  // namespace pcs
