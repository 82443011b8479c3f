// Device-side building blocks shared by the attention and acceptance kernels:
// mbarrier and bulk-copy wrappers with bounded waits, the split-KV work
// partition over all (sequence, head) key ranges, and the log-sum-exp merge
// of partial softmax results.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace glide {

constexpr uint32_t kStatusTimeout = 4;          // GLIDE_ERR_DEVICE_TIMEOUT
constexpr uint64_t kWaitLimitNs = 1000000000ull; // 1 s: far beyond any legitimate wait
constexpr float kLog2e = 1.4426950408889634f;

// ---------------------------------------------------------------- workspace
// Attention workspace: [0,256) header (the status word at byte 0; the
// cross-attention chunk-claim counter at byte 128 and its CTA-done counter at
// byte 192); then per-(b,h) arrival counters (4 bytes each, tree kernels);
// then per-(b,h) chunk ranges (8 bytes each, cross-attention scratch); then
// 256-aligned partial slots of nq*(D+2) floats.
struct WsLayout {
  static constexpr size_t kHeader = 256;
  static constexpr size_t kClaimOff = 128;
  static constexpr size_t kDoneOff = 192;
  static __host__ __device__ size_t align(size_t x) { return (x + 255) & ~size_t(255); }
  static __host__ __device__ size_t counters_off() { return kHeader; }
  static __host__ __device__ size_t ranges_off(int B, int H) {
    return align(kHeader + sizeof(unsigned) * (size_t)B * H);
  }
  static __host__ __device__ size_t partials_off(int B, int H) {
    return align(ranges_off(B, H) + 2 * sizeof(int) * (size_t)B * H);
  }
};

// -------------------------------------------------------------------- misc
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void record_status(unsigned* status, unsigned code) {
  atomicCAS(status, 0u, code);
}

// bf16 pair (one 32-bit word, element 0 in the low half) -> two floats.
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// --------------------------------------------- programmatic dependent launch
// Every kernel of the path is launched as a programmatic dependent of the
// kernel before it in the stream (launch_pdl): its CTAs may be scheduled as
// the CTAs of that kernel exit, before the whole grid has completed and its
// writes have been flushed, so the launch latency hides behind that kernel's
// tail.  pdl_wait() blocks until the previous grid has completed and its
// writes are visible; a kernel calls it before its first global-memory access
// and before it allocates tensor memory, so it never reads an input early nor
// holds resources the previous grid could wait for.  Only the two split-merge
// kernels signal their dependents early (griddepcontrol.launch_dependents, at
// their start): the next attention kernel's CTAs are then placed on the SMs
// the small merge grid leaves free and wait there, so its launch overlaps the
// merge (batch-1 Vicuna-7B round 93.8 -> 91.5 us).  An early signal from the
// attention kernels, which fill every SM, slowed them instead (dependents
// resident next to a running kernel: one 7B chain round 115 us without the
// signal, 128 us with it in every kernel, 142 us with no programmatic launch).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking probe: has the phase of `bar` with this parity completed?
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `bar` with the given parity to complete.  Gives up
// after limit_ns (default kWaitLimitNs), or at once when another thread of the
// CTA has set *abort; on giving up it records the timeout, sets *abort and
// returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          unsigned* status, uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (global_timer_ns() - t0 > limit_ns) {
      *abort = 1;
      record_status(status, kStatusTimeout);
      return false;
    }
  }
}

// Waits on the phase of `bar` with `parity`, bounded by time only (used to
// drain copies still in flight after an abort).
__device__ inline void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) return;
  }
}

// ------------------------------------------------------------- bulk copies
// 1-D bulk copy global -> this CTA's shared memory, completing `bytes` of
// transaction count on `bar`.  dst, src and bytes must be multiples of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// Named barrier among the `nthreads` consumer threads (id 1; id 0 is __syncthreads).
__device__ __forceinline__ void consumer_sync(int nthreads) {
  asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
}

// --------------------------------------------------------------- partition
// Every (b, h) owns a run of `ntiles(b)` consecutive tiles in one global
// sequence (b-major, then h, then key tile).  The G CTAs of a launch take
// equal contiguous shares of that sequence (sizes differ by at most one), so
// ragged batches stay balanced.  A CTA's share is cut into segments at (b, h)
// boundaries.  Tiles cover keys [t*TK, t*TK + TK) of a slab.
struct Partition {
  long long total;
  long long base;
  long long rem;
  int G;
  __device__ void init(long long total_tiles, int grid) {
    total = total_tiles;
    G = grid;
    base = total / grid;
    rem = total % grid;
  }
  __device__ long long begin(int c) const { return (long long)c * base + (c < rem ? c : rem); }
  __device__ long long end(int c) const { return begin(c) + base + (c < rem ? 1 : 0); }
  __device__ int cta_of(long long g) const {
    const long long big = rem * (base + 1);
    if (g < big) return (int)(g / (base + 1));
    return (int)(rem + (g - big) / base);
  }
};

// Per-sequence tile bookkeeping kept in shared memory.
struct BatchTiles {
  long long* start;  // [B+1]: first global tile of sequence b (over all its heads)
  int* len;          // [B]  : keys attended per slab (prefix, plus tree nodes)
  int* ntiles;       // [B]  : tiles per (b, h)
  int* plen;         // [B]  : clamped prefix length kv_len[b]
  int* sidx = nullptr;  // [B+1]: slabs with tiles before sequence b (filled when set)
};

// Fills BatchTiles (all threads of the block must call; ends with __syncthreads).
// keys(b) = clamp(kv_len[b], 0, max_kv_len) + extra.
__device__ inline void build_batch_tiles(BatchTiles bt, const int* kv_len, int B, int H,
                                         int max_kv_len, int extra, int TK) {
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    int L = kv_len[b];
    L = L < 0 ? 0 : (L > max_kv_len ? max_kv_len : L);
    bt.plen[b] = L;
    bt.len[b] = L + extra;
    bt.ntiles[b] = (L + extra + TK - 1) / TK;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    long long s = 0;
    int k = 0;
    for (int b = 0; b < B; ++b) {
      bt.start[b] = s;
      s += (long long)H * bt.ntiles[b];
      if (bt.sidx) {
        bt.sidx[b] = k;
        if (bt.ntiles[b] > 0) k += H;
      }
    }
    bt.start[B] = s;
    if (bt.sidx) bt.sidx[B] = k;
  }
  __syncthreads();
}

// A split of the tile sequence into G shares that charges every switch from
// one (b, h) slab to the next as w tiles of work: a share that spans k slabs
// pays for k - 1 switches (a segment epilogue and the start of the next
// segment), so shares with more segments get fewer tiles and all shares take
// about the same time.  Tile g of the s-th slab with tiles sits at position
// g + w * s of a cost line [0, C), C = tiles + w * (slabs - 1); the line is
// split into G equal parts (sizes differ by at most one) and a share holds
// the tiles whose positions fall in its part.  Needs bt.sidx.  The caller
// keeps tiles + w * slabs below 2^31, so the arithmetic is 32-bit.  Plain
// arithmetic on the table only, so the host can check it too.
struct CostPartition {
  BatchTiles bt;
  int B, G, H, w, C, base, rem, T;
  __host__ __device__ void init(const BatchTiles& t, int nb, int nh, int grid, int weight) {
    bt = t;
    B = nb;
    H = nh;
    G = grid;
    w = weight;
    T = (int)bt.start[B];
    const int S = bt.sidx[B];
    C = T + (S > 0 ? w * (S - 1) : 0);
    base = C / G;
    rem = C - base * G;
  }
  // position of the first tile of sequence b, if b has tiles
  __host__ __device__ int seq_pos(int b) const { return (int)bt.start[b] + w * bt.sidx[b]; }
  __host__ __device__ int part_begin(int c) const { return c * base + (c < rem ? c : rem); }
  // the first tile at a position >= v (T if none)
  __host__ __device__ long long tile_at(int v) const {
    if (v >= C) return T;
    int lo = 0, hi = B - 1;  // last b with seq_pos(b) <= v: a sequence with tiles
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (seq_pos(mid) <= v) lo = mid; else hi = mid - 1;
    }
    const int nt = bt.ntiles[lo];
    const int off = v - seq_pos(lo);
    int h = nt > 0 ? off / (nt + w) : 0;
    if (h > H - 1) h = H - 1;
    const int r = off - h * (nt + w);
    const int g0 = (int)bt.start[lo] + h * nt;
    return r < nt ? g0 + r : g0 + nt;  // a position between two slabs: the next slab's first tile
  }
  __host__ __device__ long long begin(int c) const { return tile_at(part_begin(c)); }
  __host__ __device__ long long end(int c) const { return tile_at(part_begin(c + 1)); }
  __host__ __device__ int cta_of(long long g64) const {
    const int g = (int)g64;
    int lo = 0, hi = B - 1;  // the sequence of tile g
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int)bt.start[mid] <= g) lo = mid; else hi = mid - 1;
    }
    const int h = (g - (int)bt.start[lo]) / bt.ntiles[lo];
    const int v = g + w * (bt.sidx[lo] + h);
    const int big = rem * (base + 1);
    if (v < big || base == 0) return v / (base + 1);
    return rem + (v - big) / base;
  }
};

// Dynamic work: the global tile sequence is cut into chunks of shrinking size
// that CTAs claim at run time.  Level 0 holds the first half of the tiles in
// G equal chunks, level 1 half of the rest in G chunks, and so on; the last
// level takes what remains.  The big early chunks keep claims few; the small
// late ones let the CTAs that stream faster take more of the work, so all of
// them finish close together.  Levels are dropped until every chunk of every
// level has at least kMinChunk tiles (fewer, smaller chunks only add partial
// results to merge) or one level is left; with one level an empty chunk
// (tiles < G) can only sit at the very end of the sequence, never inside a
// (b, h).  cta_of() names the chunk that holds a tile, which is what the
// split-merge bookkeeping needs.
constexpr int kMaxLevels = 6;
constexpr long long kMinChunk = 16;
struct Chunks {
  long long lo[kMaxLevels + 1];
  long long base[kMaxLevels];  // tiles per chunk of level l (size / G) ...
  int rem[kMaxLevels];         // ... and the first rem[l] chunks hold one more
  int G, L;
  // Built by lanes 0 .. kMaxLevels - 1 of one warp together (every lane of
  // that warp must call).  Level l's remainder r_l = total - lo[l] is
  // ceil(total / 2^l) (l halvings with the ceiling are one shift), and level
  // sizes never grow from one level to the next, so the levels that fit are a
  // prefix that one ballot counts; each lane then fills its own level, and the
  // per-level divisions run side by side.
  __device__ void init_warp(long long total, int grid, int levels, int lane) {
    const int Lmax = levels < 1 ? 1 : (levels > kMaxLevels ? kMaxLevels : levels);
    const int l = lane < kMaxLevels ? lane : kMaxLevels - 1;
    const long long r = (total + (1ll << l) - 1) >> l;
    // L levels fit when level L - 2 (the smallest halved one) holds G * kMinChunk tiles
    const bool fits = lane <= Lmax - 2 && (r >> 1) >= (long long)grid * kMinChunk;
    const int nl = 1 + __popc(__ballot_sync(0xffffffffu, fits));
    if (lane < nl) {
      lo[lane] = total - r;
      const long long size = lane == nl - 1 ? r : (r >> 1);
      base[lane] = size / grid;
      rem[lane] = (int)(size - base[lane] * grid);
    }
    if (lane == 0) {
      lo[nl] = total;
      G = grid;
      L = nl;
    }
  }
  __device__ int count() const { return G * L; }
  __device__ long long begin(int k) const {
    const int l = k / G, j = k - l * G;
    if (l >= L) return lo[L];
    return lo[l] + (long long)j * base[l] + (j < rem[l] ? j : rem[l]);
  }
  __device__ long long end(int k) const { return begin(k + 1); }
  __device__ int cta_of(long long g) const {
    int l = 0;
    while (l + 1 < L && g >= lo[l + 1]) ++l;
    const long long off = g - lo[l];
    const long long big = (long long)rem[l] * (base[l] + 1);
    const long long j = off < big ? off / (base[l] + 1) : rem[l] + (off - big) / base[l];
    return l * G + (int)j;
  }
};

struct Segment {
  int b, h;
  int t0, t1;          // tile range within the (b, h) slab, [t0, t1)
  long long g_end;     // global index one past the segment
  int c_first, c_last; // CTAs that share this (b, h)
};

// Locates the segment that starts at global tile g (< g_limit, the end of the
// CTA's share or chunk).  Part is Partition or Chunks: c_first / c_last name
// the shares (chunks) that hold the (b, h)'s first and last tile.
template <class Part>
__device__ inline Segment locate(const BatchTiles& bt, const Part& P, int B, long long g, long long g_limit) {
  int lo = 0, hi = B - 1;  // last b with start[b] <= g
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (bt.start[mid] <= g) lo = mid; else hi = mid - 1;
  }
  Segment s;
  s.b = lo;
  const int nt = bt.ntiles[lo];
  const long long off = g - bt.start[lo];
  s.h = (int)(off / nt);
  s.t0 = (int)(off % nt);
  const long long bh_begin = bt.start[lo] + (long long)s.h * nt;
  const long long bh_end = bh_begin + nt;
  s.g_end = bh_end < g_limit ? bh_end : g_limit;
  s.t1 = s.t0 + (int)(s.g_end - g);
  s.c_first = P.cta_of(bh_begin);
  s.c_last = P.cta_of(bh_end - 1);
  return s;
}

// ------------------------------------------------------------------ merging
// A partial softmax result over some keys, in the log2 domain: scores were
// pre-multiplied by scale*log2(e); m = max, l = sum 2^(s - m), o = sum 2^(s - m) v.
// Slot layout: nq rows of [m, l, o_0 .. o_{D-1}].
__device__ __forceinline__ float* partial_slot(float* partials, int slot, int nq, int D) {
  return partials + (size_t)slot * nq * (D + 2);
}

}  // namespace glide
