// Greedy tree acceptance (Section 2's greedy "speculative decoding" rule on
// the token tree of CaPE's verification, Section 3.2).
//
// One launch does both steps:
// 1. argmax over the vocabulary of every (sequence, node) logits row, lowest
//    index among equal maxima.  Rows are cut into chunks of kChunk logits and
//    the chunks are dealt round-robin over a persistent grid (one CTA per SM):
//    CTA c takes chunks c, c + G, c + 2G, ...  A producer thread streams a
//    CTA's chunks with 1-D bulk copies (TMA) into a ring of kNS shared-memory
//    stages, so nearly all of the logits are in flight at once; stage s always
//    serves consumer warp s, which reduces the whole chunk (a float max over
//    each lane's float4 groups, loaded eight at a time into eight independent
//    chains, the index recovered from the winning group, then two redux
//    max reductions of a 64-bit key: order-preserving float bits above the
//    complemented index) and folds the key into the row's slot with atomicMax.
//    The logits are a plain HBM stream.
// 2. every chunk is counted into its sequence's counter (release fence, then
//    an acquire atomic; nothing waits).  The warp that completes a sequence's
//    count walks that tree: a node is accepted iff every edge on its root
//    path matches (draft token == parent's argmax); the deepest accepted node,
//    lowest index among equals, gives the path, its length and the bonus
//    token.  The walk is pointer jumping over the parent array in registers
//    (two nodes per lane, at most six shuffle rounds for up to 64 nodes),
//    which gives every node its acceptance, depth and ancestor set at once.
//    The warp then re-arms the slots and the counter.
// Because the chunk order is sequence-major and every CTA walks it in that
// order, sequence b's chunks are all read before sequence b + 1's, and warps
// count their chunks while they wait for the next one: the walks of the early
// sequences run while the later ones still stream.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kNW = 14;                       // consumer warps (14 stages of 16 KB fill the shared memory)
constexpr int kThreads = (kNW + 1) * 32;      // + one producer warp
constexpr int kChunk = 4096;                  // logits per chunk (16 KB)
constexpr int kNS = kNW;                      // ring stages: stage s serves consumer warp s only
constexpr int kGroups = kChunk / (4 * 32);    // float4 groups of a lane in a whole chunk
constexpr size_t kRingBytes = (size_t)kNS * kChunk * sizeof(float);
constexpr size_t kSmemBytes = kRingBytes + 2 * kNS * sizeof(uint64_t) + 16;
static_assert(kNS % kNW == 0, "a stage must always serve the same consumer warp");
static_assert(kMaxTree <= 64, "two tree nodes per lane");

struct AccParams {
  const int32_t* draft;
  const int32_t* parent;
  const float* logits;
  int32_t* path;
  int32_t* len;
  int32_t* bonus;
  unsigned* status;
  unsigned* counters;
  unsigned long long* slots;
  int B, n, V, splits;
  long long nchunks;  // B * n * splits
  int bulk;           // 1: rows start 16-byte aligned, chunks arrive by bulk copy; 0: consumers read global memory
};

__device__ __forceinline__ unsigned long long argmax_key(float f, int idx) {
  uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);  // -0 and +0 compare equal
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (unsigned long long)(0xffffffffu - (uint32_t)idx);
}

__device__ __forceinline__ int key_index(unsigned long long k) {
  return (int)(0xffffffffu - (uint32_t)(k & 0xffffffffull));
}

// Counter increment with acquire semantics: a thread that sees the final
// count also sees every slot update released before the other increments.
__device__ __forceinline__ unsigned atomic_add_acquire(unsigned* addr, unsigned v) {
  unsigned old;
  asm volatile("atom.acquire.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(addr), "r"(v) : "memory");
  return old;
}

// The warp's largest key (every lane gets it): two max reductions, the high
// words first, then the low words of the lanes that hold the largest high word.
__device__ __forceinline__ unsigned long long warp_max_key(unsigned long long k) {
  const uint32_t hi = (uint32_t)(k >> 32), lo = (uint32_t)k;
  const uint32_t mhi = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
  return ((unsigned long long)mhi << 32) | mlo;
}

// Release fence at GPU scope: the writes before it (and those seen through
// a warp barrier) are visible before any write after it.
__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

// One lane's part of a chunk in shared memory: the float4 groups lane,
// lane + 32, ... below n4 (all kGroups of them when kFull).  Groups are loaded
// eight at a time into eight independent chains (group i goes to chain
// i % 8); a strict comparison keeps the first group of each chain holding the
// chain's maximum, and the chains are combined lowest group first among equal
// maxima.  Returns the lane's maximum and the group holding its first
// occurrence (-1 when the lane has no group).
template <bool kFull>
__device__ __forceinline__ int scan_lane(const float4* s4, int n4, int lane, float& best) {
  constexpr int kC = 8;
  float acc[kC];
  int grp[kC];
#pragma unroll
  for (int j = 0; j < kC; ++j) {
    acc[j] = -__int_as_float(0x7f800000);
    grp[j] = -1;
  }
#pragma unroll
  for (int b = 0; b < kGroups / kC; ++b) {
    float4 v[kC];
#pragma unroll
    for (int j = 0; j < kC; ++j) {
      const int q = lane + 32 * (b * kC + j);
      if (kFull || q < n4) v[j] = s4[q];
    }
#pragma unroll
    for (int j = 0; j < kC; ++j) {
      const int q = lane + 32 * (b * kC + j);
      if (kFull || q < n4) {
        const float g = fmaxf(fmaxf(v[j].x, v[j].y), fmaxf(v[j].z, v[j].w));
        if (b == 0 || grp[j] < 0 || g > acc[j]) {
          acc[j] = g;
          grp[j] = b * kC + j;
        }
      }
    }
  }
  float m = acc[0];
  int gi = grp[0];
#pragma unroll
  for (int j = 1; j < kC; ++j)
    if (grp[j] >= 0 && (gi < 0 || acc[j] > m || (acc[j] == m && grp[j] < gi))) {
      m = acc[j];
      gi = grp[j];
    }
  best = m;
  return gi;
}

// Value of node `c`'s copy of a per-node quantity held two nodes per lane
// (v0 for node lane, v1 for node lane + 32).  All lanes must call.
__device__ __forceinline__ uint32_t gather(uint32_t v0, uint32_t v1, int c) {
  const uint32_t x0 = __shfl_sync(0xffffffffu, v0, c & 31);
  const uint32_t x1 = __shfl_sync(0xffffffffu, v1, c & 31);
  return c >= 32 ? x1 : x0;
}

// Per-node state of the walk, packed: bit 16 = every edge of the covered part
// of the root path matches, bits 8..15 = edges covered, bits 0..7 = the next
// ancestor still to cover + 1 (0: the root has been reached).
__device__ __forceinline__ uint32_t pack(bool ok, int d, int p) {
  return (ok ? 0x10000u : 0u) | ((uint32_t)d << 8) | (uint32_t)(p + 1);
}

// Walks sequence b's tree (one whole warp; every chunk of b has been counted,
// and the count that completed it was an acquire by one lane of this warp).
__device__ void walk_tree(const AccParams& p, int b, int lane) {
  __syncwarp();  // orders the other lanes' loads after that lane's acquire
  const int n = p.n;
  const size_t base = (size_t)b * n;
  const int c0 = lane, c1 = lane + 32;
  const bool h0 = c0 < n, h1 = c1 < n;
  const unsigned long long s0 = h0 ? __ldcg(&p.slots[base + c0]) : 0ull;
  const unsigned long long s1 = h1 ? __ldcg(&p.slots[base + c1]) : 0ull;
  const int par0 = h0 ? p.parent[base + c0] : -1, par1 = h1 ? p.parent[base + c1] : -1;
  const int dr0 = h0 ? p.draft[base + c0] : 0, dr1 = h1 ? p.draft[base + c1] : 0;
  const int a0 = key_index(s0), a1 = key_index(s1);  // argmax of each node's row

  // An edge matches when the node's draft token is its parent's argmax; a
  // parent outside [0, c) leaves the node unreachable.  The root always holds.
  const bool v0 = par0 >= 0 && par0 < c0, v1 = par1 >= 0 && par1 < c1;
  const int pa0 = (int)gather((uint32_t)a0, (uint32_t)a1, v0 ? par0 : 0);
  const int pa1 = (int)gather((uint32_t)a0, (uint32_t)a1, v1 ? par1 : 0);
  const bool ok0 = h0 && (c0 == 0 || (v0 && dr0 == pa0));
  const bool ok1 = h1 && v1 && dr1 == pa1;
  const int p0 = (c0 > 0 && ok0) ? par0 : -1, p1 = ok1 ? par1 : -1;
  uint32_t w0 = pack(ok0, p0 >= 0 ? 1 : 0, p0), w1 = pack(ok1, p1 >= 0 ? 1 : 0, p1);
  // ancestor-or-self sets (64-bit, low and high words)
  uint32_t m0l = h0 ? (1u << c0) : 0u, m0h = 0u;
  uint32_t m1l = 0u, m1h = h1 ? (1u << (c1 - 32)) : 0u;

  // Pointer jumping: each round doubles the covered part of every root path
  // (all lanes read the previous round's values); 2^6 = 64 > any depth, and
  // the rounds stop once every path has reached the root.
#pragma unroll 1
  for (int r = 0; r < 6; ++r) {
    const int q0 = (int)(w0 & 0xffu) - 1, q1 = (int)(w1 & 0xffu) - 1;
    if (!__any_sync(0xffffffffu, q0 >= 0 || q1 >= 0)) break;
    const int i0 = q0 < 0 ? 0 : q0, i1 = q1 < 0 ? 0 : q1;
    const uint32_t g0 = gather(w0, w1, i0), g1 = gather(w0, w1, i1);
    const uint32_t gl0 = gather(m0l, m1l, i0), gh0 = gather(m0h, m1h, i0);
    const uint32_t gl1 = gather(m0l, m1l, i1), gh1 = gather(m0h, m1h, i1);
    if (q0 >= 0) {
      w0 = pack((w0 & 0x10000u) && (g0 & 0x10000u), (int)((w0 >> 8) & 0xffu) + (int)((g0 >> 8) & 0xffu),
                (int)(g0 & 0xffu) - 1);
      m0l |= gl0;
      m0h |= gh0;
    }
    if (q1 >= 0) {
      w1 = pack((w1 & 0x10000u) && (g1 & 0x10000u), (int)((w1 >> 8) & 0xffu) + (int)((g1 >> 8) & 0xffu),
                (int)(g1 & 0xffu) - 1);
      m1l |= gl1;
      m1h |= gh1;
    }
  }
  const int d0 = (int)((w0 >> 8) & 0xffu), d1 = (int)((w1 >> 8) & 0xffu);
  // deepest accepted node, lowest index among equals (the root always qualifies)
  const unsigned k0 = (w0 & 0x10000u) ? ((unsigned)d0 << 8) | (unsigned)(255 - c0) : 0u;
  const unsigned k1 = (w1 & 0x10000u) ? ((unsigned)d1 << 8) | (unsigned)(255 - c1) : 0u;
  const unsigned key = __reduce_max_sync(0xffffffffu, k0 > k1 ? k0 : k1);
  const int node = 255 - (int)(key & 255u);
  const int depth = (int)(key >> 8);
  const uint32_t nl = gather(m0l, m1l, node), nh = gather(m0h, m1h, node);
  const int bonus = (int)gather((uint32_t)a0, (uint32_t)a1, node);

  // The path: node c of the chosen node's ancestor set sits at position depth(c).
  int32_t* out = p.path + base;
  if (h0 && ((nl >> c0) & 1u)) out[d0] = c0;
  if (h1 && ((nh >> (c1 - 32)) & 1u)) out[d1] = c1;
  if (h0 && c0 > depth) out[c0] = -1;
  if (h1 && c1 > depth) out[c1] = -1;
  if (lane == 0) {
    p.len[b] = depth;
    p.bonus[b] = bonus;
    p.counters[b] = 0u;
  }
  if (h0) p.slots[base + c0] = 0ull;
  if (h1) p.slots[base + c1] = 0ull;
}

__global__ void __launch_bounds__(kThreads, 1) tree_accept_kernel(const AccParams p) {
  extern __shared__ __align__(1024) unsigned char smem[];
  float* ring = reinterpret_cast<float*>(smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kRingBytes);
  uint64_t* empty = full + kNS;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kNS);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&full[s], 1);   // the producer's expect-tx arrival
      mbar_init(&empty[s], 1);  // the consumer warp's release
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  // Launched as a programmatic dependent: the inputs may come from the kernel
  // before this one, so nothing is read until that kernel has completed.
  pdl_wait();

  const long long G = gridDim.x, c = blockIdx.x;
  if (warp == kNW) {
    // ------------------------------------------------------------ producer
    // Lanes 1..31 put the trees into L2 for the walks; lane 0 streams chunks.
    if (lane > 0) {
      const long long lines = ((long long)p.B * p.n * 4 + 127) / 128;
      for (long long l = c * 31 + (lane - 1); l < lines; l += G * 31) {
        asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<const char*>(p.parent) + l * 128));
        asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<const char*>(p.draft) + l * 128));
      }
      return;
    }
    if (!p.bulk) return;
    const uint64_t pol = policy_evict_first();
    long long issued = 0;
    bool ok = true;
    for (long long k = c; k < p.nchunks; k += G, ++issued) {
      const int s = (int)(issued % kNS);
      const uint32_t use = (uint32_t)(issued / kNS);
      if (!mbar_wait(&empty[s], (use & 1u) ^ 1u, abort_flag, p.status)) { ok = false; break; }
      const long long row = k / p.splits;
      const int lo = (int)(k - row * p.splits) * kChunk;
      const int cnt = min(kChunk, p.V - lo);
      const uint32_t bytes = (uint32_t)cnt * 4u;
      mbar_arrive_expect_tx(&full[s], bytes);
      bulk_g2s(ring + (size_t)s * kChunk, p.logits + (size_t)row * p.V + lo, bytes, &full[s], pol);
    }
    if (!ok)  // let copies already issued land before the CTA exits
      for (long long j = (issued > kNS ? issued - kNS : 0); j < issued; ++j)
        mbar_drain(&full[j % kNS], (uint32_t)(j / kNS) & 1u);
    return;
  }

  // -------------------------------------------------------------- consumers
  // A warp folds each chunk's key into its row slot at once but counts its
  // chunks in later, in batches of up to 32 (one lane per chunk): one fence
  // and one round of parallel atomics per batch instead of a fence and an
  // atomic round trip per chunk.  A batch is counted when it is full, when
  // the warp's next chunk has not landed yet (the count then costs no time)
  // and after the warp's last chunk.
  const unsigned per_seq = (unsigned)(p.n * p.splits);
  int pend_seq = 0, npend = 0;  // lane i: the sequence of the warp's i-th uncounted chunk
  auto count_in = [&]() {
    __syncwarp();
    fence_acq_rel_gpu();  // release: the warp's slot updates are visible before any of its counts
    const bool mine = lane < npend;
    unsigned prev = 0;
    if (mine) prev = atomic_add_acquire(&p.counters[pend_seq], 1u);
    unsigned done = __ballot_sync(0xffffffffu, mine && prev == per_seq - 1);
    while (done) {  // sequences this batch completed: walk each with the whole warp
      const int l = __ffs(done) - 1;
      done &= done - 1;
      walk_tree(p, __shfl_sync(0xffffffffu, pend_seq, l), lane);
    }
    npend = 0;
  };
  long long use = 0;  // chunks this warp has taken from its stage
  for (long long j = warp; c + j * G < p.nchunks; j += kNW, ++use) {
    const long long k = c + j * G;
    const long long row = k / p.splits;
    const int lo = (int)(k - row * p.splits) * kChunk;
    const int cnt = min(kChunk, p.V - lo);
    float m = -__int_as_float(0x7f800000);  // -inf
    int idx = 0x7fffffff;                   // a lane that holds no logit never wins
    if (p.bulk) {
      if (npend > 0 && !mbar_test_wait(&full[warp], (uint32_t)(use & 1))) count_in();
      if (!mbar_wait(&full[warp], (uint32_t)(use & 1), abort_flag, p.status)) break;
      const float4* s4 = reinterpret_cast<const float4*>(ring + (size_t)warp * kChunk);
      const int n4 = cnt >> 2;  // cnt is a multiple of 4 in this mode
      float ma;
      const int ga = n4 == kChunk / 4 ? scan_lane<true>(s4, n4, lane, ma) : scan_lane<false>(s4, n4, lane, ma);
      if (ga >= 0) {  // the index inside the winning group
        const float4 v = s4[lane + 32 * ga];
        const int e = v.x == ma ? 0 : (v.y == ma ? 1 : (v.z == ma ? 2 : 3));
        m = ma;
        idx = lo + 4 * (lane + 32 * ga) + e;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[warp]);
    } else {
      const float* src = p.logits + (size_t)row * p.V + lo;
      if (lane < cnt) {
        m = __ldcs(src + lane);
        idx = lo + lane;
        for (int q = lane + 32; q < cnt; q += 32) {
          const float x = __ldcs(src + q);
          if (x > m) {
            m = x;
            idx = lo + q;
          }
        }
      }
    }
    const unsigned long long key = warp_max_key(argmax_key(m, idx));
    if (lane == 0) atomicMax(&p.slots[row], key);
    if (lane == npend) pend_seq = (int)(row / p.n);
    if (++npend == 32) count_in();
  }
  if (npend > 0) count_in();
}

size_t counters_bytes(int B) { return ((size_t)B * sizeof(unsigned) + 255) & ~size_t(255); }

}  // namespace

size_t accept_workspace_bytes(int B, int n) {
  return 256 + counters_bytes(B) + (size_t)B * n * sizeof(unsigned long long);
}

cudaError_t launch_tree_accept(const AcceptArgs& a, cudaStream_t st) {
  static int configured_dev = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_dev != dev) {
    e = cudaFuncSetAttribute(tree_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    configured_dev = dev;
  }
  AccParams p;
  p.draft = a.draft; p.parent = a.parent; p.logits = a.logits;
  p.path = a.path; p.len = a.len; p.bonus = a.bonus;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.counters = reinterpret_cast<unsigned*>(ws + 256);
  p.slots = reinterpret_cast<unsigned long long*>(ws + 256 + counters_bytes(a.B));
  p.B = a.B; p.n = a.n; p.V = a.V;
  p.splits = (a.V + kChunk - 1) / kChunk;
  p.nchunks = (long long)a.B * a.n * p.splits;
  p.bulk = ((a.V & 3) == 0 && (reinterpret_cast<uintptr_t>(a.logits) & 15u) == 0) ? 1 : 0;
  if ((long long)a.n * p.splits > 0x7fffffffLL) return cudaErrorInvalidValue;
  long long G = sm_count();
  if (G > p.nchunks) G = p.nchunks;
  return launch_pdl(tree_accept_kernel, dim3((unsigned)G), dim3(kThreads), kSmemBytes, st, p);
}

}  // namespace glide
