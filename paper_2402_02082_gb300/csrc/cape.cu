// CaPE confidence-aware proposal expansion (Section 3.2; the fixed-size
// variant of Section 4's ablation).
//
// For every sequence b and proposal position i the draft's distribution
// probs[b, i, :] gives x_{t+i} (its most probable token), the confidence
// p_i (that probability), K_i = S(p_i) and the expansion set X_i (the K_i most
// probable other tokens).  The expanded proposal is linearized into the token
// tree that tree_verify_attn and tree_accept take: node 0 = x_t, node i = x_{t+i}
// (parent i-1), then the sets in position order, each token a sibling of its
// position's proposal token (parent i-1).
//
// Ranking uses one 64-bit key per token: order-preserving float bits above
// the complemented token id, so the larger key is the larger probability and,
// among equal probabilities, the lower id.  S(p) needs at most 7 expansion
// tokens, so the 8 largest keys of a row decide everything.
//
// One launch, no waiting:
// 1. one CTA per chunk of kChunk probabilities of a row: every thread keeps a
//    sorted top-8 of its elements in registers, a warp merges its lanes' lists
//    with 8 rounds of "warp max, winner pops" (a 64-bit warp max is two
//    redux.sync), warp 0 merges the warps' lists the same way and stores the
//    chunk's top-8;
// 2. the CTA that completes a sequence's count (atomic counter over all of
//    the sequence's chunks) merges each row's chunk lists (one warp per row)
//    and builds the sequence's tree: the set sizes, the cap on verified
//    tokens, and the node arrays; it re-arms the counter.
// Publication is release/acquire: the chunk results are written, the writers
// meet at a warp barrier, and one thread fences (acq_rel, gpu scope) and
// counts; the completing CTA fences again before anyone reads them.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kTop = 8;          // the proposal token + at most 7 expansion tokens
constexpr int kChunk = 2048;     // probabilities per CTA (8 a thread: shorter insertion chains than 16)
constexpr int kPerThread = kChunk / kThreads;
static_assert(kPerThread % 4 == 0, "a thread's share is whole float4s");
constexpr int kMaxPos = kMaxTree - 1;  // gamma <= max_tokens <= 63

typedef unsigned long long u64;

struct CapeParams {
  const float* probs;
  const int32_t* root;
  int32_t* tokens;
  int32_t* parent;
  int32_t* n_nodes;
  float* conf;               // may be null
  unsigned* seq_counters;    // [B]
  u64* slots;                // [B * gamma, splits, kTop]
  int B, gamma, V, max_tokens, fixed_k, splits;
};

__device__ __forceinline__ u64 rank_key(float f, int idx) {
  uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);  // -0 and +0 rank equal
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((u64)u << 32) | (u64)(0xffffffffu - (uint32_t)idx);
}
__device__ __forceinline__ int key_token(u64 k) { return (int)(0xffffffffu - (uint32_t)(k & 0xffffffffull)); }
__device__ __forceinline__ float key_prob(u64 k) {
  uint32_t u = (uint32_t)(k >> 32);
  u = (u & 0x80000000u) ? (u & 0x7fffffffu) : ~u;
  return __uint_as_float(u);
}

// S(p) of Section 3.2: 7, 5, 3, 1 on (0, 0.3], (0.3, 0.6], (0.6, 0.8], (0.8, 1].
// 10 * p is exact in double (a 24-bit significand times a 4-bit integer), so
// the comparisons with 3, 6 and 8 are exact comparisons of p with the decimal
// thresholds.  p <= 0 falls in the first interval, p > 1 in the last.
__device__ __forceinline__ int expansion_size(float p) {
  const double x = 10.0 * (double)p;
  return x <= 3.0 ? 7 : (x <= 6.0 ? 5 : (x <= 8.0 ? 3 : 1));
}

// Insert k into the descending list t (registers after unrolling).
__device__ __forceinline__ void top_insert(u64 (&t)[kTop], u64 k) {
  if (k <= t[kTop - 1]) return;
  t[kTop - 1] = k;
#pragma unroll
  for (int j = kTop - 1; j > 0; --j) {
    const u64 hi = t[j] > t[j - 1] ? t[j] : t[j - 1];
    const u64 lo = t[j] > t[j - 1] ? t[j - 1] : t[j];
    t[j - 1] = hi;
    t[j] = lo;
  }
}

// Warp-wide max of a 64-bit key: the max of the high words, then the max of
// the low words among the lanes that hold it.
__device__ __forceinline__ u64 warp_max_u64(u64 v) {
  const unsigned hi = (unsigned)(v >> 32), lo = (unsigned)v;
  const unsigned mhi = __reduce_max_sync(0xffffffffu, hi);
  const unsigned mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
  return ((u64)mhi << 32) | mlo;
}

__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

// Merges the 32 lanes' descending lists into the warp's top-8 (warp-uniform
// result).  Keys are distinct except the zero filler, so one lane pops per round.
__device__ __forceinline__ void warp_top(u64 (&t)[kTop], u64 (&out)[kTop]) {
#pragma unroll
  for (int r = 0; r < kTop; ++r) {
    const u64 m = warp_max_u64(t[0]);
    out[r] = m;
    if (t[0] == m) {
#pragma unroll
      for (int j = 0; j < kTop - 1; ++j) t[j] = t[j + 1];
      t[kTop - 1] = 0ull;
    }
  }
}

__global__ void __launch_bounds__(kThreads) cape_expand_kernel(const CapeParams p) {
  __shared__ u64 red[kWarps][kTop];
  __shared__ int last_seq;
  // tree build (last CTA of a sequence)
  __shared__ u64 s_top[kMaxPos][kTop];         // per position: its row's 8 best keys
  __shared__ u64 s_cand[kMaxPos * kCapeMaxSet]; // expansion candidates, cap-order keys
  __shared__ unsigned char s_keepf[kMaxPos * kCapeMaxSet];  // candidate survives the cap
  __shared__ unsigned char s_k[kMaxPos];       // set size before the cap
  __shared__ unsigned char s_kept[kMaxPos];    // set size after the cap
  __shared__ int s_coff[kMaxPos];              // first candidate of each position
  __shared__ int s_off[kMaxPos];               // first node of each kept set, minus 1 + gamma
  __shared__ int s_ncand, s_nodes;
  pdl_wait();

  const int row = blockIdx.x / p.splits;
  const int split = blockIdx.x - row * p.splits;
  const int b = row / p.gamma;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // ---- 1. top-8 of this chunk
  {
    const float* pr = p.probs + (size_t)row * p.V;
    const int lo = split * kChunk;
    const int hi = min(p.V, lo + kChunk);
    u64 t[kTop];
#pragma unroll
    for (int j = 0; j < kTop; ++j) t[j] = 0ull;
    // all of this thread's loads first (one DRAM latency), then the inserts
    if ((p.V & 3) == 0) {
      const float4* v4 = reinterpret_cast<const float4*>(pr);
      const int lo4 = lo / 4 + threadIdx.x, hi4 = hi / 4;
      float4 x[kPerThread / 4];
#pragma unroll
      for (int u = 0; u < kPerThread / 4; ++u)
        if (lo4 + u * kThreads < hi4) x[u] = __ldcs(v4 + lo4 + u * kThreads);
#pragma unroll
      for (int u = 0; u < kPerThread / 4; ++u) {
        const int j = lo4 + u * kThreads;
        if (j < hi4) {
          top_insert(t, rank_key(x[u].x, 4 * j));
          top_insert(t, rank_key(x[u].y, 4 * j + 1));
          top_insert(t, rank_key(x[u].z, 4 * j + 2));
          top_insert(t, rank_key(x[u].w, 4 * j + 3));
        }
      }
    } else {
      float x[kPerThread];
#pragma unroll
      for (int u = 0; u < kPerThread; ++u)
        if (lo + threadIdx.x + u * kThreads < hi) x[u] = __ldcs(pr + lo + threadIdx.x + u * kThreads);
#pragma unroll
      for (int u = 0; u < kPerThread; ++u) {
        const int j = lo + threadIdx.x + u * kThreads;
        if (j < hi) top_insert(t, rank_key(x[u], j));
      }
    }
    u64 w[kTop];
    warp_top(t, w);
    if (lane == 0) {
#pragma unroll
      for (int j = 0; j < kTop; ++j) red[warp][j] = w[j];
    }
    __syncthreads();
    if (warp == 0) {
      u64 c[kTop];
#pragma unroll
      for (int j = 0; j < kTop; ++j) c[j] = 0ull;
      for (int e = lane; e < kWarps * kTop; e += 32) top_insert(c, red[e / kTop][e % kTop]);
      u64 ct[kTop];
      warp_top(c, ct);
      u64* slot = p.slots + ((size_t)row * p.splits + split) * kTop;
      if (lane < kTop) {
        u64 v = ct[0];
#pragma unroll
        for (int j = 1; j < kTop; ++j)
          if (lane == j) v = ct[j];
        __stcg(slot + lane, v);
      }
      __syncwarp();
      if (lane == 0) {
        fence_acq_rel_gpu();   // release: the slot writes of this warp (seen through the barrier)
        const unsigned prev = atomicAdd(&p.seq_counters[b], 1u);
        last_seq = (prev == (unsigned)(p.gamma * p.splits - 1)) ? 1 : 0;
        if (last_seq) fence_acq_rel_gpu();  // acquire: every chunk of the sequence
      }
    }
    __syncthreads();
    if (!last_seq) return;
  }

  // ---- 2. this CTA completed sequence b: merge each row, one warp per row
  const int G = p.gamma;
  for (int i = warp; i < G; i += kWarps) {
    u64 c[kTop];
#pragma unroll
    for (int j = 0; j < kTop; ++j) c[j] = 0ull;
    const u64* slots = p.slots + ((size_t)b * G + i) * p.splits * kTop;
    for (int e = lane; e < p.splits * kTop; e += 32) top_insert(c, __ldcg(slots + e));
    u64 rt[kTop];
    warp_top(c, rt);
    if (lane == 0) {
#pragma unroll
      for (int j = 0; j < kTop; ++j) s_top[i][j] = rt[j];
    }
  }
  __syncthreads();

  // ---- 3. set sizes, the cap, the node arrays
  for (int i = threadIdx.x; i < G; i += kThreads) {
    const float pi = key_prob(s_top[i][0]);
    int k = p.fixed_k >= 0 ? p.fixed_k : expansion_size(pi);
    k = min(k, p.V - 1);
    s_k[i] = (unsigned char)k;
    if (p.conf) p.conf[(size_t)b * G + i] = pi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int c = 0;
    for (int i = 0; i < G; ++i) {
      s_coff[i] = c;
      c += s_k[i];
    }
    s_ncand = c;
  }
  __syncthreads();
  // Candidate keys in cap order: probability, then the earlier position, then
  // the earlier rank (all distinct).
  for (int e = threadIdx.x; e < G * kCapeMaxSet; e += kThreads) {
    const int i = e / kCapeMaxSet, r = 1 + e % kCapeMaxSet;
    if (r <= s_k[i])
      s_cand[s_coff[i] + r - 1] = (s_top[i][r] & 0xffffffff00000000ull) | ((u64)(255 - i) << 8) | (u64)(255 - r);
  }
  __syncthreads();
  // With more candidates than room, a candidate is kept iff fewer than `room`
  // candidates come before it (one thread per candidate).  Kept sets are
  // prefixes of their positions, so a set's kept size is its count of kept flags.
  const int room = p.max_tokens - G;
  const int nc = s_ncand;
  for (int c = threadIdx.x; c < nc; c += kThreads) {
    unsigned char keep = 1;
    if (nc > room) {
      const u64 mine = s_cand[c];
      int ahead = 0;
      for (int q = 0; q < nc; ++q) ahead += s_cand[q] > mine ? 1 : 0;
      keep = ahead < room ? 1 : 0;
    }
    s_keepf[c] = keep;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < G; i += kThreads) {
    int kept = 0;
    for (int r = 0; r < s_k[i]; ++r) kept += s_keepf[s_coff[i] + r];
    s_kept[i] = (unsigned char)kept;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int off = 0;
    for (int i = 0; i < G; ++i) {
      s_off[i] = off;
      off += s_kept[i];
    }
    s_nodes = 1 + G + off;
    p.n_nodes[b] = s_nodes;
  }
  __syncthreads();
  const int n_out = 1 + p.max_tokens;
  int32_t* tok = p.tokens + (size_t)b * n_out;
  int32_t* par = p.parent + (size_t)b * n_out;
  for (int j = threadIdx.x; j < n_out; j += kThreads) {
    int t, q;
    if (j == 0) {
      t = p.root[b];
      q = -1;
    } else if (j <= G) {
      t = key_token(s_top[j - 1][0]);
      q = j - 1;
    } else if (j < s_nodes) {
      // the last position whose set starts at or before e (empty sets share
      // their successor's offset); e < s_off[i] + s_kept[i] follows
      const int e = j - 1 - G;
      int i = 0;
      while (i + 1 < G && s_off[i + 1] <= e) ++i;
      t = key_token(s_top[i][1 + e - s_off[i]]);
      q = i;
    } else {
      t = -1;
      q = 0;
    }
    tok[j] = t;
    par[j] = q;
  }
  if (threadIdx.x == 0) p.seq_counters[b] = 0u;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int cape_splits(int V) { return (V + kChunk - 1) / kChunk; }

}  // namespace

// Workspace: [0,256) status | sequence counters [B] | chunk slots
// [B*gamma, splits, 8] u64.
size_t cape_workspace_bytes(int B, int gamma, int V) {
  const size_t rows = (size_t)B * gamma;
  return 256 + align256((size_t)B * sizeof(unsigned)) + rows * (size_t)cape_splits(V) * kTop * sizeof(u64);
}

cudaError_t launch_cape_expand(const CapeArgs& a, cudaStream_t st) {
  CapeParams p;
  p.probs = a.probs; p.root = a.root;
  p.tokens = a.tokens; p.parent = a.parent; p.n_nodes = a.n_nodes; p.conf = a.conf;
  p.B = a.B; p.gamma = a.gamma; p.V = a.V; p.max_tokens = a.max_tokens; p.fixed_k = a.fixed_k;
  p.splits = cape_splits(a.V);
  const size_t rows = (size_t)a.B * a.gamma;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  size_t off = 256;
  p.seq_counters = reinterpret_cast<unsigned*>(ws + off);
  off += align256((size_t)a.B * sizeof(unsigned));
  p.slots = reinterpret_cast<u64*>(ws + off);
  const long long grid = (long long)rows * p.splits;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_pdl(cape_expand_kernel, dim3((unsigned)grid), dim3(kThreads), 0, st, p);
}

}  // namespace glide
