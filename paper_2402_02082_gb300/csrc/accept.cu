// Greedy tree acceptance (Section 2's greedy "speculative decoding" rule on
// the token tree of CaPE's verification, Section 3.2).
//
// One launch does both steps:
// 1. argmax over the vocabulary of every (sequence, node) logits row.  The
//    row is cut into chunks, one CTA per chunk; a CTA reduces its chunk to one
//    64-bit key (order-preserving float bits above the complemented index, so
//    that the larger key is the larger value and, among equal values, the
//    lower index) and folds it into the row's slot with atomicMax.  The scan
//    is a plain HBM stream of the logits.
// 2. the CTA that completes a sequence's count (atomic counter, no waiting)
//    walks that sequence's tree with one warp: a node is accepted iff every
//    edge on its root path matches (draft token == parent's argmax); the
//    deepest accepted node, lowest index among equals, gives the path, its
//    length and the bonus token.  It then re-arms the slots and the counter.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 8192;  // logits per CTA
constexpr int kVec = kChunk / (4 * kThreads);  // float4 loads per thread, all in flight at once
static_assert(kChunk % (4 * kThreads) == 0, "chunk of whole float4 rounds");

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
};

__device__ __forceinline__ unsigned long long argmax_key(float f, int idx) {
  uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);  // -0 and +0 compare equal
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (unsigned long long)(0xffffffffu - (uint32_t)idx);
}

__device__ __forceinline__ int key_index(unsigned long long k) {
  return (int)(0xffffffffu - (uint32_t)(k & 0xffffffffull));
}

__device__ __forceinline__ unsigned long long umax64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}

__global__ void __launch_bounds__(kThreads) tree_accept_kernel(const AccParams p) {
  __shared__ unsigned long long red[kThreads / 32];
  __shared__ int last;
  __shared__ int sa[kMaxTree], sp[kMaxTree], sd[kMaxTree];

  const int row = blockIdx.x / p.splits;
  const int split = blockIdx.x - row * p.splits;
  const int b = row / p.n;
  const float* lg = p.logits + (size_t)row * p.V;
  const int lo = split * kChunk;
  const int hi = min(p.V, lo + kChunk);

  unsigned long long best = 0ull;
  if ((p.V & 3) == 0) {
    const float4* v4 = reinterpret_cast<const float4*>(lg);
    const int j0 = lo / 4 + threadIdx.x, j1 = hi / 4;
    float4 x[kVec];
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int j = j0 + u * kThreads;
      x[u] = j < j1 ? __ldcs(v4 + j) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int j = j0 + u * kThreads;
      if (j < j1) {
        const int i0 = 4 * j;
        best = umax64(best, argmax_key(x[u].x, i0));
        best = umax64(best, argmax_key(x[u].y, i0 + 1));
        best = umax64(best, argmax_key(x[u].z, i0 + 2));
        best = umax64(best, argmax_key(x[u].w, i0 + 3));
      }
    }
  } else {
    for (int j = lo + threadIdx.x; j < hi; j += kThreads) best = umax64(best, argmax_key(__ldcs(lg + j), j));
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) best = umax64(best, __shfl_xor_sync(0xffffffffu, best, off));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = best;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long k = red[0];
    for (int w = 1; w < kThreads / 32; ++w) k = umax64(k, red[w]);
    atomicMax(&p.slots[row], k);
    __threadfence();
    const unsigned prev = atomicAdd(&p.counters[b], 1u);
    last = (prev == (unsigned)(p.splits * p.n - 1)) ? 1 : 0;
  }
  __syncthreads();
  if (!last || warp != 0) return;

  // ---- tree walk for sequence b (one warp)
  __threadfence();
  const int n = p.n;
  const int32_t* par = p.parent + (size_t)b * n;
  const int32_t* dr = p.draft + (size_t)b * n;
  for (int c = lane; c < n; c += 32) {  // the argmaxes and the tree into shared memory for the walks
    sa[c] = key_index(__ldcg(&p.slots[(size_t)b * n + c]));
    sp[c] = par[c];
    sd[c] = dr[c];
  }
  __syncwarp();
  unsigned key = 0;
  for (int c = lane; c < n; c += 32) {
    bool ok = true;
    int depth = 0;
    int x = c;
    for (int step = 0; step < kMaxTree && x != 0; ++step) {
      const int px = sp[x];
      if (px < 0 || px >= x || sd[x] != sa[px]) { ok = false; break; }
      ++depth;
      x = px;
    }
    if (ok) key = max(key, ((unsigned)depth << 8) | (unsigned)(255 - c));
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, off));
  const int node = 255 - (int)(key & 255u);
  const int depth = (int)(key >> 8);
  int32_t* out_path = p.path + (size_t)b * n;
  for (int d = depth + 1 + lane; d < n; d += 32) out_path[d] = -1;
  if (lane == 0) {
    int x = node;
    for (int d = depth; d >= 0; --d) {
      out_path[d] = x;
      x = d > 0 ? sp[x] : -1;
    }
    p.len[b] = depth;
    p.bonus[b] = sa[node];
  }
  for (int c = lane; c < n; c += 32) p.slots[(size_t)b * n + c] = 0ull;
  if (lane == 0) p.counters[b] = 0u;
}

size_t counters_bytes(int B) { return ((size_t)B * sizeof(unsigned) + 255) & ~size_t(255); }

}  // namespace

size_t accept_workspace_bytes(int B, int n) {
  return 256 + counters_bytes(B) + (size_t)B * n * sizeof(unsigned long long);
}

cudaError_t launch_tree_accept(const AcceptArgs& a, cudaStream_t st) {
  AccParams p;
  p.draft = a.draft; p.parent = a.parent; p.logits = a.logits;
  p.path = a.path; p.len = a.len; p.bonus = a.bonus;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.counters = reinterpret_cast<unsigned*>(ws + 256);
  p.slots = reinterpret_cast<unsigned long long*>(ws + 256 + counters_bytes(a.B));
  p.B = a.B; p.n = a.n; p.V = a.V;
  p.splits = (a.V + kChunk - 1) / kChunk;
  const long long grid = (long long)a.B * a.n * p.splits;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidValue;
  tree_accept_kernel<<<(unsigned)grid, kThreads, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace glide
