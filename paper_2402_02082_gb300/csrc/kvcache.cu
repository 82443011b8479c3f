// KV-cache update after verification (Section 3.1: after a verification step
// the target keeps the cache entries of the tokens it accepted and discards
// those of the rejected ones).
//
// The verified tree's entries sit at rows kv_len[b] + j (node j, linearized
// order of Section 3.2).  Acceptance returns the accepted root path
// path[b, 0..len[b]] (node 0 = x_t).  Keeping it means moving the entry of
// node path[b, k] to row kv_len[b] + k for k = 0..len[b], in every layer and
// head, for keys and values alike; the new cache length is kv_len[b] + len[b] + 1.
//
// One warp per (layer, b, h) slab.  Along a root path node indices grow at
// least as fast as depth (a parent precedes its child), so path[k] >= k: an
// entry only moves towards lower rows, rows with path[k] == k stay, and once
// one row moves every later row moves too.  Moving rows in increasing k is
// then safe as long as each batch of rows is read completely before any of it
// is written (a later row's source is never an earlier row's destination, but
// inside a batch one row's destination can be another's source).  Rows are
// copied as 16-byte chunks; a batch of 8 rows is held in registers.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kBatch = 8;  // rows per read-then-write batch

struct CompactParams {
  unsigned char* K;
  unsigned char* V;
  const int32_t* kv_len;
  const int32_t* path;
  const int32_t* len;
  int32_t* new_kv_len;
  long long layer_stride;  // bytes between layers
  long long slab_bytes;    // bytes of one (b, h) slab: S_cap rows
  int layers, B, H, S_cap, n;
};

// RC = 16-byte chunks per row (row bytes / 16).
template <int RC>
__global__ void __launch_bounds__(kThreads) kv_compact_kernel(const CompactParams p) {
  constexpr int kRowBytes = RC * 16;
  constexpr int kPerLane = kBatch * RC / 32;  // chunks per lane and tensor per batch
  static_assert(kPerLane >= 1, "row too short");
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const long long slabs = (long long)p.layers * p.B * p.H;
  const long long warps = (long long)gridDim.x * kWarps;
  for (long long slab = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5); slab < slabs; slab += warps) {
    const int layer = (int)(slab / ((long long)p.B * p.H));
    const int bh = (int)(slab - (long long)layer * p.B * p.H);
    const int b = bh / p.H;
    const int h = bh - b * p.H;
    // kv_len, len and the path are independent loads: issue them together
    const int32_t* pb = p.path + (size_t)b * p.n;
    int L = p.kv_len[b];
    int m = p.len[b];
    int s0 = lane < p.n ? pb[lane] : lane;
    int s1 = lane + 32 < p.n ? pb[lane + 32] : lane + 32;
    L = L < 0 ? 0 : (L > p.S_cap - p.n ? p.S_cap - p.n : L);
    m = (m < 0 ? 0 : (m > p.n - 1 ? p.n - 1 : m)) + 1;
    if (layer == 0 && h == 0 && lane == 0) p.new_kv_len[b] = L + m;

    // source node of path position k (clamped into the tree), two per lane;
    // positions at or beyond m do not move
    s0 = s0 < 0 ? 0 : (s0 > p.n - 1 ? p.n - 1 : s0);
    s1 = s1 < 0 ? 0 : (s1 > p.n - 1 ? p.n - 1 : s1);
    unsigned long long moves =
        (unsigned long long)__ballot_sync(0xffffffffu, lane < m && s0 != lane) |
        ((unsigned long long)__ballot_sync(0xffffffffu, lane + 32 < m && s1 != lane + 32) << 32);
    if (moves == 0ull) continue;

    const size_t slab_off = (size_t)layer * p.layer_stride + (size_t)bh * p.slab_bytes;
    unsigned char* Kb = p.K + slab_off + (size_t)L * kRowBytes;
    unsigned char* Vb = p.V + slab_off + (size_t)L * kRowBytes;
    while (moves) {
      int dst[kBatch], src[kBatch];
      int cnt = 0;
#pragma unroll
      for (int r = 0; r < kBatch; ++r) {
        dst[r] = 0;
        src[r] = 0;
        if (moves) {
          const int k = __ffsll((long long)moves) - 1;
          moves &= moves - 1;
          const int sk = __shfl_sync(0xffffffffu, k < 32 ? s0 : s1, k & 31);
          dst[r] = k;
          src[r] = sk;
          cnt = r + 1;
        }
      }
      uint4 kr[kPerLane], vr[kPerLane];
#pragma unroll
      for (int j = 0; j < kPerLane; ++j) {
        const int c = lane + 32 * j;
        const int r = c / RC, ch = c % RC;
        if (r < cnt) {
          int sr = src[0];
#pragma unroll
          for (int q = 1; q < kBatch; ++q)
            if (r == q) sr = src[q];
          kr[j] = reinterpret_cast<const uint4*>(Kb + (size_t)sr * kRowBytes)[ch];
          vr[j] = reinterpret_cast<const uint4*>(Vb + (size_t)sr * kRowBytes)[ch];
        }
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < kPerLane; ++j) {
        const int c = lane + 32 * j;
        const int r = c / RC, ch = c % RC;
        if (r < cnt) {
          int dr = dst[0];
#pragma unroll
          for (int q = 1; q < kBatch; ++q)
            if (r == q) dr = dst[q];
          reinterpret_cast<uint4*>(Kb + (size_t)dr * kRowBytes)[ch] = kr[j];
          reinterpret_cast<uint4*>(Vb + (size_t)dr * kRowBytes)[ch] = vr[j];
        }
      }
      __syncwarp();
    }
  }
}

}  // namespace

cudaError_t launch_kv_compact(const CompactArgs& a, cudaStream_t st) {
  CompactParams p;
  p.K = static_cast<unsigned char*>(a.K);
  p.V = static_cast<unsigned char*>(a.V);
  p.kv_len = a.kv_len; p.path = a.path; p.len = a.len; p.new_kv_len = a.new_kv_len;
  const int elt = a.dtype == 0 ? 2 : 4;
  const int row_bytes = a.D * elt;
  p.layer_stride = a.layer_stride * elt;
  p.slab_bytes = (long long)a.S_cap * row_bytes;
  p.layers = a.layers; p.B = a.B; p.H = a.H; p.S_cap = a.S_cap; p.n = a.n;
  const long long slabs = (long long)a.layers * a.B * a.H;
  long long grid = (slabs + kWarps - 1) / kWarps;
  const long long cap = (long long)sm_count() * 8;
  if (grid > cap) grid = cap;
  const dim3 g((unsigned)grid), blk(kThreads);
  switch (row_bytes / 16) {
    case 8: return launch_pdl(kv_compact_kernel<8>, g, blk, 0, st, p);
    case 16: return launch_pdl(kv_compact_kernel<16>, g, blk, 0, st, p);
    case 32: return launch_pdl(kv_compact_kernel<32>, g, blk, 0, st, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace glide
