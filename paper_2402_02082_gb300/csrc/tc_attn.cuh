// Device helpers shared by the tcgen05 attention kernels (tree verification
// in 64- and 128-row tiles, the training-time block mask) and the merge of
// split-KV verification partials.  Everything here has internal linkage: each
// kernel file gets its own copy.
#pragma once

#include <cuda_bf16.h>
#include <math_constants.h>

#include "attn_common.cuh"
#include "common.cuh"
#include "kernels.h"

namespace glide {
namespace {

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// Warp-uniform bounded wait: every lane probes once and the warp votes; only
// if the phase is not complete yet does lane 0 run the bounded wait and the
// warp follow it.  Every lane sees the same outcome, so the warp-collective
// tcgen05 instructions after it stay convergent.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, unsigned* status) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, status) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Packed pairs of fp32 (element 0 in the low word) for the f32x2 instructions.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unf2(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// A shared-memory descriptor advanced by `bytes`: the start address is the
// descriptor's low field in 16-byte units, and shared addresses stay below
// 2^18, so the sum never carries out of it.
__host__ __device__ constexpr uint64_t desc_step(uint32_t bytes) { return bytes >> 4; }

// Named barrier of the two softmax warps of one TMEM lane quarter (ids 4-7;
// id 0 is __syncthreads).
__device__ __forceinline__ void pair_sync(int quarter) {
  asm volatile("bar.sync %0, 64;" ::"r"(4 + quarter) : "memory");
}

// The ancestor-or-self set (bit j: node j) of `node` in the tree `parent[0..n)`
// (parent[j] in [0, j) or anything else for a root), for every lane of the
// warp at once: lane x holds nodes x and x + 32, each with the set A found so
// far and the next ancestor P not yet in it (A = {x}, P = parent(x) at first);
// a round of pointer jumping sets A |= A[P] and P = P[P], so six rounds cover
// the 64 levels a tree of at most 64 nodes can have.  Two coalesced loads and
// shuffles replace one dependent global load per tree level.  Warp-collective;
// a lane with want == false gets 0.
__device__ inline uint64_t ancestors(const int* parent, int n, int node, bool want, int lane) {
  uint64_t a[2];
  int q[2];
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int x = lane + 32 * k;
    const int px = x < n ? parent[x] : -1;
    a[k] = x < n ? 1ull << x : 0ull;
    q[k] = (px >= 0 && px < x) ? px : -1;
  }
#pragma unroll
  for (int round = 0; round < 6; ++round) {
    uint64_t na[2];
    int nq[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int y = q[k] < 0 ? 0 : q[k];  // every lane shuffles; a root keeps its set
      const uint64_t ay0 = __shfl_sync(0xffffffffu, a[0], y & 31), ay1 = __shfl_sync(0xffffffffu, a[1], y & 31);
      const int qy0 = __shfl_sync(0xffffffffu, q[0], y & 31), qy1 = __shfl_sync(0xffffffffu, q[1], y & 31);
      na[k] = q[k] < 0 ? a[k] : a[k] | (y < 32 ? ay0 : ay1);
      nq[k] = q[k] < 0 ? -1 : (y < 32 ? qy0 : qy1);
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      a[k] = na[k];
      q[k] = nq[k];
    }
  }
  const int v = want ? node : 0;
  const uint64_t r0 = __shfl_sync(0xffffffffu, a[0], v & 31), r1 = __shfl_sync(0xffffffffu, a[1], v & 31);
  return want ? (v < 32 ? r0 : r1) : 0ull;
}

// Merges the partials of every split slab: one warp per query row r of slab
// (b, cached head h) with share range [c_first, c_last] (ranges[bh]); the
// partial of share c sits in slot c + bh, row r: [max, sum, o[D]] (log2
// domain).  out = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c, M = max_c m_c.
// Each lane holds D / 32 columns (float2 pairs: a partial row is 8-byte
// aligned); the loads of up to kMergeGroup shares are issued before any is
// used, and groups fold into a running (max, sum, o).  A share whose max is
// -inf (no visible key) has weight 0 and its o never reaches a sum.
constexpr int kMergeGroup = 8;
constexpr int kMergeWarps = 8;
template <int D>
__global__ void __launch_bounds__(kMergeWarps * 32) tree_merge_kernel(const int2* ranges, const float* partials,
                                                                     float* out, int BH, int rows, int group, int Hq,
                                                                     int Hkv) {
  constexpr int kPairs = D / 64;  // float2 pairs per lane
  // The next kernel may be scheduled now, onto the SMs this small grid leaves
  // free; it waits for this merge to complete before it touches memory.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  pdl_wait();  // the partials and ranges of the verification kernel are complete
  const int lane = threadIdx.x & 31;
  const long long total = (long long)BH * rows;
  for (long long wr = (long long)blockIdx.x * kMergeWarps + (threadIdx.x >> 5); wr < total;
       wr += (long long)gridDim.x * kMergeWarps) {
    const int bh = (int)(wr / rows), r = (int)(wr - (long long)bh * rows);
    const int2 rg = ranges[bh];
    if (rg.x < 0) continue;
    const size_t sstride = (size_t)rows * (D + 2);
    const float* row0 = partials + (size_t)(rg.x + bh) * sstride + (size_t)r * (D + 2);
    const int nsl = rg.y - rg.x + 1;
    float M = -CUDART_INF_F, L = 0.f;
    float2 acc[kPairs];
#pragma unroll
    for (int k = 0; k < kPairs; ++k) acc[k] = make_float2(0.f, 0.f);
    for (int c0 = 0; c0 < nsl; c0 += kMergeGroup) {
      float2 ml[kMergeGroup], o[kMergeGroup][kPairs];
#pragma unroll
      for (int u = 0; u < kMergeGroup; ++u) {
        const int c = c0 + u < nsl ? c0 + u : c0;
        const float* pr = row0 + (size_t)c * sstride;
        ml[u] = __ldcg(reinterpret_cast<const float2*>(pr));
#pragma unroll
        for (int k = 0; k < kPairs; ++k) o[u][k] = __ldcg(reinterpret_cast<const float2*>(pr + 2 + 64 * k + 2 * lane));
        if (c0 + u >= nsl) ml[u].x = -CUDART_INF_F;
      }
      float Mg = M;
#pragma unroll
      for (int u = 0; u < kMergeGroup; ++u) Mg = fmaxf(Mg, ml[u].x);
      if (Mg == -CUDART_INF_F) continue;
      const float f = M == -CUDART_INF_F ? 0.f : fast_exp2(M - Mg);
      L *= f;
#pragma unroll
      for (int k = 0; k < kPairs; ++k) acc[k] = make_float2(acc[k].x * f, acc[k].y * f);
#pragma unroll
      for (int u = 0; u < kMergeGroup; ++u) {
        const bool live = ml[u].x != -CUDART_INF_F;
        const float w = live ? fast_exp2(ml[u].x - Mg) : 0.f;
        L += live ? w * ml[u].y : 0.f;
#pragma unroll
        for (int k = 0; k < kPairs; ++k) {
          acc[k].x += live ? w * o[u][k].x : 0.f;  // a select: an unwritten o never reaches acc
          acc[k].y += live ? w * o[u][k].y : 0.f;
        }
      }
      M = Mg;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    const int b = bh / Hkv, h = bh - b * Hkv;
    float* dst = out + out_row(b, h, r, rows, group, Hq) * D;
#pragma unroll
    for (int k = 0; k < kPairs; ++k)
      *reinterpret_cast<float2*>(dst + 64 * k + 2 * lane) = make_float2(acc[k].x * inv, acc[k].y * inv);
  }
}


// The merge launch of a split verification: one warp per query row, at most
// four waves of CTAs over the SMs.
template <int D>
cudaError_t launch_tree_merge(const int2* ranges, const float* partials, float* out, int BH, int rows, int group,
                              int Hq, int Hkv, cudaStream_t st) {
  const long long rows_total = (long long)BH * rows;
  long long mg = (rows_total + kMergeWarps - 1) / kMergeWarps;
  const long long cap = 4LL * sm_count() * (2048 / (kMergeWarps * 32));
  if (mg > cap) mg = cap;
  return launch_pdl(tree_merge_kernel<D>, dim3((unsigned)mg), dim3(kMergeWarps * 32), 0, st, ranges, partials, out,
                    BH, rows, group, Hq, Hkv);
}

}  // namespace
}  // namespace glide
