// Pieces shared by the CUDA-core attention kernels: per-lane element loads,
// the warp transpose-reduction of 32 partial dot products, and the
// last-CTA-done merge of split partials.
#pragma once

#include <cuda_bf16.h>
#include <math_constants.h>

#include "common.cuh"

namespace glide {

// E consecutive elements at p, widened to fp32.  p is aligned to E*sizeof(T).
template <typename T, int E>
__device__ __forceinline__ void load_row_chunk(const T* p, float (&f)[E]);

template <>
__device__ __forceinline__ void load_row_chunk<__nv_bfloat16, 4>(const __nv_bfloat16* p, float (&f)[4]) {
  const uint2 w = *reinterpret_cast<const uint2*>(p);
  f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
}
template <>
__device__ __forceinline__ void load_row_chunk<__nv_bfloat16, 2>(const __nv_bfloat16* p, float (&f)[2]) {
  const uint32_t w = *reinterpret_cast<const uint32_t*>(p);
  f[0] = bf16lo(w); f[1] = bf16hi(w);
}
template <>
__device__ __forceinline__ void load_row_chunk<float, 4>(const float* p, float (&f)[4]) {
  const float4 w = *reinterpret_cast<const float4*>(p);
  f[0] = w.x; f[1] = w.y; f[2] = w.z; f[3] = w.w;
}
template <>
__device__ __forceinline__ void load_row_chunk<float, 2>(const float* p, float (&f)[2]) {
  const float2 w = *reinterpret_cast<const float2*>(p);
  f[0] = w.x; f[1] = w.y;
}

// 32 lanes each hold partial sums part[k] for 32 keys k (over the lane's own
// slice of the head dimension).  Five exchange rounds leave lane k holding
// the full sum for key k in part[0] (31 shuffles instead of 32 x 5).
__device__ __forceinline__ float transpose_reduce32(float (&part)[32], int lane) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const bool upper = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < off; ++j) {
      const float send = upper ? part[j] : part[j + off];
      const float keep = upper ? part[j + off] : part[j];
      part[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
    }
  }
  return part[0];
}

// The same for 16 keys: four exchange rounds and one final pairwise sum leave
// lanes 2k and 2k+1 both holding the full sum for key k (16 shuffles).
__device__ __forceinline__ float transpose_reduce16(float (&part)[16], int lane) {
#pragma unroll
  for (int off = 16, cnt = 8; off >= 2; off >>= 1, cnt >>= 1) {
    const bool upper = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < cnt; ++j) {
      const float send = upper ? part[j] : part[j + cnt];
      const float keep = upper ? part[j + cnt] : part[j];
      part[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
    }
  }
  return part[0] + __shfl_xor_sync(0xffffffffu, part[0], 1);
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// After this CTA wrote its partial for (b, h) into its slot, count the CTA in;
// the CTA that completes the count merges every slot of (b, h) into `out` and
// re-arms the counter.  Nothing waits: the last arrival does the work.
// Called by all `nthreads` consumer threads.
__device__ inline void combine_if_last(const Segment& s, int B, int H, int nq, int D, float* partials,
                                       unsigned* counters, float* out, int ctid, int nthreads,
                                       volatile int* flag) {
  const int bh = s.b * H + s.h;
  __threadfence();
  consumer_sync(nthreads);
  if (ctid == 0) {
    const unsigned prev = atomicAdd(&counters[bh], 1u);
    *flag = (prev == (unsigned)(s.c_last - s.c_first)) ? 1 : 0;
  }
  consumer_sync(nthreads);
  if (*flag) {
    __threadfence();
    for (int idx = ctid; idx < nq * D; idx += nthreads) {
      const int iq = idx / D, d = idx - iq * D;
      float M = -CUDART_INF_F;
      for (int c = s.c_first; c <= s.c_last; ++c) {
        const float* row = partial_slot(partials, c + bh, nq, D) + (size_t)iq * (D + 2);
        M = fmaxf(M, __ldcg(row));
      }
      float L = 0.f, O = 0.f;
      for (int c = s.c_first; c <= s.c_last; ++c) {
        const float* row = partial_slot(partials, c + bh, nq, D) + (size_t)iq * (D + 2);
        const float w = fast_exp2(__ldcg(row) - M);
        L += w * __ldcg(row + 1);
        O += w * __ldcg(row + 2 + d);
      }
      out[(((size_t)s.b * nq + iq) * H + s.h) * D + d] = O / L;
    }
    if (ctid == 0) counters[bh] = 0u;
  }
  consumer_sync(nthreads);
}

// Waits on the phase of `bar` with `parity`, bounded by time only (used to
// drain copies still in flight after an abort).
__device__ inline void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) return;
  }
}

}  // namespace glide
