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

// ---------------------------------------------- lane-group mapping (cross)
// The cross-attention consumers split a warp into 4 groups of 8 lanes: group
// g takes keys 4g..4g+3 of a 16-key tile, and lane sub = lane & 7 owns the
// 16-byte chunks sub, sub + 8, ... of every K/V row, so the 8 lanes of a group
// read 128 contiguous bytes per chunk (no shared-memory bank conflicts).
template <typename T, int D>
struct GroupMap {
  static constexpr int kChunkElems = 16 / (int)sizeof(T);
  static constexpr int kRowBytes = D * (int)sizeof(T);
  static constexpr int kNC = kRowBytes / (8 * 16);  // chunks per lane and row
  static constexpr int kPairsPerChunk = kChunkElems / 2;
  static constexpr int kPairs = kNC * kPairsPerChunk;
};

// fp32 pairs in one 64-bit register, for the packed f32x2 arithmetic of sm_100+.
__device__ __forceinline__ uint64_t f2pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 f2unpack(uint64_t v) {
  float lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
  return make_float2(lo, hi);
}
__device__ __forceinline__ uint64_t f2mul(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ void f2fma(uint64_t& d, uint64_t a, uint64_t b) {
  asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(d) : "l"(a), "l"(b));
}
// bf16 pair (one word, element 0 low) widened to an fp32 pair.
__device__ __forceinline__ uint64_t bf16pair(uint32_t w) {
  return f2pack(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
// c + a.lo*b.lo + a.hi*b.hi with bf16 operands and fp32 accumulation (each
// bf16 product is exact in fp32; one rounding per fma).
__device__ __forceinline__ float fma_bf16x2(uint32_t a, uint32_t b, float c) {
  asm("{\n\t.reg .b16 al, ah, bl, bh;\n\t"
      "mov.b32 {al, ah}, %1;\n\tmov.b32 {bl, bh}, %2;\n\t"
      "fma.rn.f32.bf16 %0, al, bl, %0;\n\t"
      "fma.rn.f32.bf16 %0, ah, bh, %0;\n\t}"
      : "+f"(c)
      : "r"(a), "r"(b));
  return c;
}

// acc[0..1] += q . k over one 16-byte chunk (two independent chains).
template <typename T>
__device__ __forceinline__ void dot_chunk(const uint4& q, const uint4& k, float (&acc)[2]);
template <>
__device__ __forceinline__ void dot_chunk<__nv_bfloat16>(const uint4& q, const uint4& k, float (&acc)[2]) {
  acc[0] = fma_bf16x2(q.x, k.x, acc[0]);
  acc[1] = fma_bf16x2(q.y, k.y, acc[1]);
  acc[0] = fma_bf16x2(q.z, k.z, acc[0]);
  acc[1] = fma_bf16x2(q.w, k.w, acc[1]);
}
template <>
__device__ __forceinline__ void dot_chunk<float>(const uint4& q, const uint4& k, float (&acc)[2]) {
  acc[0] = fmaf(__uint_as_float(q.x), __uint_as_float(k.x), acc[0]);
  acc[1] = fmaf(__uint_as_float(q.y), __uint_as_float(k.y), acc[1]);
  acc[0] = fmaf(__uint_as_float(q.z), __uint_as_float(k.z), acc[0]);
  acc[1] = fmaf(__uint_as_float(q.w), __uint_as_float(k.w), acc[1]);
}

// o (fp32 pairs) += p * v over one 16-byte chunk of a V row.
template <typename T>
__device__ __forceinline__ void axpy_chunk(uint64_t p2, const uint4& v, uint64_t* o2);
template <>
__device__ __forceinline__ void axpy_chunk<__nv_bfloat16>(uint64_t p2, const uint4& v, uint64_t* o2) {
  f2fma(o2[0], p2, bf16pair(v.x));
  f2fma(o2[1], p2, bf16pair(v.y));
  f2fma(o2[2], p2, bf16pair(v.z));
  f2fma(o2[3], p2, bf16pair(v.w));
}
template <>
__device__ __forceinline__ void axpy_chunk<float>(uint64_t p2, const uint4& v, uint64_t* o2) {
  f2fma(o2[0], p2, f2pack(__uint_as_float(v.x), __uint_as_float(v.y)));
  f2fma(o2[1], p2, f2pack(__uint_as_float(v.z), __uint_as_float(v.w)));
}

// Each lane of a group of 8 holds partial sums for the group's 4 keys; two
// exchange rounds and a pairwise sum leave lanes 2k and 2k+1 of the group with
// the full sum for key k (4 shuffles).
__device__ __forceinline__ float group8_reduce4(float (&part)[4], int lane) {
  {
    const bool up = (lane & 4) != 0;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const float send = up ? part[j] : part[j + 2];
      const float keep = up ? part[j + 2] : part[j];
      part[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
  }
  {
    const bool up = (lane & 2) != 0;
    const float send = up ? part[0] : part[1];
    const float keep = up ? part[1] : part[0];
    part[0] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
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

// Output row of query row r of slab (b, cached head h): rows are node-major,
// `group` query heads per node, Hq query heads in all (group = 1, Hq = H: one
// query head per slab).
__device__ __forceinline__ size_t out_row(int b, int h, int r, int nrows, int group, int Hq) {
  const int node = r / group;
  return ((size_t)b * (nrows / group) + node) * Hq + (size_t)h * group + (r - node * group);
}

// Split-KV bookkeeping of a slab (b, cached head h) whose nq query rows are
// served in row tiles of at most 64: each row tile has its own arrival
// counter (index cidx, see row_tile_counter) and merges its rows [r0, r0 + nr)
// of the partial slots.  One row tile covers all rows when nq <= 64.
__device__ __forceinline__ int row_tile_counter(int b, int h, int H, int R, int y) {
  return (b * H + h) * R + y;
}

// After this CTA wrote its partial rows [r0, r0 + nr) for (b, h) into its
// slot, count the CTA in; the CTA that completes the count merges those rows
// of every slot of (b, h) into `out` and re-arms the counter.  Nothing waits:
// the last arrival does the work.  The slab's nq query rows map to outputs by
// out_row.  Called by all `nthreads` consumer threads.
__device__ inline void combine_if_last(const Segment& s, int H, int nq, int r0, int nr, int cidx, int D, int group,
                                       int Hq, float* partials, unsigned* counters, float* out, int ctid,
                                       int nthreads, volatile int* flag) {
  const int bh = s.b * H + s.h;
  __threadfence();
  consumer_sync(nthreads);
  if (ctid == 0) {
    const unsigned prev = atomicAdd(&counters[cidx], 1u);
    *flag = (prev == (unsigned)(s.c_last - s.c_first)) ? 1 : 0;
  }
  consumer_sync(nthreads);
  if (*flag) {
    __threadfence();
    for (int idx = ctid; idx < nr * D; idx += nthreads) {
      const int iq = r0 + idx / D, d = idx % D;
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
      out[out_row(s.b, s.h, iq, nq, group, Hq) * D + d] = O / L;
    }
    if (ctid == 0) counters[cidx] = 0u;
  }
  consumer_sync(nthreads);
}

// Where query row r of slab (b, h) goes in the output: out_row with nq / group
// nodes (tree verification and grouped-query cross-attention).
struct OutMap {
  int group, Hq;
  __device__ long long row(int b, int h, int r, int nq) const { return (long long)out_row(b, h, r, nq, group, Hq); }
};

}  // namespace glide
