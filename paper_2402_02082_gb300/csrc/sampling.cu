// Speculative-sampling acceptance of a chain proposal (the acceptance strategy
// that Section 2 names and Section 4.1 uses for GliDe alone): position i
// accepts x_i when u_i * p_D,i(x_i) < p_T,i(x_i), with p_T = SoftMax(target
// logits); after the first rejection (position i) one more token is drawn from
// max(0, p_T,i - p_D,i), else from p_T,gamma+1, by inverse CDF with v: the
// first token whose running weight exceeds v * (total weight).
//
// One launch, no waiting:
// 1. one CTA per (sequence, position) row of target logits: an online
//    (max, sum of exp) over the row, then, for a proposal position, p_T(x_i)
//    and the acceptance decision; the CTA counts itself in for its sequence;
// 2. the CTA that completes a sequence's count finds the first rejection and
//    draws the extra token from the row it names.  Each warp owns a contiguous
//    segment of the row and sums its weights with unit-stride loads; a scan
//    over the 32 segment totals places the segments on the running total; the
//    warp whose segment reaches past v * total walks it in 32-token groups
//    (a shuffle scan per group) to the first token past the target.
// Floating point decides integers here (a decision, a token), in fp32 with
// this kernel's summation order; an exact real-number computation can differ
// only where u * p_D(x) or v * total lies within rounding of its threshold.
#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>

#include "attn_common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kBatch = 8;   // row-scan loads in flight per thread
constexpr int kGrp = 8;     // draw: 32-token groups whose loads are issued together

struct SampleParams {
  const int32_t* draft;    // [B, gamma]
  const float* q;          // [B, gamma, V]
  const float* logits;     // [B, gamma + 1, V]
  const float* u;          // [B, gamma + 1]
  int32_t* n_acc;          // [B]
  int32_t* next_tok;       // [B]
  unsigned* counters;      // [B]
  float2* stats;           // [B, gamma + 1]: (max, sum of 2^((l - max) * log2 e))
  int* accept;             // [B, gamma]
  int B, gamma, V;
};

__device__ __forceinline__ void online_add(float& m, float& s, float x) {
  if (x > m) {
    s = s * fast_exp2((m - x) * kLog2e) + 1.f;
    m = x;
  } else {
    s += fast_exp2((x - m) * kLog2e);
  }
}

__device__ __forceinline__ void online_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -CUDART_INF_F) return;
  if (m2 > m) {
    s = s * fast_exp2((m - m2) * kLog2e) + s2;
    m = m2;
  } else {
    s += s2 * fast_exp2((m2 - m) * kLog2e);
  }
}

__global__ void __launch_bounds__(kThreads) spec_sample_kernel(const SampleParams p) {
  __shared__ float2 red[kWarps];
  __shared__ float seg_up[kWarps];
  __shared__ int last, s_tok, s_lastpos, s_win;
  pdl_wait();

  const int G1 = p.gamma + 1;
  const int row = blockIdx.x;
  const int b = row / G1, i = row - b * G1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* lg = p.logits + (size_t)row * p.V;

  // ---- 1. (max, sum) of the row; batches of kBatch loads per thread, all
  // issued before any use
  float m = -CUDART_INF_F, s = 0.f;
  if ((p.V & 3) == 0) {
    const float4* l4 = reinterpret_cast<const float4*>(lg);
    const int n4 = p.V / 4;
    for (int j0 = threadIdx.x; j0 < n4; j0 += kBatch * kThreads) {
      float4 x[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        if (j0 + k * kThreads < n4) x[k] = __ldg(l4 + j0 + k * kThreads);
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        if (j0 + k * kThreads < n4) {
          online_add(m, s, x[k].x);
          online_add(m, s, x[k].y);
          online_add(m, s, x[k].z);
          online_add(m, s, x[k].w);
        }
    }
  } else {
    for (int j0 = threadIdx.x; j0 < p.V; j0 += kBatch * kThreads) {
      float x[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        if (j0 + k * kThreads < p.V) x[k] = __ldg(lg + j0 + k * kThreads);
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        if (j0 + k * kThreads < p.V) online_add(m, s, x[k]);
    }
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off), s2 = __shfl_xor_sync(0xffffffffu, s, off);
    online_merge(m, s, m2, s2);
  }
  if (lane == 0) red[warp] = make_float2(m, s);
  __syncthreads();
  if (threadIdx.x == 0) {
    float M = red[0].x, S = red[0].y;
    for (int w = 1; w < kWarps; ++w) online_merge(M, S, red[w].x, red[w].y);
    p.stats[row] = make_float2(M, S);
    if (i < p.gamma) {
      int x = p.draft[(size_t)b * p.gamma + i];
      x = x < 0 ? 0 : (x >= p.V ? p.V - 1 : x);
      const float pt = fast_exp2((__ldg(lg + x) - M) * kLog2e) / S;
      const float qd = p.q[((size_t)b * p.gamma + i) * p.V + x];
      p.accept[(size_t)b * p.gamma + i] = (p.u[(size_t)b * G1 + i] * qd < pt) ? 1 : 0;
    }
    __threadfence();
    const unsigned prev = atomicAdd(&p.counters[b], 1u);
    last = prev == (unsigned)p.gamma ? 1 : 0;  // gamma + 1 rows per sequence
    if (last) __threadfence();
  }
  __syncthreads();
  if (!last) return;

  // ---- 2. the first rejection and the extra token of sequence b
  int n = p.gamma;
  for (int k = 0; k < p.gamma; ++k)
    if (!__ldcg(p.accept + (size_t)b * p.gamma + k)) {
      n = k;
      break;
    }
  const float2 st = __ldcg(p.stats + (size_t)b * G1 + n);
  const float* L = p.logits + ((size_t)b * G1 + n) * p.V;
  const float* Q = n < p.gamma ? p.q + ((size_t)b * p.gamma + n) * p.V : nullptr;  // null: draw from p_T
  const float inv = 1.f / st.y;
  const float v = p.u[(size_t)b * G1 + p.gamma];
  const int seg = (p.V + kWarps - 1) / kWarps;  // contiguous segment per warp
  const int x0 = min(p.V, warp * seg), x1 = min(p.V, x0 + seg);

  // weights of kGrp 32-token groups starting at base (lane j: token base + 32k + j);
  // every load first, then the arithmetic; 0 past the segment
  auto groups = [&](int base, float (&w)[kGrp]) {
    float lv[kGrp], qv[kGrp];
#pragma unroll
    for (int k = 0; k < kGrp; ++k) {
      const int x = base + 32 * k + lane;
      lv[k] = x < x1 ? __ldg(L + x) : 0.f;
      qv[k] = (Q && x < x1) ? __ldg(Q + x) : 0.f;
    }
#pragma unroll
    for (int k = 0; k < kGrp; ++k) {
      const float pt = fast_exp2((lv[k] - st.x) * kLog2e) * inv;
      w[k] = base + 32 * k + lane < x1 ? (Q ? fmaxf(0.f, pt - qv[k]) : pt) : 0.f;
    }
  };

  // Inverse-CDF draw from the current weights; -1 when they sum to 0.
  auto draw = [&]() -> int {
    float part = 0.f;
    int lastpos = -1;
    for (int base = x0; base < x1; base += 32 * kGrp) {
      float w[kGrp];
      groups(base, w);
#pragma unroll
      for (int k = 0; k < kGrp; ++k) {
        part += w[k];
        if (w[k] > 0.f) lastpos = base + 32 * k + lane;
      }
    }
    const float segsum = warp_sum(part);
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) lastpos = max(lastpos, __shfl_xor_sync(0xffffffffu, lastpos, off));
    __syncthreads();  // the shared slots of a previous draw are free again
    if (threadIdx.x == 0) {
      s_tok = -1;
      s_lastpos = -1;
      s_win = kWarps;
    }
    if (lane == 0) seg_up[warp] = segsum;
    __syncthreads();
    if (lane == 0) atomicMax(&s_lastpos, lastpos);
    if (warp == 0) {
      float t = seg_up[lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, t, off);
        if (lane >= off) t += y;
      }
      seg_up[lane] = t;  // upper end of each segment on the running total
      const float target = v * __shfl_sync(0xffffffffu, t, 31);
      const unsigned hit = __ballot_sync(0xffffffffu, t > target);
      if (lane == 0 && hit) s_win = __ffs(hit) - 1;  // the first segment past the target
    }
    __syncthreads();
    const float total = seg_up[kWarps - 1];
    if (!(total > 0.f)) return -1;
    if (warp == s_win) {
      const float target = v * total;
      float running = warp > 0 ? seg_up[warp - 1] : 0.f;
      int tok = -1;
      for (int base = x0; base < x1 && tok < 0; base += 32 * kGrp) {
        float w[kGrp];
        groups(base, w);
#pragma unroll
        for (int k = 0; k < kGrp; ++k) {
          float incl = w[k];
#pragma unroll
          for (int off = 1; off < 32; off <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
          }
          const unsigned hit = __ballot_sync(0xffffffffu, running + incl > target && w[k] > 0.f);
          if (tok < 0 && hit) tok = base + 32 * k + __ffs(hit) - 1;
          running += __shfl_sync(0xffffffffu, incl, 31);
        }
      }
      // rounding can leave the walk just short of the target: the segment's last token
      if (lane == 0) s_tok = tok >= 0 ? tok : lastpos;
    }
    __syncthreads();
    return s_tok >= 0 ? s_tok : s_lastpos;  // no segment past the target: rounding at the very end
  };

  int tok = draw();
  if (tok < 0) {  // max(0, p_T - p_D) summed to 0 in fp32: draw from p_T instead
    Q = nullptr;
    tok = draw();
  }
  if (threadIdx.x == 0) {
    p.n_acc[b] = n;
    p.next_tok[b] = tok;
    p.counters[b] = 0u;
  }
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

// Workspace: [0,256) status | counters [B] | stats [B*(gamma+1)] float2 | decisions [B*gamma] int.
size_t sample_workspace_bytes(int B, int gamma) {
  return 256 + align256((size_t)B * 4) + align256((size_t)B * (gamma + 1) * 8) + align256((size_t)B * gamma * 4);
}

cudaError_t launch_spec_sample(const SampleArgs& a, cudaStream_t st) {
  SampleParams p;
  p.draft = a.draft; p.q = a.q; p.logits = a.logits; p.u = a.u;
  p.n_acc = a.n_acc; p.next_tok = a.next_tok;
  p.B = a.B; p.gamma = a.gamma; p.V = a.V;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  size_t off = 256;
  p.counters = reinterpret_cast<unsigned*>(ws + off);
  off += align256((size_t)a.B * 4);
  p.stats = reinterpret_cast<float2*>(ws + off);
  off += align256((size_t)a.B * (a.gamma + 1) * 8);
  p.accept = reinterpret_cast<int*>(ws + off);
  const long long grid = (long long)a.B * (a.gamma + 1);
  if (grid > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_pdl(spec_sample_kernel, dim3((unsigned)grid), dim3(kThreads), 0, st, p);
}

}  // namespace glide
