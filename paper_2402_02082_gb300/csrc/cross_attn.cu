// GliDe cross-attention (Section 3.1): one draft query per (sequence, head)
// attends to every cached key/value of the target layer,
//   hd_j = SoftMax(Q^{m,j} (K^{l,j})^T / sqrt(d_k)) V^{l,j},
// with no mask at inference.
//
// The step reads every cached K and V byte once and does ~1 flop per byte, so
// it is bound by HBM bandwidth.  Design:
// * persistent grid (one CTA per SM); the key ranges of all (b, h) are cut
//   into 16-key tiles and dealt to CTAs in equal contiguous shares (split-KV
//   with exact balance, ragged batches included);
// * four producer threads (one per producer warp; issuing a bulk copy keeps
//   a thread busy for hundreds of cycles) stream K and V tiles with 1-D bulk
//   copies (TMA) into shared-memory stages guarded by mbarriers; tile i goes
//   to consumer warp i % NW, and every consumer warp owns a private ring of
//   SW stages that it drains strictly in order (a warp never waits on a stage
//   whose earlier phase is still pending, so the mbarrier parity cannot
//   alias);
// * each of the NW = 8 consumer warps (two per SM sub-partition, so one
//   warp's shuffle and shared-memory latencies hide behind the other's work)
//   takes whole tiles: lanes split the head dimension, a transpose-reduction
//   turns 16x(D/32)-element partial dot products into one score per lane pair,
//   and an fp32 online softmax (log2 domain) accumulates P.V;
// * per segment the warps merge in shared memory; a (b, h) split across CTAs
//   is finished by the last CTA to arrive (atomic counter, no waiting).
#include <cuda_bf16.h>
#include <math_constants.h>

#include "attn_common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kTK = 16;      // keys per tile
constexpr int kNW = 8;       // consumer warps
constexpr int kNP = 4;       // producer warps, each feeding kNW / kNP consumer rings
constexpr int kThreads = (kNW + kNP) * 32;

template <typename T, int D>
struct CrossCfg {
  static constexpr int kTile = kTK * D * (int)sizeof(T);
  static constexpr int kFit = (192 * 1024) / (2 * kTile * kNW);
  static constexpr int SW = kFit > 3 ? 3 : (kFit < 1 ? 1 : kFit);   // stages per consumer warp
  static constexpr int NS = SW * kNW;
  static constexpr size_t kStageBytes = (size_t)NS * kTile;
  static constexpr size_t off_K = 0;
  static constexpr size_t off_V = kStageBytes;
  static constexpr size_t off_bar = 2 * kStageBytes;                   // full[NS], empty[NS]
  static constexpr size_t off_scratch = off_bar + 2 * NS * sizeof(uint64_t);
  static constexpr size_t off_misc = off_scratch + (size_t)kNW * (D + 2) * sizeof(float);
  static constexpr size_t off_tab = off_misc + 16;                     // batch tile table
  static size_t smem_bytes(int B) {
    return off_tab + (size_t)(B + 1) * 8 + (size_t)3 * B * 4;
  }
};

struct CrossParams {
  const void* q;
  const void* K;
  const void* V;
  const int* kv_len;
  float* out;
  unsigned* status;
  unsigned* counters;
  float* partials;
  int B, H, S_cap, max_kv_len;
  float scale_log2;
};

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 1) cross_attn_kernel(const CrossParams p) {
  using C = CrossCfg<T, D>;
  using G = GroupMap<T, D>;
  constexpr int NS = C::NS;
  extern __shared__ __align__(1024) unsigned char smem[];
  T* sK = reinterpret_cast<T*>(smem + C::off_K);
  T* sV = reinterpret_cast<T*>(smem + C::off_V);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::off_bar);
  uint64_t* empty = full + NS;
  float* scratch = reinterpret_cast<float*>(smem + C::off_scratch);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::off_misc);
  volatile int* last_flag = abort_flag + 1;
  BatchTiles bt;
  bt.start = reinterpret_cast<long long*>(smem + C::off_tab);
  bt.len = reinterpret_cast<int*>(bt.start + p.B + 1);
  bt.ntiles = bt.len + p.B;
  bt.plen = bt.ntiles + p.B;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  build_batch_tiles(bt, p.kv_len, p.B, p.H, p.max_kv_len, 0, kTK);  // ends with __syncthreads

  Partition P;
  P.init(bt.start[p.B], gridDim.x);
  const long long g_begin = P.begin(blockIdx.x), g_end = P.end(blockIdx.x);

  // A sequence with no cached keys has an empty softmax: its output is zero.
  for (int bh = blockIdx.x; bh < p.B * p.H; bh += gridDim.x) {
    if (bt.ntiles[bh / p.H] == 0)
      for (int d = threadIdx.x; d < D; d += blockDim.x) p.out[(size_t)bh * D + d] = 0.f;
  }

  const T* Kg = static_cast<const T*>(p.K);
  const T* Vg = static_cast<const T*>(p.V);

  if (warp >= kNW) {
    // ----------------------------------------------------------- producers
    // Issuing a bulk copy keeps the issuing thread busy for hundreds of cycles,
    // so one thread cannot feed all the rings at HBM speed: producer pw feeds
    // the rings of consumer warps kNW/kNP*pw .. kNW/kNP*(pw+1)-1.
    const int pw = warp - kNW;
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int i = 0;
      bool ok = true;
      for (long long g = g_begin; g < g_end && ok;) {
        const Segment s = locate(bt, P, p.B, g, g_end);
        const size_t slab = ((size_t)s.b * p.H + s.h) * p.S_cap;
        for (int t = s.t0; t < s.t1; ++t, ++i) {
          if ((i % kNW) / (kNW / kNP) != pw) continue;  // another producer's ring
          const int r = i / kNW;  // use count of this warp's ring
          const int st = (i % kNW) * C::SW + r % C::SW;
          if (!mbar_wait(&empty[st], ((r / C::SW) & 1) ^ 1, abort_flag, p.status)) { ok = false; break; }
          const int key0 = t * kTK;
          const int rows = min(kTK, bt.len[s.b] - key0);
          const uint32_t bytes = (uint32_t)(rows * D * sizeof(T));
          mbar_arrive_expect_tx(&full[st], 2 * bytes);
          bulk_g2s(sK + (size_t)st * kTK * D, Kg + (slab + key0) * D, bytes, &full[st], pol);
          bulk_g2s(sV + (size_t)st * kTK * D, Vg + (slab + key0) * D, bytes, &full[st], pol);
        }
        g = s.g_end;
      }
      if (!ok) {  // let copies already issued land before the CTA exits
        for (int j = (i > NS ? i - NS : 0); j < i; ++j) {
          if ((j % kNW) / (kNW / kNP) != pw) continue;
          const int r = j / kNW;
          mbar_drain(&full[(j % kNW) * C::SW + r % C::SW], (r / C::SW) & 1);
        }
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int ctid = threadIdx.x;
  constexpr int kCT = kNW * 32;
  const int sub = lane & 7, g4 = (lane >> 3) * 4;  // lane group g takes keys 4g..4g+3 of each tile
  const float sl2 = p.scale_log2;
  int i_base = 0;
  for (long long g = g_begin; g < g_end;) {
    const Segment s = locate(bt, P, p.B, g, g_end);
    const int ntile = s.t1 - s.t0;
    const int len = bt.len[s.b];

    // q chunks of this lane (raw; the scale is applied to the finished score)
    uint4 qc[G::kNC];
    {
      const unsigned char* qrow =
          reinterpret_cast<const unsigned char*>(static_cast<const T*>(p.q) + ((size_t)s.b * p.H + s.h) * D);
#pragma unroll
      for (int m = 0; m < G::kNC; ++m) qc[m] = *reinterpret_cast<const uint4*>(qrow + (sub + 8 * m) * 16);
    }
    float m = -CUDART_INF_F, l = 0.f;
    uint64_t o2[G::kPairs];
#pragma unroll
    for (int e = 0; e < G::kPairs; ++e) o2[e] = 0ull;

    const int first = i_base + (((warp - i_base) % kNW) + kNW) % kNW;
    for (int i = first; i < i_base + ntile; i += kNW) {
      const int r = i / kNW;
      const int st = warp * C::SW + r % C::SW;
      if (!mbar_wait(&full[st], (r / C::SW) & 1, abort_flag, p.status)) break;
      const int t = s.t0 + (i - i_base);
      const int rows = min(kTK, len - t * kTK);
      const unsigned char* Kb = reinterpret_cast<const unsigned char*>(sK + (size_t)st * kTK * D);
      const unsigned char* Vb = reinterpret_cast<const unsigned char*>(sV + (size_t)st * kTK * D);

      // Copy this lane's K and V chunks of the tile to registers and hand the
      // stage back at once, so the ring stays in flight while the warp computes.
      uint4 kr[4][G::kNC], vr[4][G::kNC];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
#pragma unroll
        for (int mm = 0; mm < G::kNC; ++mm) {
          kr[kk][mm] = *reinterpret_cast<const uint4*>(Kb + (g4 + kk) * G::kRowBytes + (sub + 8 * mm) * 16);
          vr[kk][mm] = *reinterpret_cast<const uint4*>(Vb + (g4 + kk) * G::kRowBytes + (sub + 8 * mm) * 16);
        }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);

      // partial scores of this group's 4 keys over this lane's dims
      float part[4];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        float acc[2] = {0.f, 0.f};
#pragma unroll
        for (int mm = 0; mm < G::kNC; ++mm) dot_chunk<T>(qc[mm], kr[kk][mm], acc);
        part[kk] = acc[0] + acc[1];
      }
      float sc = group8_reduce4(part, lane) * sl2;  // score of key lane / 2 of the tile
      if ((lane >> 1) >= rows) sc = -CUDART_INF_F;
      const float m_new = fmaxf(m, warp_max(sc));
      const float corr = fast_exp2(m - m_new);
      const float pe = fast_exp2(sc - m_new);
      l = l * corr + ((lane & 1) ? 0.f : pe);  // each key is held by two lanes: count it once
      const uint64_t corr2 = f2pack(corr, corr);
#pragma unroll
      for (int e = 0; e < G::kPairs; ++e) o2[e] = f2mul(o2[e], corr2);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const float pk = __shfl_sync(0xffffffffu, pe, (lane & ~7) + 2 * kk);
        if (g4 + kk < rows) {  // rows past the slab end hold stale data (even NaN): skip them
          const uint64_t p2 = f2pack(pk, pk);
#pragma unroll
          for (int mm = 0; mm < G::kNC; ++mm) axpy_chunk<T>(p2, vr[kk][mm], o2 + mm * G::kPairsPerChunk);
        }
      }
      m = m_new;
    }

    // ---- merge: lane groups within the warp, then the warps of the CTA
    l = warp_sum(l);
    float* my = scratch + warp * (D + 2);
    if (lane == 0) { my[0] = m; my[1] = l; }
#pragma unroll
    for (int e = 0; e < G::kPairs; ++e) {
      float2 v = f2unpack(o2[e]);
      v.x += __shfl_xor_sync(0xffffffffu, v.x, 8);
      v.y += __shfl_xor_sync(0xffffffffu, v.y, 8);
      v.x += __shfl_xor_sync(0xffffffffu, v.x, 16);
      v.y += __shfl_xor_sync(0xffffffffu, v.y, 16);
      if (lane < 8) {
        const int d = (sub + 8 * (e / G::kPairsPerChunk)) * G::kChunkElems + 2 * (e % G::kPairsPerChunk);
        my[2 + d] = v.x;
        my[3 + d] = v.y;
      }
    }
    consumer_sync(kCT);

    float M = -CUDART_INF_F;
#pragma unroll
    for (int w = 0; w < kNW; ++w) M = fmaxf(M, scratch[w * (D + 2)]);
    float wt[kNW];
    float L = 0.f;
#pragma unroll
    for (int w = 0; w < kNW; ++w) {
      wt[w] = fast_exp2(scratch[w * (D + 2)] - M);
      L += wt[w] * scratch[w * (D + 2) + 1];
    }
    const int bh = s.b * p.H + s.h;
    if (s.c_first == s.c_last) {
      for (int d = ctid; d < D; d += kCT) {
        float O = 0.f;
#pragma unroll
        for (int w = 0; w < kNW; ++w) O += wt[w] * scratch[w * (D + 2) + 2 + d];
        p.out[(size_t)bh * D + d] = O / L;
      }
      consumer_sync(kCT);
    } else {
      float* slot = partial_slot(p.partials, blockIdx.x + bh, 1, D);
      if (ctid == 0) { slot[0] = M; slot[1] = L; }
      for (int d = ctid; d < D; d += kCT) {
        float O = 0.f;
#pragma unroll
        for (int w = 0; w < kNW; ++w) O += wt[w] * scratch[w * (D + 2) + 2 + d];
        slot[2 + d] = O;
      }
      combine_if_last(s, p.B, p.H, 1, D, p.partials, p.counters, p.out, ctid, kCT, last_flag);
    }
    i_base += ntile;
    g = s.g_end;
  }
}

template <typename T, int D>
cudaError_t launch_typed(const AttnArgs& a, cudaStream_t st) {
  using C = CrossCfg<T, D>;
  const size_t smem = C::smem_bytes(a.B);
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(cross_attn_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::smem_bytes(kMaxBatch));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const long long tiles_ub = (long long)a.B * a.H * ((a.max_kv_len + kTK - 1) / kTK);
  long long G = a.max_ctas > 0 ? a.max_ctas : sm_count();
  if (G > kMaxCtas) G = kMaxCtas;
  if (G > tiles_ub) G = tiles_ub;
  if (G < 1) G = 1;
  CrossParams p;
  p.q = a.q; p.K = a.K; p.V = a.V; p.kv_len = a.kv_len; p.out = a.out;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.counters = reinterpret_cast<unsigned*>(ws + WsLayout::counters_off());
  p.partials = reinterpret_cast<float*>(ws + WsLayout::partials_off(a.B, a.H));
  p.B = a.B; p.H = a.H; p.S_cap = a.S_cap; p.max_kv_len = a.max_kv_len;
  p.scale_log2 = a.scale * kLog2e;
  cross_attn_kernel<T, D><<<(unsigned)G, kThreads, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_cross_attn(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype == 0 && a.D == 128) return launch_typed<__nv_bfloat16, 128>(a, st);
  if (a.dtype == 0 && a.D == 64) return launch_typed<__nv_bfloat16, 64>(a, st);
  if (a.dtype == 1 && a.D == 128) return launch_typed<float, 128>(a, st);
  if (a.dtype == 1 && a.D == 64) return launch_typed<float, 64>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace glide
