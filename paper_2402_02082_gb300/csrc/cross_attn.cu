// GliDe cross-attention (Section 3.1): one draft query per (sequence, head)
// attends to every cached key/value of the target layer,
//   hd_j = SoftMax(Q^{m,j} (K^{l,j})^T / sqrt(d_k)) V^{l,j},
// with no mask at inference.
//
// The step reads every cached K and V byte once and does ~1 flop per byte, so
// it is bound by HBM bandwidth.  Design:
// * persistent grid (one CTA per SM); the key ranges of all (b, h) are cut
//   into 16-key tiles, and the tile sequence into chunks of shrinking size
//   (Chunks) that the CTAs claim at run time: SMs do not all stream at the
//   same rate, and a static equal split leaves the kernel waiting on the
//   slowest ones;
// * producer warp 0 claims the chunks (atomic counter in the workspace; a
//   CTA's first chunk is its own block index, one of level 0's G chunks, so
//   no claim delays the first copies) and passes their ids to the other warps
//   through a small shared-memory queue; all twelve warps walk the same chunk
//   sequence;
// * four producer threads (one per producer warp; issuing a bulk copy keeps
//   a thread busy for hundreds of cycles) stream K and V tiles with 1-D bulk
//   copies (TMA) into shared-memory stages guarded by mbarriers; tile j of a
//   chunk goes to consumer warp j % NW (fixed by the chunk alone, so results
//   do not depend on which CTA claimed what), and every consumer warp owns a
//   private ring of SW stages that it drains strictly in order (a warp never
//   waits on a stage whose earlier phase is still pending, so the mbarrier
//   parity cannot alias);
// * each of the NW = 8 consumer warps (two per SM sub-partition, so one
//   warp's shuffle and shared-memory latencies hide behind the other's work)
//   takes whole tiles: lanes split the head dimension, a group reduction turns
//   partial dot products into scores, and an fp32 online softmax (log2
//   domain) accumulates P.V;
// * at the end of a (b, h) segment every consumer warp stores its own partial
//   (max, sum, o) and moves on: no warp waits for another, no CTA for another
//   CTA, and no fence or atomic sits between two segments;
// * a second, small kernel (launched as a programmatic dependent of the first,
//   so its launch overlaps the first one's tail) merges the partials of each
//   (b, h), one warp each, into the output.
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
constexpr int kQN = 4;       // chunk-queue entries
constexpr int kLevels = 6;   // chunk levels (fewer when the chunks would not fit the partial slots)

template <typename T, int D>
struct CrossCfg {
  static constexpr int kTile = kTK * D * (int)sizeof(T);
  static constexpr int kFit = (192 * 1024) / (2 * kTile * kNW);
  static constexpr int SW = kFit > 3 ? 3 : (kFit < 1 ? 1 : kFit);   // stages per consumer warp
  static constexpr int NS = SW * kNW;
  static constexpr size_t kStageBytes = (size_t)NS * kTile;
  static constexpr size_t off_K = 0;
  static constexpr size_t off_V = kStageBytes;
  static constexpr size_t off_bar = 2 * kStageBytes;                   // full[NS], empty[NS], qfull[kQN], qempty[kQN]
  static constexpr size_t off_queue = off_bar + (2 * NS + 2 * kQN) * sizeof(uint64_t);   // chunk ids
  static constexpr size_t off_misc = off_queue + kQN * sizeof(int);
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
  unsigned* claim;      // chunk-claim counter (zero between launches)
  unsigned* done;       // CTAs that made their last claim (zero between launches)
  int2* ranges;         // per (b, h): first and last chunk that hold its tiles (-1: none)
  float* partials;
  int B, H, S_cap, max_kv_len;
  int levels;
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
  uint64_t* qfull = empty + NS;
  uint64_t* qempty = qfull + kQN;
  volatile int* qchunk = reinterpret_cast<volatile int*>(smem + C::off_queue);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::off_misc);
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
    for (int s = 0; s < kQN; ++s) {
      mbar_init(&qfull[s], 1);                 // the claiming thread
      mbar_init(&qempty[s], kNP - 1 + kNW);    // every other warp has read the entry
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  pdl_wait();  // shared-memory set-up above; every global access below
  build_batch_tiles(bt, p.kv_len, p.B, p.H, p.max_kv_len, 0, kTK);  // ends with __syncthreads

  __shared__ Chunks s_chunks;  // one copy of the level table, not one per thread
  if (warp == 0) s_chunks.init_warp(bt.start[p.B], gridDim.x, p.levels, lane);
  __syncthreads();
  const Chunks& CK = s_chunks;
  const int nchunks = CK.count();

  // The id of the q-th chunk this CTA works on (-1: no more work), read from
  // the queue by every warp but the claiming one.  Returns false on abort.
  auto next_chunk = [&](int q, int& k) -> bool {
    const int slot = q % kQN;
    if (!mbar_wait(&qfull[slot], (q / kQN) & 1, abort_flag, p.status)) return false;
    k = qchunk[slot];
    __syncwarp();
    if (lane == 0) mbar_arrive(&qempty[slot]);
    return true;
  };

  const T* Kg = static_cast<const T*>(p.K);
  const T* Vg = static_cast<const T*>(p.V);

  if (warp >= kNW) {
    // ----------------------------------------------------------- producers
    // Issuing a bulk copy keeps the issuing thread busy for hundreds of cycles,
    // so one thread cannot feed all the rings at HBM speed: producer pw feeds
    // the rings of consumer warps kNW/kNP*pw .. kNW/kNP*(pw+1)-1.  Producer 0
    // also claims the chunks, each when it starts on it.
    const int pw = warp - kNW;
    constexpr int kPer = kNW / kNP;  // consumer rings per producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int uses[kPer] = {};  // tiles issued so far into each of this producer's rings
      int q = 0;
      bool ok = true;
      while (ok) {
        int k;
        if (pw == 0) {
          const int slot = q % kQN;
          if (!mbar_wait(&qempty[slot], ((q / kQN) & 1) ^ 1, abort_flag, p.status)) { ok = false; break; }
          // The first chunk of CTA c is chunk c (the G chunks of level 0, one
          // each: no atomic on the path to the first copy); later ones are
          // claimed from the counter, which hands out chunks G, G + 1, ...
          const unsigned c = q == 0 ? blockIdx.x : gridDim.x + atomicAdd(p.claim, 1u);
          k = c < (unsigned)nchunks ? (int)c : -1;
          qchunk[slot] = k;
          mbar_arrive(&qfull[slot]);
          if (k < 0) {  // this CTA's last claim; the last CTA to make it re-arms the counters
            if (atomicAdd(p.done, 1u) == gridDim.x - 1) {
              *p.claim = 0u;
              *p.done = 0u;
            }
          }
        } else if (!next_chunk(q, k)) {
          ok = false;
          break;
        }
        ++q;
        if (k < 0) break;
        const long long c_begin = CK.begin(k), c_end = CK.end(k);
        for (long long g = c_begin; g < c_end && ok;) {
          const Segment s = locate(bt, CK, p.B, g, c_end);
          const size_t slab = ((size_t)s.b * p.H + s.h) * p.S_cap;
          const int j0 = (int)(g - c_begin);  // chunk-relative index of the segment's first tile
          for (int t = s.t0; t < s.t1; ++t) {
            const int w = (j0 + t - s.t0) % kNW;
            if (w / kPer != pw) continue;  // another producer's ring
            int r = 0;  // use count of warp w's ring
#pragma unroll
            for (int e = 0; e < kPer; ++e)
              if (w % kPer == e) r = uses[e]++;
            const int st = w * C::SW + r % C::SW;
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
      }
      if (!ok) {  // let copies already issued land before the CTA exits
#pragma unroll
        for (int e = 0; e < kPer; ++e) {
          const int w = pw * kPer + e;
          for (int r = (uses[e] > C::SW ? uses[e] - C::SW : 0); r < uses[e]; ++r)
            mbar_drain(&full[w * C::SW + r % C::SW], (r / C::SW) & 1);
        }
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  // The chunk range of every (b, h), for the merge kernel (written here, off
  // the producers' path to their first copies).
  for (int bh = blockIdx.x * (kNW * 32) + threadIdx.x; bh < p.B * p.H; bh += gridDim.x * (kNW * 32)) {
    const int b = bh / p.H, h = bh - b * p.H;
    const int nt = bt.ntiles[b];
    int2 r = make_int2(-1, -1);
    if (nt > 0) {
      const long long first = bt.start[b] + (long long)h * nt;
      r = make_int2(CK.cta_of(first), CK.cta_of(first + nt - 1));
    }
    p.ranges[bh] = r;
  }

  // A sequence with no cached keys has an empty softmax: its output is zero.
  for (int bh = blockIdx.x; bh < p.B * p.H; bh += gridDim.x) {
    if (bt.ntiles[bh / p.H] == 0)
      for (int d = threadIdx.x; d < D; d += kNW * 32) p.out[(size_t)bh * D + d] = 0.f;
  }

  const int sub = lane & 7, g4 = (lane >> 3) * 4;  // lane group g takes keys 4g..4g+3 of each tile
  const float sl2 = p.scale_log2;
  int uses = 0, q = 0;  // tiles this warp has taken from its ring so far
  bool ok = true;
  while (ok) {
    int k;
    if (!next_chunk(q, k)) break;
    ++q;
    if (k < 0) break;
    const long long c_begin = CK.begin(k), c_end = CK.end(k);
    for (long long g = c_begin; g < c_end && ok;) {
      const Segment s = locate(bt, CK, p.B, g, c_end);
      const int j0 = (int)(g - c_begin);  // chunk-relative index of the segment's first tile
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

      const int first = j0 + (((warp - j0) % kNW) + kNW) % kNW;
      for (int j = first; j < j0 + ntile; j += kNW) {
        const int r = uses++;
        const int st = warp * C::SW + r % C::SW;
        if (!mbar_wait(&full[st], (r / C::SW) & 1, abort_flag, p.status)) { ok = false; break; }
        const int t = s.t0 + (j - j0);
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
      if (!ok) break;

      // ---- this warp's partial of the segment: lane groups merged, lanes 0-7
      // hold o; written to the warp's slot of (chunk k, b, h)
      l = warp_sum(l);
      const int bh = s.b * p.H + s.h;
      float* my = partial_slot(p.partials, k + bh, kNW, D) + (size_t)warp * (D + 2);
#pragma unroll
      for (int e = 0; e < G::kPairs; ++e) {
        float2 v = f2unpack(o2[e]);
        v.x += __shfl_xor_sync(0xffffffffu, v.x, 8);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, 8);
        v.x += __shfl_xor_sync(0xffffffffu, v.x, 16);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, 16);
        if (lane < 8 && m != -CUDART_INF_F) {
          const int d = (sub + 8 * (e / G::kPairsPerChunk)) * G::kChunkElems + 2 * (e % G::kPairsPerChunk);
          *reinterpret_cast<float2*>(my + 2 + d) = v;
        }
      }
      if (lane == 0) *reinterpret_cast<float2*>(my) = make_float2(m, l);
      g = s.g_end;
    }
  }
}

// Merges, for each (b, h), the partials of every consumer warp of every chunk
// that holds part of its keys (slots (c + b*H + h) * 8 + w for c in its chunk
// range): out = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s.  One CTA per
// (b, h): warp w takes partials w, w + 16, ..., the loads of up to
// kMergeGroup of them issued together (one round of loads for a (b, h) with
// up to 128 partials), each lane holding D / 32 columns as float2 pairs (a
// partial row is 8-byte aligned), and folds them into a running (max, sum, o);
// the 16 warps' results meet in shared memory.  A partial whose max is -inf
// (a warp that had no tile of the segment) has weight 0 and its o never
// reaches a sum.
constexpr int kMergeWarps = 16;
constexpr int kMergeGroup = 8;  // partials per warp whose loads are issued together
template <int D>
__global__ void __launch_bounds__(kMergeWarps * 32) cross_merge_kernel(const int2* ranges, const float* partials,
                                                                      float* out, int BH) {
  constexpr int kPairs = D / 64;
  __shared__ float red[kMergeWarps][D];
  __shared__ float2 stat[kMergeWarps];
  // The next kernel may be scheduled now, onto the SMs this small grid leaves
  // free; it waits for this merge to complete before it touches memory.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  pdl_wait();  // the partials of the attention kernel are complete
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int bh = blockIdx.x; bh < BH; bh += gridDim.x) {
    const int2 r = ranges[bh];
    if (r.x < 0) continue;  // a sequence with no cached keys: the attention kernel wrote zeros
    const int nsl = kNW * (r.y - r.x + 1);
    const float* base = partials + (size_t)(r.x + bh) * kNW * (D + 2);  // the slots are adjacent
    float M = -CUDART_INF_F, L = 0.f;
    float2 acc[kPairs];
#pragma unroll
    for (int k = 0; k < kPairs; ++k) acc[k] = make_float2(0.f, 0.f);
    for (int q0 = warp; q0 < nsl; q0 += kMergeWarps * kMergeGroup) {
      float2 ml[kMergeGroup], o[kMergeGroup][kPairs];
#pragma unroll
      for (int u = 0; u < kMergeGroup; ++u) {
        const int qq = q0 + u * kMergeWarps;
        const float* row = base + (size_t)(qq < nsl ? qq : q0) * (D + 2);
        ml[u] = __ldcg(reinterpret_cast<const float2*>(row));
#pragma unroll
        for (int k = 0; k < kPairs; ++k) o[u][k] = __ldcg(reinterpret_cast<const float2*>(row + 2 + 64 * k + 2 * lane));
        if (qq >= nsl) ml[u].x = -CUDART_INF_F;
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
    if (lane == 0) stat[warp] = make_float2(M, L);
#pragma unroll
    for (int k = 0; k < kPairs; ++k) *reinterpret_cast<float2*>(&red[warp][64 * k + 2 * lane]) = acc[k];
    __syncthreads();
    float Mt = -CUDART_INF_F;
#pragma unroll
    for (int w = 0; w < kMergeWarps; ++w) Mt = fmaxf(Mt, stat[w].x);
    float Lt = 0.f, wt[kMergeWarps];
#pragma unroll
    for (int w = 0; w < kMergeWarps; ++w) {
      wt[w] = stat[w].x == -CUDART_INF_F ? 0.f : fast_exp2(stat[w].x - Mt);
      Lt += wt[w] * stat[w].y;
    }
    const float li = Lt > 0.f ? 1.f / Lt : 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < kMergeWarps; ++w) v += wt[w] * red[w][d];
      out[(size_t)bh * D + d] = v * li;
    }
    __syncthreads();
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
  p.claim = reinterpret_cast<unsigned*>(ws + WsLayout::kClaimOff);
  p.done = reinterpret_cast<unsigned*>(ws + WsLayout::kDoneOff);
  p.ranges = reinterpret_cast<int2*>(ws + WsLayout::ranges_off(a.B, a.H));
  p.partials = reinterpret_cast<float*>(ws + WsLayout::partials_off(a.B, a.H));
  p.B = a.B; p.H = a.H; p.S_cap = a.S_cap; p.max_kv_len = a.max_kv_len;
  // chunks (levels x G) index the partial slots, of which there are kMaxCtas
  int levels = (int)(kMaxCtas / G);
  p.levels = levels > kLevels ? kLevels : (levels < 1 ? 1 : levels);
  p.scale_log2 = a.scale * kLog2e;
  cudaError_t e = launch_pdl(cross_attn_kernel<T, D>, dim3((unsigned)G), dim3(kThreads), smem, st, p);
  if (e != cudaSuccess) return e;
  // The merge, also a programmatic dependent: it may be scheduled while the
  // attention kernel drains and waits (griddepcontrol.wait) until that kernel
  // has completed and its writes are visible.
  const int BH = a.B * a.H;
  return launch_pdl(cross_merge_kernel<D>, dim3((unsigned)(BH < 65535 ? BH : 65535)), dim3(kMergeWarps * 32), 0, st,
                    (const int2*)p.ranges, (const float*)p.partials, p.out, BH);
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
