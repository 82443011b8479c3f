// Tree verification attention on CUDA cores (Section 3.2): n tree queries per
// (sequence, head) attend to every cached prefix key and to the tree keys of
// their ancestors and themselves.  With grouped-query attention a slab is a
// (sequence, cached head) and serves the n x group query rows of the heads
// that share it (up to kMaxRows, in row tiles of 64, one CTA per row tile:
// the R CTAs of a share are adjacent, stream the same keys at the same time and
// so read them from DRAM about once); without tree keys (prefix only) the same
// kernel is grouped-query cross-attention.  The CaPE mask is this
// ancestor-or-self mask on CaPE's trees (proposal spine plus expansion
// leaves); the kernel takes any parent array.
//
// This is the general kernel: any dtype (bf16, fp32), D in {64, 128}.  The
// tensor-core kernel (tree_attn_tc.cu) replaces it for bf16 where it applies.
// Structure as in cross_attn.cu (persistent split-KV grid, bulk-copy ring,
// last-CTA merge); here each consumer warp owns a fixed subset of the queries
// and reads every tile, and the ancestor mask lives in shared memory as one
// 64-bit set per node, rebuilt from parent_idx at each segment.
#include <cuda_bf16.h>
#include <math_constants.h>

#include "attn_common.cuh"
#include "kernels.h"

namespace glide {
namespace {

constexpr int kTK = 32;
constexpr int kNW = 8;
constexpr int kQPW = kRowTile / kNW;  // queries per warp at most
constexpr int kThreads = (kNW + 1) * 32;

template <typename T, int D>
struct TreeCfg {
  static constexpr int E = D / 32;
  static constexpr int kTile = kTK * D * (int)sizeof(T);
  static constexpr int NS = (160 * 1024) / (2 * kTile) > 8 ? 8 : (160 * 1024) / (2 * kTile);
  static constexpr size_t kStageBytes = (size_t)NS * kTile;
  static constexpr size_t off_K = 0;
  static constexpr size_t off_V = kStageBytes;
  static constexpr size_t off_bar = 2 * kStageBytes;
  static constexpr size_t off_anc = off_bar + 2 * NS * sizeof(uint64_t);
  static constexpr size_t off_misc = off_anc + kMaxTree * sizeof(uint64_t);
  static constexpr size_t off_tab = off_misc + 16;
  static size_t smem_bytes(int B) { return off_tab + (size_t)(B + 1) * 8 + (size_t)3 * B * 4; }
};

struct TreeParams {
  const void* q;
  const void* K;
  const void* V;
  const int* kv_len;
  const int* parent;
  float* out;
  unsigned* status;
  unsigned* counters;
  float* partials;
  int B, H, S_cap, max_kv_len, n;
  int Hkv;    // cached heads (slabs are (b, cached head))
  int group;  // query heads per cached head (H / Hkv)
  int rows;   // query rows per slab: n nodes x group heads, node-major, <= kMaxRows
  int R;      // row tiles per slab: CTA x * R + y serves rows [64y, 64y + 64) of share x
  int tree;   // 1: the n tree keys follow the prefix (verification); 0: prefix only
  float scale_log2;
};

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 1) tree_attn_fma_kernel(const TreeParams p) {
  using C = TreeCfg<T, D>;
  constexpr int E = C::E;
  constexpr int NS = C::NS;
  pdl_wait();
  extern __shared__ __align__(1024) unsigned char smem[];
  T* sK = reinterpret_cast<T*>(smem + C::off_K);
  T* sV = reinterpret_cast<T*>(smem + C::off_V);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::off_bar);
  uint64_t* empty = full + NS;
  uint64_t* anc = reinterpret_cast<uint64_t*>(smem + C::off_anc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::off_misc);
  volatile int* last_flag = abort_flag + 1;
  BatchTiles bt;
  bt.start = reinterpret_cast<long long*>(smem + C::off_tab);
  bt.len = reinterpret_cast<int*>(bt.start + p.B + 1);
  bt.ntiles = bt.len + p.B;
  bt.plen = bt.ntiles + p.B;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = p.n;
  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kNW);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  build_batch_tiles(bt, p.kv_len, p.B, p.Hkv, p.max_kv_len, p.tree ? n : 0, kTK);
  if (!p.tree) {  // prefix only: a sequence with no cached keys has an empty softmax, output zero
    const long long total = (long long)p.B * n * p.H * D;
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x)
      if (bt.ntiles[idx / ((long long)n * p.H * D)] == 0) p.out[idx] = 0.f;
  }

  // this CTA: share x of the key sequence, row tile y of every slab in it
  const int x = blockIdx.x / p.R, y = blockIdx.x - x * p.R;
  const int row0 = y * kRowTile, rows_here = min(kRowTile, p.rows - row0);
  Partition P;
  P.init(bt.start[p.B], gridDim.x / p.R);
  const long long g_begin = P.begin(x), g_end = P.end(x);
  const T* Kg = static_cast<const T*>(p.K);
  const T* Vg = static_cast<const T*>(p.V);

  if (warp == kNW) {
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int i = 0;
      bool ok = true;
      for (long long g = g_begin; g < g_end && ok;) {
        const Segment s = locate(bt, P, p.B, g, g_end);
        const size_t slab = ((size_t)s.b * p.Hkv + s.h) * p.S_cap;
        for (int t = s.t0; t < s.t1; ++t, ++i) {
          const int st = i % NS;
          if (!mbar_wait(&empty[st], ((i / NS) & 1) ^ 1, abort_flag, p.status)) { ok = false; break; }
          const int key0 = t * kTK;
          const int rows = min(kTK, bt.len[s.b] - key0);
          const uint32_t bytes = (uint32_t)(rows * D * sizeof(T));
          mbar_arrive_expect_tx(&full[st], 2 * bytes);
          bulk_g2s(sK + (size_t)st * kTK * D, Kg + (slab + key0) * D, bytes, &full[st], pol);
          bulk_g2s(sV + (size_t)st * kTK * D, Vg + (slab + key0) * D, bytes, &full[st], pol);
        }
        g = s.g_end;
      }
      if (!ok) {
        for (int j = (i > NS ? i - NS : 0); j < i; ++j) mbar_drain(&full[j % NS], (j / NS) & 1);
      }
    }
    return;
  }

  const int ctid = threadIdx.x;
  constexpr int kCT = kNW * 32;
  const float sl2 = p.scale_log2;
  int i_base = 0;
  for (long long g = g_begin; g < g_end;) {
    const Segment s = locate(bt, P, p.B, g, g_end);
    const int ntile = s.t1 - s.t0;
    const int len = bt.len[s.b];
    const int plen = bt.plen[s.b];

    // ancestor-or-self set of every node; a parent outside [-1, j) ends the walk
    if (ctid < n && p.tree) {  // prefix only: no tree keys, no parent array
      uint64_t mask = 0;
      int j = ctid;
      for (int step = 0; step < kMaxTree && j >= 0; ++step) {
        mask |= 1ull << j;
        const int pj = p.parent[(size_t)s.b * n + j];
        j = (pj >= 0 && pj < j) ? pj : -1;
      }
      anc[ctid] = mask;
    }
    consumer_sync(kCT);

    float q[kQPW][E], o[kQPW][E], m[kQPW], l[kQPW];
    uint64_t am[kQPW];
    // query row iq of the slab (row0 + warp + j * kNW): node iq / group, head
    // s.h * group + iq % group
#pragma unroll
    for (int j = 0; j < kQPW; ++j) {
      const int iq = row0 + warp + j * kNW;
      m[j] = -CUDART_INF_F;
      l[j] = 0.f;
      am[j] = 0;
#pragma unroll
      for (int e = 0; e < E; ++e) { o[j][e] = 0.f; q[j][e] = 0.f; }
      if (warp + j * kNW < rows_here) {
        const int node = iq / p.group;
        load_row_chunk<T, E>(static_cast<const T*>(p.q) + out_row(s.b, s.h, iq, p.rows, p.group, p.H) * D + lane * E,
                             q[j]);
#pragma unroll
        for (int e = 0; e < E; ++e) q[j][e] *= sl2;
        am[j] = p.tree ? anc[node] : 0ull;
      }
    }

    for (int i = i_base; i < i_base + ntile; ++i) {
      const int st = i % NS;
      if (!mbar_wait(&full[st], (i / NS) & 1, abort_flag, p.status)) break;
      const int t = s.t0 + (i - i_base);
      const int key = t * kTK + lane;
      const int rows = min(kTK, len - t * kTK);
      const T* Kt = sK + (size_t)st * kTK * D + lane * E;
      const T* Vt = sV + (size_t)st * kTK * D + lane * E;
#pragma unroll
      for (int j = 0; j < kQPW; ++j) {
        if (warp + j * kNW >= rows_here) break;
        float part[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          float kf[E];
          load_row_chunk<T, E>(Kt + k * D, kf);
          float acc = 0.f;
#pragma unroll
          for (int e = 0; e < E; ++e) acc = fmaf(q[j][e], kf[e], acc);
          part[k] = acc;
        }
        float sc = transpose_reduce32(part, lane);
        const bool visible = lane < rows && (key < plen || ((am[j] >> (key - plen)) & 1ull));
        if (!visible) sc = -CUDART_INF_F;
        const float tmax = warp_max(sc);
        if (tmax == -CUDART_INF_F) continue;  // nothing visible to this query here
        const float m_new = fmaxf(m[j], tmax);
        const float corr = fast_exp2(m[j] - m_new);
        const float pe = fast_exp2(sc - m_new);
        l[j] = l[j] * corr + pe;
#pragma unroll
        for (int e = 0; e < E; ++e) o[j][e] *= corr;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          if (k < rows) {
            const float pk = __shfl_sync(0xffffffffu, pe, k);
            float vf[E];
            load_row_chunk<T, E>(Vt + k * D, vf);
#pragma unroll
            for (int e = 0; e < E; ++e) o[j][e] = fmaf(pk, vf[e], o[j][e]);
          }
        }
        m[j] = m_new;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }

    const int bh = s.b * p.Hkv + s.h;
    const bool single = s.c_first == s.c_last;
    float* slot = partial_slot(p.partials, x + bh, p.rows, D);
#pragma unroll
    for (int j = 0; j < kQPW; ++j) {
      if (warp + j * kNW >= rows_here) break;
      const int iq = row0 + warp + j * kNW;
      const float L = warp_sum(l[j]);
      if (single) {
        float* dst = p.out + out_row(s.b, s.h, iq, p.rows, p.group, p.H) * D + lane * E;
#pragma unroll
        for (int e = 0; e < E; ++e) dst[e] = o[j][e] / L;
      } else {
        float* row = slot + (size_t)iq * (D + 2);
        if (lane == 0) { row[0] = m[j]; row[1] = L; }
#pragma unroll
        for (int e = 0; e < E; ++e) row[2 + lane * E + e] = o[j][e];
      }
    }
    if (single) consumer_sync(kCT);
    else combine_if_last(s, p.Hkv, p.rows, row0, rows_here, row_tile_counter(s.b, s.h, p.Hkv, p.R, y), D, p.group,
                         p.H, p.partials, p.counters, p.out, ctid, kCT, last_flag);
    i_base += ntile;
    g = s.g_end;
  }
}

template <typename T, int D>
cudaError_t launch_typed(const AttnArgs& a, cudaStream_t st) {
  using C = TreeCfg<T, D>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tree_attn_fma_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::smem_bytes(kMaxBatch));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const long long tiles_ub = (long long)a.B * a.Hkv * ((a.max_kv_len + (a.tree ? a.nq : 0) + kTK - 1) / kTK);
  const int rows = a.nq * (a.H / a.Hkv);
  const int R = (rows + kRowTile - 1) / kRowTile;
  // G shares of the key sequence, R CTAs (row tiles) per share
  long long G = a.max_ctas > 0 ? a.max_ctas : sm_count() / R;
  if (G > kMaxCtas) G = kMaxCtas;
  if (G > tiles_ub) G = tiles_ub;
  if (G < 1) G = 1;
  TreeParams p;
  p.q = a.q; p.K = a.K; p.V = a.V; p.kv_len = a.kv_len; p.parent = a.parent; p.out = a.out;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.counters = reinterpret_cast<unsigned*>(ws + WsLayout::counters_off());
  p.partials = reinterpret_cast<float*>(ws + WsLayout::partials_off(a.B, a.H));
  p.B = a.B; p.H = a.H; p.S_cap = a.S_cap; p.max_kv_len = a.max_kv_len; p.n = a.nq;
  p.Hkv = a.Hkv; p.group = a.H / a.Hkv; p.rows = rows; p.R = R; p.tree = a.tree;
  p.scale_log2 = a.scale * kLog2e;
  return launch_pdl(tree_attn_fma_kernel<T, D>, dim3((unsigned)(G * R)), dim3(kThreads), C::smem_bytes(a.B), st, p);
}

}  // namespace

cudaError_t launch_tree_attn_fma(const AttnArgs& a, cudaStream_t st) {
  if (a.nq * (a.H / a.Hkv) > kMaxRows) return cudaErrorInvalidValue;  // the abi rejects this first
  if (a.dtype == 0 && a.D == 128) return launch_typed<__nv_bfloat16, 128>(a, st);
  if (a.dtype == 0 && a.D == 64) return launch_typed<__nv_bfloat16, 64>(a, st);
  if (a.dtype == 1 && a.D == 128) return launch_typed<float, 128>(a, st);
  if (a.dtype == 1 && a.D == 64) return launch_typed<float, 64>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace glide
