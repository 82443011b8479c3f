// Tree verification attention in 128-row tiles on the tcgen05 tensor cores,
// for grouped-query slabs (Section 3.2's verification of a CaPE tree, under
// the ancestor-or-self mask, on a target with fewer cached heads than query
// heads such as Mistral-7B, Section 4.1) and any slab of more than 64 query
// rows; without tree keys (a prefix-only mode) the same kernel serves the
// draft's grouped-query cross-attention (Section 3.1), the group's queries as
// a slab's rows.
//
// A slab is a (sequence, cached head) with n tree nodes x H / H_kv query
// heads as its rows, node-major: a 33-node CaPE tree on Mistral-7B's 32 query
// over 8 cached heads has 132.  The 64-row kernel serves such a slab in three
// row tiles whose CTAs each run the whole 64-key tile loop (the softmax chain
// sets a ~1400-cycle period per tile), so the work grows with the row tiles
// while the bytes stay the same.  Here a row tile is 128 rows and a key tile
// 128 keys, the shape of the training-time block-mask kernel:
//   S = Q K^T : M = 128 query rows, N = 128 keys, K = D, operands in shared memory
//   O += P V  : M = 128, N = D, K = 64 keys per key half, P in tensor memory
// which does four times the (row, key) pairs of a 64 x 64 tile per softmax
// pass; at one row tile that leaves the loop ~20% faster than the HBM pace of
// an SM, where the 64-row kernel's loop runs right at it, so grouped-query
// slabs of few rows come here too.  Tensor memory holds three S buffers of
// 128 columns (S of tile i + 3 waits for P.V of tile i) and the O
// accumulator.  Two softmax groups of four
// warps take the two 64-key halves of every tile, one thread per row; the two
// threads of a row agree on each tile's row max through one TMEM column, so
// both halves use one reference max and accumulate into the one O, and each
// group writes P over the first 32 columns of its half of the S buffer.
//
// Work: the slabs' 128-key tiles are cut into G shares of equal cost (a
// segment switch counted as kSegWeight tiles), and R = ceil(rows / 128)
// adjacent CTAs serve each share, CTA x * R + y taking row tile y of every
// slab in share x: the R CTAs stream the same K/V tiles at about the same
// time, so DRAM serves each tile about once and L2 the other reads.  A slab
// whose keys all fall in one share is written out directly; a split slab
// leaves one partial (max, sum, o) per share and row, and the split merge
// kernel, launched as a programmatic dependent, combines them.
//
// Q comes by 3-D TMA: the [B n, H, D] queries as a box of 128 / group nodes x
// group heads x 64 head dims is exactly the 128 node-major rows of a row tile
// (so group must divide 128).  Rows past the slab's n x group are padding:
// whatever they read (another sequence's queries or the zero fill), their
// results are never written.
//
// Roles (384 threads, one CTA per SM):
//   warps 0-7  softmax and the segment epilogues: warp w reads TMEM lane
//              quarter w % 4 (one thread per row) and key half w / 4.
//   warp 8     lane 0: the queries of each segment and the K ring (2-D TMA,
//              128-byte swizzle), polling both.
//   warp 9     S issue (lane 0) and the TMEM allocation.
//   warp 10    P.V issue (lane 0).
//   warp 11    lane 0: the V ring.
//
// Masking: keys below the sequence's prefix length are visible to every row;
// tree key c (at prefix + c) is visible to the rows of node i iff c is an
// ancestor-or-self of i (the set built from the parent array by pointer
// jumping, at the first tile that reaches the tree keys); keys past the
// prefix and the n tree keys are masked, and their V rows are zeroed in
// shared memory before P.V (the cache beyond them may hold anything).  In the
// prefix-only mode a sequence without cached keys gets zeros.
// Online softmax in the log2 domain with a lazy reference max: O is rescaled
// in TMEM only when a tile's max exceeds the reference by more than 8.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math_constants.h>

#include "attn_common.cuh"
#include "kernels.h"
#include "tc_attn.cuh"
#include "tc_ptx.cuh"
#include "tensor_map.h"

namespace glide {
namespace {

constexpr int kBM = 128;          // query rows per row tile (MMA rows, TMEM lanes)
constexpr int kBN = 128;          // keys per tile
constexpr int kMaxStages = 4;     // K/V ring stages (the launch picks as many as fit)
constexpr int kSoftWarps = 8;     // two groups of four: the key halves of every tile
constexpr int kKProdWarp = 8;     // the queries and the K ring
constexpr int kSWarp = 9;
constexpr int kPVWarp = 10;
constexpr int kVProdWarp = 11;
constexpr int kThreads = 384;
constexpr int kTmemCols = 512;
constexpr int kSBufs = 3;                   // S / P buffers at columns 0, 128, 256
constexpr uint32_t kTmemO = kSBufs * kBN;   // the O accumulator from column 384
constexpr uint32_t kAtom = 128 * 128;       // one 128-byte-swizzle atom of 128 rows
constexpr float kRescaleLog2 = 8.0f;
// What a switch from one slab to the next costs a CTA, in 128-key tiles (the
// segment's epilogue and the pipeline start of the next, with its queries).
constexpr int kSegWeight = 4;

// ODONE has four slots (tile mod 4).  P.V completions are waited on only now
// and then (a rescale, the epilogue), when up to three products may still be
// in flight: P.V of tile i - 3 has completed once S of tile i has been read,
// but those of tiles i - 2 .. i may not have.  Four slots keep every such wait
// within one phase of its barrier; with two, a wait for tile i could pass on
// the completion of tile i - 2 (measured: the last tiles of a segment missing
// from O when the values arrived late from DRAM).
constexpr int B_KFULL = 0, B_KEMPTY = 4, B_VFULL = 8, B_VEMPTY = 12, B_QFULL = 16, B_QEMPTY = 17, B_SFULL = 18,
              B_PFULL = 21, B_BFREE = 24, B_ODONE = 27, B_MDONE = 31, kNumBars = 33;

template <int D>
struct WideCfg {
  static constexpr int kHalves = D / 64;                // swizzle atoms across the head dim
  static constexpr uint32_t kQBytes = kHalves * kAtom;  // 128 rows x D
  static constexpr uint32_t kKV = kHalves * kAtom;      // 128 keys x D
  static constexpr uint32_t off_Q = 0;
  static constexpr uint32_t off_K = kQBytes;
  // K ring of nk stages, then the V ring of nv, barriers, misc, row sums, batch table
  static __host__ __device__ uint32_t off_V(int nk) { return off_K + nk * kKV; }
  static __host__ __device__ uint32_t off_bar(int nk, int nv) { return off_V(nk) + nv * kKV; }
  static __host__ __device__ uint32_t off_misc(int nk, int nv) { return off_bar(nk, nv) + 512; }
  // the segment's row sums, [key half][row], between the two softmax groups
  static __host__ __device__ uint32_t off_lsum(int nk, int nv) { return off_misc(nk, nv) + 16; }
  static __host__ __device__ uint32_t off_tab(int nk, int nv) { return off_lsum(nk, nv) + 2 * kBM * 4; }
  static size_t smem_bytes(int B, int nk, int nv) {
    return 1024 + off_tab(nk, nv) + (size_t)(B + 1) * 8 + (size_t)(4 * B + 1) * 4;
  }
  static_assert(kTmemO + D <= kTmemCols, "TMEM columns");
  static_assert(kNumBars * 8 <= 512, "barrier area");
};

struct WideParams {
  const int* kv_len;
  const int* parent;
  float* out;
  unsigned* status;
  int2* ranges;      // per slab: the share range of a split slab, (-1, -1) otherwise
  float* partials;
  int B, H, Hkv, group, S_cap, max_kv_len, n;
  int rows;          // query rows per slab: n nodes x group heads, node-major
  int R;             // row tiles of 128 per slab
  int tree;          // 1: the n tree keys follow the prefix (verification); 0: prefix only
  int nk, nv;        // K and V ring stages
  float scale_log2;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_wide_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                          const __grid_constant__ CUtensorMap tmV, const WideParams p) {
  using C = WideCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int nk = p.nk, nv = p.nv;  // K and V ring depths
  const uint32_t off_V = C::off_V(nk);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::off_bar(nk, nv));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + C::off_misc(nk, nv));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::off_misc(nk, nv) + 4);
  float* lsum = reinterpret_cast<float*>(base + C::off_lsum(nk, nv));
  BatchTiles bt;
  bt.start = reinterpret_cast<long long*>(base + C::off_tab(nk, nv));
  bt.len = reinterpret_cast<int*>(bt.start + p.B + 1);
  bt.ntiles = bt.len + p.B;
  bt.plen = bt.ntiles + p.B;
  bt.sidx = bt.plen + p.B;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Shared-memory set-up and the tensor-map fetches come before the wait for
  // the previous kernel; every global access and the TMEM allocation after it.
  if (threadIdx.x == 0) {
    tc::prefetch_tmap(&tmQ);
    tc::prefetch_tmap(&tmK);
    tc::prefetch_tmap(&tmV);
    for (int b = 0; b < kNumBars; ++b) mbar_init(&bars[b], (b >= B_PFULL && b < B_PFULL + kSBufs) ? kSoftWarps : 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  pdl_wait();
  if (warp == kSWarp) {
    tc::tmem_alloc(tmem_slot, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  build_batch_tiles(bt, p.kv_len, p.B, p.Hkv, p.max_kv_len, p.tree ? p.n : 0, kBN);  // __syncthreads inside
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  // this CTA: share x of the key tiles, row tile y of every slab in it
  const int G = gridDim.x / p.R;
  const int x = blockIdx.x / p.R, y = blockIdx.x - x * p.R;
  const int row0 = y * kBM;
  CostPartition P;
  P.init(bt, p.B, p.Hkv, G, kSegWeight);
  const long long g_begin = P.begin(x), g_end = P.end(x);
  // one reader per tile: evict it first; R row tiles read each tile R times
  const bool one_reader = p.R == 1;

  if (warp == kKProdWarp) {
    // -------------------------------------------- producer: queries and keys
    // The queries of segment s go in once S of segment s - 1 has read the
    // previous ones; the keys run ahead independently, up to the ring depth.
    if (lane == 0) {
      const uint64_t pol_q = policy_evict_first();
      const uint64_t pol_kv = one_reader ? policy_evict_first() : policy_evict_normal();
      long long gk = g_begin, gq = g_begin;  // the next K tile's segment start, the next Q's segment
      Segment sk;
      int tk = 0;
      if (gk < g_end) {
        sk = locate(bt, P, p.B, gk, g_end);
        tk = sk.t0;
      }
      int i = 0, qs = 0;  // K tiles and query tiles issued
      uint64_t t_last = global_timer_ns();
      int spins = 0, seen = 0;
      while (gk < g_end || gq < g_end) {
        bool progressed = false;
        if (gq < g_end && mbar_test_wait(&bars[B_QEMPTY], (qs & 1) ^ 1)) {
          const Segment sq = locate(bt, P, p.B, gq, g_end);
          mbar_arrive_expect_tx(&bars[B_QFULL], C::kQBytes);
          const int z = sq.b * p.n + row0 / p.group;  // the row tile's first node in [B n, H, D]
          for (int hd = 0; hd < C::kHalves; ++hd)
            tc::tma_load_3d(base + C::off_Q + hd * kAtom, &tmQ, hd * 64, sq.h * p.group, z, &bars[B_QFULL], pol_q);
          ++qs;
          gq = sq.g_end;
          progressed = true;
        }
        if (gk < g_end && mbar_test_wait(&bars[B_KEMPTY + i % nk], ((i / nk) & 1) ^ 1)) {
          const int st = i % nk;
          const int row = (sk.b * p.Hkv + sk.h) * p.S_cap + tk * kBN;
          mbar_arrive_expect_tx(&bars[B_KFULL + st], C::kKV);
          for (int hd = 0; hd < C::kHalves; ++hd)
            tc::tma_load_2d(base + C::off_K + st * C::kKV + hd * kAtom, &tmK, hd * 64, row, &bars[B_KFULL + st],
                            pol_kv);
          ++i;
          if (++tk == sk.t1) {
            gk = sk.g_end;
            if (gk < g_end) {
              sk = locate(bt, P, p.B, gk, g_end);
              tk = sk.t0;
            }
          }
          progressed = true;
        }
        if (progressed) continue;
        __nanosleep(32);
        if (++spins < 32) continue;
        spins = 0;  // every 32 idle polls: check for an abort or a stall of more than kWaitLimitNs
        const uint64_t now = global_timer_ns();
        if (i + qs != seen) {
          seen = i + qs;
          t_last = now;
        }
        if (*abort_flag) break;
        if (now - t_last > kWaitLimitNs) {
          *abort_flag = 1;
          record_status(p.status, kStatusTimeout);
          break;
        }
      }
      if (gk < g_end || gq < g_end) {  // aborted: let issued loads land before the CTA exits
        for (int j = (i > nk ? i - nk : 0); j < i; ++j) mbar_drain(&bars[B_KFULL + j % nk], (j / nk) & 1);
        if (qs > 0) mbar_drain(&bars[B_QFULL], (qs - 1) & 1);
      }
    }
  } else if (warp == kVProdWarp) {
    // ------------------------------------------------------ producer: values
    if (lane == 0) {
      const uint64_t pol_kv = one_reader ? policy_evict_first() : policy_evict_normal();
      int i = 0;
      bool ok = true;
      for (long long g = g_begin; g < g_end && ok;) {
        const Segment sg = locate(bt, P, p.B, g, g_end);
        const int row0k = (sg.b * p.Hkv + sg.h) * p.S_cap;
        for (int t = sg.t0; t < sg.t1; ++t, ++i) {
          const int st = i % nv;
          if (!mbar_wait(&bars[B_VEMPTY + st], ((i / nv) & 1) ^ 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bars[B_VFULL + st], C::kKV);
          for (int hd = 0; hd < C::kHalves; ++hd)
            tc::tma_load_2d(base + off_V + st * C::kKV + hd * kAtom, &tmV, hd * 64, row0k + t * kBN,
                            &bars[B_VFULL + st], pol_kv);
        }
        g = sg.g_end;
      }
      if (!ok)  // aborted: let issued loads land before the CTA exits
        for (int j = (i > nv ? i - nv : 0); j < i; ++j) mbar_drain(&bars[B_VFULL + j % nv], (j / nv) & 1);
    }
  } else if (warp == kSWarp || warp == kPVWarp) {
    // ----------------------------------------------------------- MMA issue
    if (lane == 0) {
      const bool s_role = warp == kSWarp;
      constexpr uint32_t idS = tc::idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t idO = tc::idesc_bf16_f32(kBM, D, false, true);
      const uint64_t dQ = tc::sw128_desc(smem_u32(base + C::off_Q), 16, 1024);
      const uint32_t sK = smem_u32(base + C::off_K), sV = smem_u32(base + off_V);
      bool ok = true;
      int i = 0, seg = 0;
      for (long long g = g_begin; g < g_end && ok; ++seg) {
        const Segment s = locate(bt, P, p.B, g, g_end);
        for (int t = s.t0; t < s.t1; ++t, ++i) {
          const int bi = i % kSBufs;
          if (s_role) {
            // S(i) = Q K(i)^T into buffer i % 3, once P.V of tile i - 3 has read that buffer
            if ((t == s.t0 && !mbar_wait(&bars[B_QFULL], seg & 1, abort_flag, p.status)) ||
                !mbar_wait(&bars[B_KFULL + i % nk], (i / nk) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_BFREE + bi], ((i / kSBufs) & 1) ^ 1, abort_flag, p.status)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint64_t dK = tc::sw128_desc(sK + (i % nk) * C::kKV, 16, 1024);
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint64_t step = desc_step((ks >> 2) * kAtom + (ks & 3) * 32);
              tc::mma_bf16(tmem + bi * kBN, dQ + step, dK + step, idS, ks > 0 ? 1u : 0u);
            }
            tc::mma_commit(&bars[B_SFULL + bi]);
            tc::mma_commit(&bars[B_KEMPTY + i % nk]);
            if (t == s.t1 - 1) tc::mma_commit(&bars[B_QEMPTY]);
          } else {
            // O (+)= P_0(i) V_0(i) + P_1(i) V_1(i) over the key halves h = 0, 1: P_h in
            // columns 64h .. 64h+31 of buffer i % 3; the segment's first tile starts O
            if (!mbar_wait(&bars[B_PFULL + bi], (i / kSBufs) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_VFULL + i % nv], (i / nv) & 1, abort_flag, p.status)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint64_t dV = tc::sw128_desc(sV + (i % nv) * C::kKV, kAtom, 1024);
            const uint32_t pcol = tmem + bi * kBN;
            tc::mma_bf16_ts(tmem + kTmemO, pcol, dV, idO, t == s.t0 ? 0u : 1u);
#pragma unroll
            for (int ks = 1; ks < kBN / 16; ++ks)
              tc::mma_bf16_ts(tmem + kTmemO, pcol + (ks >> 2) * 64 + (ks & 3) * 8, dV + desc_step(ks * 16 * 128),
                              idO, 1u);
            tc::mma_commit(&bars[B_VEMPTY + i % nv]);
            tc::mma_commit(&bars[B_ODONE + (i & 3)]);
            tc::mma_commit(&bars[B_BFREE + bi]);
          }
        }
        g = s.g_end;
      }
      const int role = s_role ? 0 : 1;
      tc::mma_commit(&bars[B_MDONE + role]);  // every MMA finished before TMEM is released
      mbar_drain(&bars[B_MDONE + role], 0);
    }
  } else {
    // ----------------------------------------------- softmax and epilogues
    const int kh = warp >> 2, quarter = warp & 3;
    const int r = quarter * 32 + lane;  // this thread's row in the tile (its TMEM lane)
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    const uint32_t o_col = kTmemO + kh * (D / 2);  // this group's half of the O columns
    const int sid = threadIdx.x;                   // 0..255 among the softmax threads
    const float sl2 = p.scale_log2;
    const int qrow = row0 + r;  // the slab's query row
    const bool valid = qrow < p.rows;
    const int node = valid ? qrow / p.group : 0;
    const OutMap om{p.group, p.H};
    bool dead = false;

    // The share range of every slab split over several shares, for the merge
    // kernel ((-1, -1): written out directly).
    constexpr int kST = kSoftWarps * 32;
    if (y == 0)
      for (int bh = x * kST + sid; bh < p.B * p.Hkv; bh += G * kST) {
        const int b = bh / p.Hkv, nt = bt.ntiles[b];
        int2 rg = make_int2(-1, -1);
        if (nt > 0) {
          const long long first = bt.start[b] + (long long)(bh - b * p.Hkv) * nt;
          const int cf = P.cta_of(first), cl = P.cta_of(first + nt - 1);
          if (cf != cl) rg = make_int2(cf, cl);
        }
        p.ranges[bh] = rg;
      }
    if (!p.tree) {  // prefix only: a sequence without cached keys gets zeros (an empty softmax)
      const long long total = (long long)p.B * p.n * p.H * D;
      for (long long idx = (long long)blockIdx.x * kST + sid; idx < total; idx += (long long)gridDim.x * kST)
        if (bt.ntiles[idx / ((long long)p.n * p.H * D)] == 0) p.out[idx] = 0.f;
    }

    int i = 0;  // CTA-local key tile
    for (long long g = g_begin; g < g_end;) {
      const Segment s = locate(bt, P, p.B, g, g_end);
      const int plen = bt.plen[s.b], len = bt.len[s.b];
      // this row's node's ancestor-or-self set, found at the first tile that
      // reaches the tree keys
      uint64_t anc = 0;
      bool anc_ready = false;
      float m_used = -CUDART_INF_F, l = 0.f;  // l: this key half's share of the row sum
      for (int t = s.t0; t < s.t1; ++t, ++i) {
        const int bi = i % kSBufs;
        uint32_t sv[64];
        if (!dead) dead = !warp_wait(&bars[B_SFULL + bi], (i / kSBufs) & 1, abort_flag, p.status);
        if (!dead) {
          tc::fence_after_sync();
          tc::tmem_ld32(lane_base + bi * kBN + kh * 64, *reinterpret_cast<uint32_t(*)[32]>(sv));
          tc::tmem_ld32(lane_base + bi * kBN + kh * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(sv + 32));
          tc::tmem_wait_ld();
        } else {
#pragma unroll
          for (int e = 0; e < 64; ++e) sv[e] = 0u;
        }
        // keys of this half from k0: the prefix is visible, tree key c only to
        // the rows of c's descendants-or-self, and nothing past the tree
        const int k0 = t * kBN + kh * 64;
        if (k0 + 64 > plen) {  // warp-uniform
          if (p.tree && !anc_ready) {
            anc = ancestors(p.parent + (size_t)s.b * p.n, p.n, node, valid, lane);
            anc_ready = true;
          }
#pragma unroll
          for (int e = 0; e < 64; ++e) {
            const int kk = k0 + e;
            const bool vis = kk < plen || (kk < len && ((anc >> ((kk - plen) & 63)) & 1ull));
            sv[e] = vis ? sv[e] : 0xff800000u;
          }
        }
        float mx[4] = {__uint_as_float(sv[0]), __uint_as_float(sv[1]), __uint_as_float(sv[2]),
                       __uint_as_float(sv[3])};
#pragma unroll
        for (int e = 4; e < 64; e += 8) {
          mx[0] = fmax3(mx[0], __uint_as_float(sv[e]), __uint_as_float(sv[e + 1]));
          mx[1] = fmax3(mx[1], __uint_as_float(sv[e + 2]), __uint_as_float(sv[e + 3]));
          if (e + 4 < 64) {
            mx[2] = fmax3(mx[2], __uint_as_float(sv[e + 4]), __uint_as_float(sv[e + 5]));
            mx[3] = fmax3(mx[3], __uint_as_float(sv[e + 6]), __uint_as_float(sv[e + 7]));
          }
        }
        float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;
        // the row max over both key halves: through column 63 of each half,
        // already read; the pair barrier orders the partner's read after the write
        if (!dead) {
          tc::tmem_st1(lane_base + bi * kBN + kh * 64 + 63, __float_as_uint(tmax));
          tc::tmem_wait_st();
        }
        tc::fence_before_sync();
        pair_sync(quarter);
        if (!dead) {
          tc::fence_after_sync();
          const uint32_t o = tc::tmem_ld1(lane_base + bi * kBN + (kh ^ 1) * 64 + 63);
          tc::tmem_wait_ld();
          tmax = fmaxf(tmax, __uint_as_float(o));
        }
        const bool need = tmax > m_used + kRescaleLog2;
        if (__any_sync(0xffffffffu, need)) {
          const float m_new = need ? tmax : m_used;
          const float f = need ? fast_exp2(m_used - m_new) : 1.f;
          l *= f;
          if (t > s.t0 && !dead) {  // O holds the P.V of this segment's earlier tiles: rescale this group's half
            dead = !warp_wait(&bars[B_ODONE + ((i - 1) & 3)], ((i - 1) >> 2) & 1, abort_flag, p.status);
            if (!dead) {
              tc::fence_after_sync();
#pragma unroll 1
              for (int c = 0; c < D / 64; ++c) {
                uint32_t o[32];
                tc::tmem_ld32(lane_base + o_col + c * 32, o);
                tc::tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * f);
                tc::tmem_st32(lane_base + o_col + c * 32, o);
              }
              tc::tmem_wait_st();
            }
          }
          m_used = m_new;
        }
        const float m_eff = m_used == -CUDART_INF_F ? 0.f : m_used;
        const uint64_t sc2 = f2(sl2, sl2), nm2 = f2(-m_eff, -m_eff);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
        uint32_t pk[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          float x0, x1;
          unf2(ffma2(f2(__uint_as_float(sv[2 * e]), __uint_as_float(sv[2 * e + 1])), sc2, nm2), x0, x1);
          const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
          acc[e & 3] = fadd2(acc[e & 3], f2(p0, p1));
          pk[e] = pack_bf16x2(p0, p1);
        }
        {
          float a0, a1, b0, b1;
          unf2(fadd2(acc[0], acc[1]), a0, a1);
          unf2(fadd2(acc[2], acc[3]), b0, b1);
          l += (a0 + a1) + (b0 + b1);
        }
        if (!dead) {  // P over the first 32 columns of this half's part of the S buffer
          tc::tmem_st32(lane_base + bi * kBN + kh * 64, pk);
          tc::tmem_wait_st();
        }
        const int vrows = len - t * kBN;
        if (vrows < kBN) {  // the slab's last tile: clear V rows past its last key
          const int st = i % nv;
          if (!dead) dead = !warp_wait(&bars[B_VFULL + st], (i / nv) & 1, abort_flag, p.status);
          if (!dead)
            for (int idx = sid; idx < (kBN - vrows) * C::kHalves * 8; idx += kST) {
              const int row = vrows + idx / (C::kHalves * 8), rem = idx % (C::kHalves * 8);
              *reinterpret_cast<uint4*>(base + off_V + st * C::kKV + (rem >> 3) * kAtom + row * 128 + (rem & 7) * 16) =
                  make_uint4(0u, 0u, 0u, 0u);
            }
          tc::fence_async_smem();
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_PFULL + bi]);
      }

      // ---- segment epilogue: the row sum over both halves, then each group
      // writes its half of the head dims, O / l or a split partial.  The next
      // segment's first P.V (which starts O afresh) waits for this group's
      // P of that tile, so O is read here before it is overwritten.
      lsum[kh * kBM + r] = l;
      pair_sync(quarter);
      const float L = lsum[r] + lsum[kBM + r];
      const int jl = i - 1;  // the segment's last tile
      if (!dead) dead = !warp_wait(&bars[B_ODONE + (jl & 3)], (jl >> 2) & 1, abort_flag, p.status);
      if (!dead) {
        tc::fence_after_sync();
        uint32_t o[D / 2];
#pragma unroll
        for (int c = 0; c < D / 64; ++c)
          tc::tmem_ld32(lane_base + o_col + c * 32, *reinterpret_cast<uint32_t(*)[32]>(o + 32 * c));
        tc::tmem_wait_ld();
        if (valid) {
          if (s.c_first == s.c_last) {  // the whole slab in this share: the output row
            const float inv = L > 0.f ? 1.f / L : 0.f;
            float* dst = p.out + om.row(s.b, s.h, qrow, p.rows) * D + kh * (D / 2);
#pragma unroll
            for (int e = 0; e < D / 2; e += 4)
              *reinterpret_cast<float4*>(dst + e) =
                  make_float4(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv,
                              __uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
          } else {  // the share's partial [max, sum, o] (a partial row is 8-byte aligned)
            float* dst = partial_slot(p.partials, x + s.b * p.Hkv + s.h, p.rows, D) + (size_t)qrow * (D + 2);
            if (kh == 0) *reinterpret_cast<float2*>(dst) = make_float2(m_used, L);
#pragma unroll
            for (int e = 0; e < D / 2; e += 2)
              *reinterpret_cast<float2*>(dst + 2 + kh * (D / 2) + e) =
                  make_float2(__uint_as_float(o[e]), __uint_as_float(o[e + 1]));
          }
        }
      }
      g = s.g_end;
    }
  }

  __syncwarp();  // the producer and MMA warps reconverge after their single-lane loops
  tc::fence_before_sync();
  __syncthreads();
  if (warp == kSWarp) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------- host
template <int D>
cudaError_t launch_typed(const AttnArgs& a, cudaStream_t st) {
  using C = WideCfg<D>;
  static bool configured = false;
  const int limit = smem_optin_bytes();
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tree_attn_wide_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  // As many stages as fit, the K ring first: S runs up to three tiles ahead of
  // P.V, so the keys are needed earlier than the values.
  int nk = kMaxStages, nv = kMaxStages;
  while ((nk > 2 || nv > 2) && C::smem_bytes(a.B, nk, nv) > (size_t)limit) {
    if (nv >= nk && nv > 2)
      --nv;
    else
      --nk;
  }
  if (C::smem_bytes(a.B, nk, nv) > (size_t)limit) return cudaErrorNotSupported;
  const int group = a.H / a.Hkv;
  CUtensorMap mq, mk, mv;
  const long long kv_rows = (long long)a.B * a.Hkv * a.S_cap;
  if (!make_bf16_rows3_map(&mq, a.q, D, a.H, (long long)a.B * a.nq, group, kBM / group) ||
      !make_bf16_map(&mk, a.K, kv_rows, D, D, kBN) || !make_bf16_map(&mv, a.V, kv_rows, D, D, kBN))
    return cudaErrorNotSupported;
  WideParams p;
  p.kv_len = a.kv_len;
  p.parent = a.parent;
  p.out = a.out;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.ranges = reinterpret_cast<int2*>(ws + WsLayout::ranges_off(a.B, a.H));
  p.partials = reinterpret_cast<float*>(ws + WsLayout::partials_off(a.B, a.H));
  p.B = a.B; p.H = a.H; p.Hkv = a.Hkv; p.group = group; p.S_cap = a.S_cap;
  p.max_kv_len = a.max_kv_len; p.n = a.nq;
  p.rows = a.nq * group;
  p.R = (p.rows + kBM - 1) / kBM;
  p.tree = a.tree;
  p.nk = nk;
  p.nv = nv;
  p.scale_log2 = a.scale * kLog2e;
  // G shares of the key tiles, R CTAs (row tiles) per share
  const long long tiles_ub = (long long)a.B * a.Hkv * ((a.max_kv_len + (a.tree ? a.nq : 0) + kBN - 1) / kBN);
  long long G = a.max_ctas > 0 ? a.max_ctas : sm_count() / p.R;
  if (G > kMaxCtas) G = kMaxCtas;
  if (G > tiles_ub) G = tiles_ub;
  if (G < 1) G = 1;
  cudaError_t e = launch_pdl(tree_attn_wide_kernel<D>, dim3((unsigned)(G * p.R)), dim3(kThreads),
                             C::smem_bytes(a.B, nk, nv), st, mq, mk, mv, p);
  if (e != cudaSuccess) return e;
  return launch_tree_merge<D>(p.ranges, p.partials, p.out, a.B * a.Hkv, p.rows, group, a.H, a.Hkv, st);
}

}  // namespace

cudaError_t launch_tree_attn_wide(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype != 0 || (a.D != 128 && a.D != 64) || a.Hkv < 1) return cudaErrorNotSupported;
  const int group = a.H / a.Hkv;
  // Grouped-query slabs, and any slab of more than 64 rows; multi-head slabs
  // of up to 64 rows stream faster through the 64-row kernel's deeper rings.
  if ((group == 1 && a.nq <= 64) || a.nq * group > kMaxRows || kBM % group != 0) return cudaErrorNotSupported;
  // 32-bit TMA coordinates, including a tile's reach past the last row
  if ((long long)a.B * a.Hkv * a.S_cap + kBN > 0x7fffffffLL || (long long)a.B * a.nq + kBM > 0x7fffffffLL)
    return cudaErrorNotSupported;
  if (a.D == 128) return launch_typed<128>(a, st);
  return launch_typed<64>(a, st);
}

}  // namespace glide
