// Tree verification attention on the tcgen05 tensor cores (Section 3.2:
// the CaPE verification mask, here as the general ancestor-or-self mask of a
// linearized token tree).  bf16 Q/K/V, fp32 accumulation, D in {64, 128},
// n <= 64 tree queries per (sequence, head).
//
// At n = 26..64 queries the verification does n flops per KV byte, beyond
// what CUDA-core FMA can sustain at HBM speed, so both products run on the
// tensor cores while the KV stream stays the bound:
//   S = Q K^T   : M = 64 (query rows, zero-padded), N = 64 keys, K = D
//   O += P V    : M = 64, N = D, K = 32 keys, once per key half
// Operands sit in shared memory in the 128-byte-swizzled K-major layout
// (Q, K, P) or M/N-major layout (V); accumulators live in tensor memory
// (TMEM): four S buffers of 64 columns and one O accumulator of D columns for
// each key half.
//
// Grouped-query slabs (a sequence's cached head and the n x H/H_kv query rows
// it serves) with more than 64 rows are served in row tiles of 64: the grid
// holds R CTAs per share of the key sequence, CTA x * R + y taking row tile y
// of every slab in share x.  The R CTAs of a share are adjacent, so they run
// together and stream the same K/V tiles at about the same time: DRAM serves
// each tile about once and L2 the other R - 1 reads.
//
// Roles (416 threads, persistent grid of one CTA per SM, split-KV partition
// shared with the other attention kernels):
//   warps 0-7  softmax.  An M = 64 accumulator keeps rows 16q..16q+15 in
//              TMEM lanes 32q..32q+15; warp w reads lane quarter q = w % 4
//              with the 16x64b shape (two threads per row, even and odd
//              columns) and key half w / 4 (32 of the tile's 64 keys).  Each
//              (row, key half) keeps its own running max and sum and its own
//              O accumulator, so no values cross warps inside the key loop;
//              the halves are merged once per segment.  Query i sits in row
//              (i % 4) * 16 + i / 4, which spreads any tree over all four lane
//              quarters (all four SM sub-partitions).
//   warps 8, 12 producers: lane 0 of warp 8 feeds the K ring, lane 0 of
//              warp 12 the V ring, with 2-D TMA (64 keys x 64 head dims per
//              box, 128-byte swizzle); K slots free up after S, V slots only
//              after P.V, so each ring has its own thread.
//   warps 9-11 MMA issue.  A tcgen05.mma keeps its issuing thread busy for
//              ~150 cycles whatever its shape, so one thread cannot feed a
//              64-key tile (8 S + 4 P.V instructions) at HBM speed: warp 9
//              issues S for even tiles, warp 10 S for odd tiles, warp 11 all
//              P.V products.  Warp 9 also owns the TMEM allocation.
//
// Online softmax in the log2 domain with a lazy reference max: the max used
// for the exponent only moves when a tile's max exceeds it by more than 8
// (factor 256), so O is rescaled in TMEM rarely; the final division by the
// sum taken with the same reference makes the result exact up to rounding.
// V rows past the end of a slab are zeroed in shared memory before P.V (the
// cache beyond kv_len + n may hold anything, even NaN).
//
// A slab whose keys fall in one CTA's share is written out directly.  A slab
// split over several shares leaves one partial (max, sum, o) per share in the
// workspace, and the kernel records the slab's share range; a second kernel,
// tree_merge_kernel, launched as a programmatic dependent, merges them with
// one warp per query row.  No CTA counts arrivals or merges at its end, so
// the segment epilogues carry no fence or atomic and the merges run spread
// over the whole GPU instead of on the last CTAs.
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

constexpr int kTK = 64;          // keys per tile
constexpr int kHK = 32;          // keys per key half
constexpr int kM = 64;           // MMA rows (tree queries, zero-padded)
constexpr int kMaxStages = 8;    // K/V stages (the launch picks as many as fit)
constexpr int kSBuf = 4;         // S buffers in TMEM (two per S issuer)
constexpr int kSoftWarps = 8;
constexpr int kProdWarp = 8;     // the K ring's producer
constexpr int kMmaWarp = 9;      // warps 9, 10: S issuers; warp 11: P.V issuer
constexpr int kVProdWarp = 12;   // the V ring's producer
constexpr int kThreads = 416;
constexpr float kRescaleLog2 = 8.0f;
// What a switch from one slab to the next costs a CTA, in 64-key tiles: per
// CTA, the end times of a static split grow by ~2.7 us per extra segment at 4
// query rows, ~5 us at 24 and ~5.5 us at 64 (the epilogue of one slab, with
// its output or partial rows, and the pipeline start of the next) at ~0.7 us
// per tile, so shares are balanced on tiles + w * (segments - 1) with
// w = 4 + rows / 16.
__host__ __device__ constexpr int seg_weight(int rows) { return 4 + rows / 16; }

// barrier slots
// ODONE has four slots (tile mod 4): the softmax waits on it only now and
// then, and four slots keep every such wait within one phase of the barrier.
// QFULL has two slots (segment parity): an S issuer waits only for segments
// in which it has a tile, and each issuer has a tile in every two consecutive
// segments, so no slot runs two phases ahead of a waiter.
constexpr int B_KFULL = 0, B_VFULL = 8, B_KEMPTY = 16, B_VEMPTY = 24, B_SFULL = 32, B_SFREE = 36, B_PFULL = 40,
              B_PFREE = 42, B_ODONE = 44, B_OFREE = 48, B_QFULL = 49, B_MDONE = 51, kNumBars = 54;

template <int D>
struct TcCfg {
  static constexpr int kHalves = D / 64;              // 128-byte swizzle atoms across the head dim
  static constexpr uint32_t kQHalf = kM * 128;        // 64 rows x 128 B
  static constexpr uint32_t kQBytes = kHalves * kQHalf;
  static constexpr uint32_t kPBytes = kM * kTK * 2;   // 64 rows x 64 keys bf16
  static constexpr uint32_t kKVHalf = kTK * 128;      // 64 keys x 128 B
  static constexpr uint32_t kKVTile = kHalves * kKVHalf;
  static constexpr uint32_t off_Q = 0;
  static constexpr uint32_t off_P = off_Q + kQBytes;
  static constexpr uint32_t off_K = off_P + 2 * kPBytes;
  // then ns K stages, ns V stages, barriers, (max, sum) of both key halves, misc, batch table
  static __host__ __device__ uint32_t off_V(int ns) { return off_K + ns * kKVTile; }
  static __host__ __device__ uint32_t off_bar(int ns) { return off_V(ns) + ns * kKVTile; }
  static __host__ __device__ uint32_t off_ml(int ns) { return off_bar(ns) + 512; }
  static __host__ __device__ uint32_t off_misc(int ns) { return off_ml(ns) + 2 * kM * 8; }
  static __host__ __device__ uint32_t off_tab(int ns) { return off_misc(ns) + 48; }
  static constexpr uint32_t kTmemO = kSBuf * kTK;                  // S buffers at columns 0, 64, 128, 192
  static constexpr uint32_t kTmemCols = kTmemO + 2 * D <= 256 ? 256 : 512;
  static_assert(kTmemO + 2 * D <= 512, "TMEM columns");
  static_assert(kNumBars * 8 <= 512, "barrier area");
  static size_t smem_bytes(int B, int ns) { return 1024 + off_tab(ns) + (size_t)(B + 1) * 8 + (size_t)(4 * B + 1) * 4; }
};

struct TcParams {
  const __nv_bfloat16* q;
  const int* kv_len;
  const int* parent;
  float* out;
  unsigned* status;
  int2* ranges;      // per slab: the share range of a split slab, (-1, -1) otherwise
  float* partials;
  int B, H, S_cap, max_kv_len, n;
  int Hkv;    // cached heads (slabs are (b, cached head))
  int group;  // query heads per cached head (H / Hkv)
  int rows;   // query rows per slab: n nodes x group heads, node-major, <= kMaxRows
  int R;      // row tiles per slab (rows / 64 rounded up)
  int tree;   // 1: the n tree keys follow the prefix (verification); 0: prefix only
  int ns;  // K/V stages
  float scale_log2;
};

// Named barrier among the 256 softmax threads (id 2; id 1 belongs to the split merge).
__device__ __forceinline__ void softmax_sync() { asm volatile("bar.sync 2, 256;" ::: "memory"); }
// Barrier 3: every softmax thread has read the other half's (max, sum) of the
// segment, so both exchange slots may be written again.
__device__ __forceinline__ void ml_sync() { asm volatile("bar.sync 3, 256;" ::: "memory"); }

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                        const TcParams p) {
  using C = TcCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int ns = p.ns;
  const uint32_t off_V = C::off_V(ns);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::off_bar(ns));
  float2* ml = reinterpret_cast<float2*>(base + C::off_ml(ns));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + C::off_misc(ns));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::off_misc(ns) + 4);
  BatchTiles bt;
  bt.start = reinterpret_cast<long long*>(base + C::off_tab(ns));
  bt.len = reinterpret_cast<int*>(bt.start + p.B + 1);
  bt.ntiles = bt.len + p.B;
  bt.plen = bt.ntiles + p.B;
  bt.sidx = bt.plen + p.B;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = p.n;
  // Shared-memory set-up and the tensor-map fetches (kernel parameters) come
  // before the wait for the previous kernel; every global access and the TMEM
  // allocation come after it.
  if (threadIdx.x == 0) {
    tc::prefetch_tmap(&tmK);
    tc::prefetch_tmap(&tmV);
    for (int b = 0; b < kNumBars; ++b) {
      uint32_t cnt = 1;
      if ((b >= B_SFREE && b < B_SFREE + kSBuf) || b == B_PFULL || b == B_PFULL + 1) cnt = kSoftWarps;
      if (b == B_OFREE) cnt = kSoftWarps;                  // both halves read O
      if (b == B_QFULL || b == B_QFULL + 1) cnt = 4;       // the key-half-0 warps write Q
      mbar_init(&bars[b], cnt);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  pdl_wait();
  if (warp == kMmaWarp) {
    tc::tmem_alloc(tmem_slot, C::kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  build_batch_tiles(bt, p.kv_len, p.B, p.Hkv, p.max_kv_len, p.tree ? n : 0, kTK);  // __syncthreads inside
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  // this CTA: share x of the key sequence, row tile y of every slab in it
  const int x = blockIdx.x / p.R, y = blockIdx.x - x * p.R;
  const int row0 = y * kM, rows_here = min(kM, p.rows - row0);
  CostPartition P;  // shares of equal cost, a segment switch counted as seg_weight tiles
  P.init(bt, p.B, p.Hkv, gridDim.x / p.R, seg_weight(p.rows < kM ? p.rows : kM));
  const long long g_begin = P.begin(x), g_end = P.end(x);

  if (warp == kProdWarp || warp == kVProdWarp) {
    // ----------------------------------------------------------- producers
    // Warp 8 feeds the K ring and warp 12 the V ring, one thread each: a
    // 2-D tensor copy keeps its issuing thread busy for hundreds of cycles,
    // and one thread issuing both rings' copies (four per 64-key tile) set
    // the pace of the whole kernel at ~1430 cycles per tile (per-tile trace:
    // each copy left 1.3-1.9 tile periods after its slot was free).
    if (lane == 0) {
      const bool is_k = warp == kProdWarp;
      const CUtensorMap* map = is_k ? &tmK : &tmV;
      tc::prefetch_tmap(map);
      uint64_t* full = &bars[is_k ? B_KFULL : B_VFULL];
      uint64_t* empty = &bars[is_k ? B_KEMPTY : B_VEMPTY];
      const uint32_t dst0 = is_k ? C::off_K : off_V;
      // one reader per tile: evict it first; R row tiles read each tile R times
      const uint64_t pol = p.R == 1 ? policy_evict_first() : policy_evict_normal();
      int i = 0;
      bool ok = true;
      for (long long g = g_begin; g < g_end && ok;) {
        const Segment sg = locate(bt, P, p.B, g, g_end);
        const int row0k = (sg.b * p.Hkv + sg.h) * p.S_cap;
        for (int t = sg.t0; t < sg.t1; ++t, ++i) {
          const int st = i % ns;
          if (!mbar_wait(&empty[st], ((i / ns) & 1) ^ 1, abort_flag, p.status)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[st], C::kKVTile);
          for (int hd = 0; hd < C::kHalves; ++hd)
            tc::tma_load_2d(base + dst0 + st * C::kKVTile + hd * C::kKVHalf, map, hd * 64, row0k + t * kTK, &full[st],
                            pol);
        }
        g = sg.g_end;
      }
      if (!ok)  // aborted: let issued loads land before the CTA exits
        for (int j = (i > ns ? i - ns : 0); j < i; ++j) mbar_drain(&full[j % ns], (j / ns) & 1);
    }
  } else if (warp >= kMmaWarp) {  // warps 9-11
    // ----------------------------------------------------------- MMA issue
    const int role = warp - kMmaWarp;  // 0, 1: S of tiles with j % 2 == role; 2: P.V
    if (lane == 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(kM, kTK, false, false);
      constexpr uint32_t idO = tc::idesc_bf16_f32(kM, D, false, true);
      const uint32_t sQ = smem_u32(base + C::off_Q), sP = smem_u32(base + C::off_P);
      const uint32_t sK = smem_u32(base + C::off_K), sV = smem_u32(base + off_V);
      int i = 0, seg = 0;
      bool ok = true;
      // S(j) = Q K(j)^T into S buffer j % kSBuf
      auto issue_s = [&](int j) -> bool {
        if (!mbar_wait(&bars[B_KFULL + j % ns], (j / ns) & 1, abort_flag, p.status) ||
            !mbar_wait(&bars[B_SFREE + j % kSBuf], ((j / kSBuf) & 1) ^ 1, abort_flag, p.status))
          return false;
        tc::fence_after_sync();
        const uint32_t kb = sK + (j % ns) * C::kKVTile;
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint64_t a = tc::sw128_desc(sQ + (ks / 4) * C::kQHalf + (ks % 4) * 32, 16, 1024);
          const uint64_t bdesc = tc::sw128_desc(kb + (ks / 4) * C::kKVHalf + (ks % 4) * 32, 16, 1024);
          tc::mma_bf16(tmem + (j % kSBuf) * kTK, a, bdesc, idS, ks > 0 ? 1u : 0u);
        }
        tc::mma_commit(&bars[B_SFULL + j % kSBuf]);
        tc::mma_commit(&bars[B_KEMPTY + j % ns]);
        return true;
      };
      // O_h += P[:, 32h .. 32h+31] V[32h .. 32h+31, :] for key halves h = 0, 1
      auto issue_pv = [&](int jj, bool first_in_seg) -> bool {
        if (!mbar_wait(&bars[B_PFULL + (jj & 1)], (jj >> 1) & 1, abort_flag, p.status)) return false;
        if (!mbar_wait(&bars[B_VFULL + jj % ns], (jj / ns) & 1, abort_flag, p.status)) return false;
        if (first_in_seg && seg > 0 && !mbar_wait(&bars[B_OFREE], (seg - 1) & 1, abort_flag, p.status)) return false;
        tc::fence_after_sync();
        const uint32_t vb = sV + (jj % ns) * C::kKVTile;
        const uint32_t pb = sP + (jj & 1) * C::kPBytes;
#pragma unroll
        for (int ks = 0; ks < kTK / 16; ++ks) {
          const int h = ks >> 1;
          const uint64_t a = tc::sw128_desc(pb + ks * 32, 16, 1024);
          const uint64_t bdesc = tc::sw128_desc(vb + ks * 16 * 128, C::kKVHalf, 1024);
          tc::mma_bf16(tmem + C::kTmemO + h * D, a, bdesc, idO, (first_in_seg && (ks & 1) == 0) ? 0u : 1u);
        }
        tc::mma_commit(&bars[B_PFREE + (jj & 1)]);
        tc::mma_commit(&bars[B_VEMPTY + jj % ns]);
        tc::mma_commit(&bars[B_ODONE + (jj & 3)]);
        return true;
      };
      for (long long g = g_begin; g < g_end && ok;) {
        const Segment s = locate(bt, P, p.B, g, g_end);
        if (role < 2) {
          // S of the tiles j with j % 2 == role; Q of the segment must be in place first
          const int ntile = s.t1 - s.t0;
          const bool mine = ntile > 1 || (i & 1) == role;
          if (mine && !mbar_wait(&bars[B_QFULL + (seg & 1)], (seg >> 1) & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          for (int t = s.t0; t < s.t1 && ok; ++t, ++i)
            if ((i & 1) == role) ok = issue_s(i);
        } else {
          for (int t = s.t0; t < s.t1 && ok; ++t, ++i) ok = issue_pv(i, t == s.t0);
        }
        ++seg;
        g = s.g_end;
      }
      tc::mma_commit(&bars[B_MDONE + role]);  // every MMA finished before TMEM is released
      mbar_drain(&bars[B_MDONE + role], 0);
    }
  } else {
    // ------------------------------------------------------------- softmax
    // Warp w reads lane quarter q = w % 4 (MMA rows 16q..16q+15) and key half
    // w / 4 with the 16x64b TMEM shape: lane pair (t, t^2) shares one row,
    // thread t takes the row's even or odd columns (cpar), 16 of the 32 keys.
    const int quarter = warp & 3, half = warp >> 2;
    const int rr = (lane >> 2) + 8 * (lane & 1);  // row within the quarter
    const int cpar = (lane >> 1) & 1;             // column parity of this thread
    const int row = quarter * 16 + rr;            // MMA row
    const int qi = rr * 4 + quarter;              // the query row of this MMA row, within the row tile
    const bool valid = qi < rows_here;
    const int node = valid ? (row0 + qi) / p.group : 0;  // its tree node
    const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
    const uint32_t o_col = C::kTmemO + half * D;
    const int sid = threadIdx.x;                  // 0..255 among the softmax threads
    const float sl2 = p.scale_log2;
    bool dead = false;
    int i = 0, seg = 0;
    // Segment sg's queries into the swizzled Q tile (padding rows are zero);
    // the two threads of a row write chunks 0-3 and 4-7 of each 128-byte atom.
    // Key-half-0 warps only.
    const OutMap om{p.group, p.H};
    // this thread's query row of slab (sb, h): its row in q / out (-1: none),
    // and the prefix keys it sees (< lim)
    auto row_at = [&](const Segment& sq, int& lim) -> long long {
      lim = bt.plen[sq.b];
      if (!valid) return -1;
      return om.row(sq.b, sq.h, row0 + qi, p.rows);
    };
    auto write_q = [&](const Segment& sq, int sg) {
      unsigned char* qrow = base + C::off_Q + (row >> 3) * 1024 + (row & 7) * 128;
      int lim_unused;
      const long long qr = row_at(sq, lim_unused);
      const uint4* src = reinterpret_cast<const uint4*>(p.q + (qr >= 0 ? qr : 0) * D);
#pragma unroll
      for (int hd = 0; hd < C::kHalves; ++hd)
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          const int c = cpar * 4 + cc;
          uint4 v = make_uint4(0u, 0u, 0u, 0u);
          if (qr >= 0) v = src[hd * 8 + c];
          *reinterpret_cast<uint4*>(qrow + hd * C::kQHalf + ((c ^ (row & 7)) << 4)) = v;
        }
      tc::fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_QFULL + (sg & 1)]);
    };
    // The first segment's queries first: the first S products wait for them.
    if (half == 0 && g_begin < g_end) write_q(locate(bt, P, p.B, g_begin, g_end), 0);
    // Then, off the path to the first S products: the share range of every
    // slab split over several shares, for the merge kernel ((-1, -1): written
    // out directly, or no keys), and zeros for a prefix-only call's sequences
    // without cached keys (an empty softmax).
    constexpr int kST = kSoftWarps * 32;
    if (y == 0)
      for (int bh = x * kST + (int)threadIdx.x; bh < p.B * p.Hkv; bh += (gridDim.x / p.R) * kST) {
        const int b = bh / p.Hkv, nt = bt.ntiles[b];
        int2 r = make_int2(-1, -1);
        if (nt > 0) {
          const long long first = bt.start[b] + (long long)(bh - b * p.Hkv) * nt;
          const int cf = P.cta_of(first), cl = P.cta_of(first + nt - 1);
          if (cf != cl) r = make_int2(cf, cl);
        }
        p.ranges[bh] = r;
      }
    if (!p.tree) {
      const long long total = (long long)p.B * n * p.H * D;
      for (long long idx = (long long)blockIdx.x * kST + threadIdx.x; idx < total; idx += (long long)gridDim.x * kST)
        if (bt.ntiles[idx / ((long long)n * p.H * D)] == 0) p.out[idx] = 0.f;
    }
    for (long long g = g_begin; g < g_end; ++seg) {
      const Segment s = locate(bt, P, p.B, g, g_end);
      const int plen = bt.plen[s.b], len = bt.len[s.b];
      int rowlim;  // keys below it are visible to this row (the prefix)
      const long long orow = row_at(s, rowlim);

      // the ancestor-or-self set of this row's tree node, found when the first
      // tile with tree keys comes (prefix only: no tree keys)
      uint64_t anc = 0;
      bool anc_ready = !p.tree;

      float m_used = -CUDART_INF_F, l = 0.f;  // l: this thread's share of the row sum
      // S of the next tile is loaded while this tile's exponentials run (within
      // the segment only: the next segment's S needs a Q written after it ends)
      uint32_t sr[16];
      if (!dead) dead = !warp_wait(&bars[B_SFULL + i % kSBuf], (i / kSBuf) & 1, abort_flag, p.status);
      if (!dead) {
        tc::fence_after_sync();
        tc::tmem_ld16x64b_x16(lane_addr + (i % kSBuf) * kTK + half * kHK, sr);
      }
      for (int t = s.t0; t < s.t1; ++t, ++i) {
        const int j = i;
        tc::tmem_wait_ld();
        uint32_t cur[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          asm volatile("" : "+r"(sr[k]));  // sr is only valid after the wait: keep reads below it
          cur[k] = sr[k];
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_SFREE + j % kSBuf]);

        // scores of keys key0 + 2k + cpar, k = 0..15, in the log2 domain, masked
        const int key0 = t * kTK + half * kHK + cpar;
        float sc[16];
        if (t * kTK + half * kHK + kHK <= plen) {
#pragma unroll
          for (int k = 0; k < 16; ++k) sc[k] = __uint_as_float(cur[k]) * sl2;
        } else {
          if (!anc_ready) {  // warp-uniform: t, half and plen are the same in every lane
            anc = ancestors(p.parent + (size_t)s.b * n, n, node, valid, lane);
            anc_ready = true;
          }
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const int key = key0 + 2 * k;
            const bool vis = key < rowlim || (key < len && ((anc >> ((key - plen) & 63)) & 1ull));
            sc[k] = vis ? __uint_as_float(cur[k]) * sl2 : -CUDART_INF_F;
          }
        }
        if (t + 1 < s.t1) {  // start loading S of the next tile
          const int jn = j + 1;
          if (!dead) dead = !warp_wait(&bars[B_SFULL + jn % kSBuf], (jn / kSBuf) & 1, abort_flag, p.status);
          if (!dead) {
            tc::fence_after_sync();
            tc::tmem_ld16x64b_x16(lane_addr + (jn % kSBuf) * kTK + half * kHK, sr);
          }
        }
        float mx[4] = {sc[0], sc[1], sc[2], sc[3]};
#pragma unroll
        for (int k = 4; k < 16; ++k) mx[k & 3] = fmaxf(mx[k & 3], sc[k]);
        float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 2));  // the row's max over both threads

        const bool need = tmax > m_used + kRescaleLog2;
        if (__any_sync(0xffffffffu, need)) {
          const float m_new = need ? tmax : m_used;
          const float f = need ? fast_exp2(m_used - m_new) : 1.f;
          l *= f;
          if (t > s.t0 && !dead) {  // O holds the P.V of earlier tiles of this segment
            dead = !warp_wait(&bars[B_ODONE + ((j - 1) & 3)], ((j - 1) >> 2) & 1, abort_flag, p.status);
            if (!dead) {
              tc::fence_after_sync();
#pragma unroll 1
              for (int c = 0; c < D / 32; ++c) {
                uint32_t o[16];
                tc::tmem_ld16x64b_x16(lane_addr + o_col + c * 32, o);
                tc::tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 16; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * f);
                tc::tmem_st16x64b_x16(lane_addr + o_col + c * 32, o);
              }
              tc::tmem_wait_st();
            }
          }
          m_used = m_new;
        }
        const float m_eff = m_used == -CUDART_INF_F ? 0.f : m_used;
        float pv[16];
        float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          pv[k] = fast_exp2(sc[k] - m_eff);
          ls[k & 3] += pv[k];
        }
        l += (ls[0] + ls[1]) + (ls[2] + ls[3]);
        // bf16 pairs of consecutive keys: the even-column thread keeps keys 0..15
        // of the half, the odd-column thread keys 16..31; swap the other halves
        uint32_t pk[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float send = cpar ? pv[k] : pv[8 + k];
          const float recv = __shfl_xor_sync(0xffffffffu, send, 2);
          pk[k] = cpar ? pack_bf16x2(recv, pv[8 + k]) : pack_bf16x2(pv[k], recv);
        }

        if (!dead) dead = !warp_wait(&bars[B_PFREE + (j & 1)], ((j >> 1) & 1) ^ 1, abort_flag, p.status);
        {
          unsigned char* prow = base + C::off_P + (j & 1) * C::kPBytes + (row >> 3) * 1024 + (row & 7) * 128;
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const int chunk = half * 4 + cpar * 2 + c;  // 8 keys per 16-byte chunk
            *reinterpret_cast<uint4*>(prow + ((chunk ^ (row & 7)) << 4)) =
                make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
          }
        }
        const int vrows = len - t * kTK;
        if (vrows < kTK) {  // last tile of the slab: clear V rows past its end
          const int st = j % ns;
          if (!dead) dead = !warp_wait(&bars[B_VFULL + st], (j / ns) & 1, abort_flag, p.status);
          for (int idx = sid; idx < (kTK - vrows) * C::kHalves; idx += kSoftWarps * 32) {
            const int r = vrows + idx / C::kHalves, hd = idx % C::kHalves;
            uint4* dst = reinterpret_cast<uint4*>(base + off_V + st * C::kKVTile + hd * C::kKVHalf + r * 128);
#pragma unroll
            for (int c = 0; c < 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
          }
        }
        tc::fence_async_smem();
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_PFULL + (j & 1)]);
      }

      // Every S product of this segment has been consumed, so Q is free: write
      // the next segment's queries now and let its S products overlap this
      // epilogue.
      if (half == 0 && s.g_end < g_end) write_q(locate(bt, P, p.B, s.g_end, g_end), seg + 1);

      // ---- segment epilogue: merge the two key halves, then O / l or a split
      // partial.  Each half writes half of the head dims, reading both halves'
      // accumulators there.
      l += __shfl_xor_sync(0xffffffffu, l, 2);  // the row's sum over both threads
      if (cpar == 0) ml[half * kM + row] = make_float2(m_used, l);
      softmax_sync();
      const float2 other = ml[(half ^ 1) * kM + row];
      // every (max, sum) is read before any half can reach the next segment's
      // epilogue and overwrite its slot (the next segment's Q is written ahead,
      // so a half can get there early)
      ml_sync();
      {
        const int jl = i - 1;
        if (!dead) dead = !warp_wait(&bars[B_ODONE + (jl & 3)], (jl >> 2) & 1, abort_flag, p.status);
        const float m0 = half == 0 ? m_used : other.x, l0 = half == 0 ? l : other.y;
        const float m1 = half == 0 ? other.x : m_used, l1 = half == 0 ? other.y : l;
        const float M = fmaxf(m0, m1);
        const float f0 = m0 == -CUDART_INF_F ? 0.f : fast_exp2(m0 - M);
        const float f1 = m1 == -CUDART_INF_F ? 0.f : fast_exp2(m1 - M);
        const float L = l0 * f0 + l1 * f1;
        const bool single = s.c_first == s.c_last;
        const int bh = s.b * p.Hkv + s.h;
        float* dst = single ? p.out + (orow >= 0 ? orow : 0) * D
                            : partial_slot(p.partials, x + bh, p.rows, D) + (size_t)(row0 + (valid ? qi : 0)) * (D + 2) + 2;
        const bool write = single ? orow >= 0 : valid;
        if (!dead) {
          tc::fence_after_sync();
          const float invL = L > 0.f ? 1.f / L : 0.f;  // a padding row has no key: zeros
          const float g0 = single ? f0 * invL : f0;
          const float g1 = single ? f1 * invL : f1;
          constexpr int kChunks = D / 64;  // 32-column chunks per half
          uint32_t a[kChunks][16], b[kChunks][16];
#pragma unroll
          for (int cc = 0; cc < kChunks; ++cc) {
            const int c = half * kChunks + cc;
            tc::tmem_ld16x64b_x16(lane_addr + C::kTmemO + c * 32, a[cc]);
            tc::tmem_ld16x64b_x16(lane_addr + C::kTmemO + D + c * 32, b[cc]);
          }
          tc::tmem_wait_ld();
#pragma unroll
          for (int cc = 0; cc < kChunks; ++cc) {
            const int c = half * kChunks + cc;
            float v[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) v[k] = __uint_as_float(a[cc][k]) * g0 + __uint_as_float(b[cc][k]) * g1;
            // The row's two threads hold its even (cpar 0) and odd (cpar 1)
            // columns; one exchange of two values per 8 columns gives each
            // thread 4 consecutive columns: cpar 0 columns 8j..8j+3, cpar 1
            // columns 8j+4..8j+7.
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float r0 = __shfl_xor_sync(0xffffffffu, cpar ? v[4 * j] : v[4 * j + 2], 2);
              const float r1 = __shfl_xor_sync(0xffffffffu, cpar ? v[4 * j + 1] : v[4 * j + 3], 2);
              const float4 q4 = cpar ? make_float4(r0, v[4 * j + 2], r1, v[4 * j + 3])
                                     : make_float4(v[4 * j], r0, v[4 * j + 1], r1);
              float* d4 = dst + c * 32 + 8 * j + 4 * cpar;
              if (write) {
                if (single) {
                  *reinterpret_cast<float4*>(d4) = q4;
                } else {  // a partial row starts 8 bytes into a 16-byte boundary
                  reinterpret_cast<float2*>(d4)[0] = make_float2(q4.x, q4.y);
                  reinterpret_cast<float2*>(d4)[1] = make_float2(q4.z, q4.w);
                }
              }
            }
          }
          if (!single && valid && cpar == 0 && half == 0) {
            dst[-2] = M;
            dst[-1] = L;
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_OFREE]);
      }
      g = s.g_end;
    }
  }

  __syncwarp();  // the producer and MMA warps reconverge after their single-lane loops
  tc::fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------- host
template <int D>
cudaError_t launch_typed(const AttnArgs& a, cudaStream_t st) {
  using C = TcCfg<D>;
  static bool configured = false;
  const int limit = smem_optin_bytes();
  if (!configured) {
    cudaError_t e =
        cudaFuncSetAttribute(tree_attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  // As many K/V stages as the shared memory holds, and an even number: K slot
  // j % ns then only ever carries tiles of one parity, i.e. of one S issuer.
  const int group = a.H / a.Hkv;
  int ns = kMaxStages;
  while (ns > 2 && C::smem_bytes(a.B, ns) > (size_t)limit) ns -= 2;
  if (C::smem_bytes(a.B, ns) > (size_t)limit) return cudaErrorNotSupported;
  const long long rows = (long long)a.B * a.Hkv * a.S_cap;
  CUtensorMap mk, mv;
  if (!make_bf16_map(&mk, a.K, rows, D, D, kTK) || !make_bf16_map(&mv, a.V, rows, D, D, kTK)) return cudaErrorNotSupported;
  const long long tiles_ub = (long long)a.B * a.Hkv * ((a.max_kv_len + (a.tree ? a.nq : 0) + kTK - 1) / kTK);
  const int R = (a.nq * group + kM - 1) / kM;
  // G shares of the key sequence, R CTAs (row tiles) per share
  long long G = a.max_ctas > 0 ? a.max_ctas : sm_count() / R;
  if (G > kMaxCtas) G = kMaxCtas;
  if (G > tiles_ub) G = tiles_ub;
  if (G < 1) G = 1;
  TcParams p;
  p.q = static_cast<const __nv_bfloat16*>(a.q);
  p.kv_len = a.kv_len;
  p.parent = a.parent;
  p.out = a.out;
  unsigned char* ws = static_cast<unsigned char*>(a.ws);
  p.status = reinterpret_cast<unsigned*>(ws);
  p.ranges = reinterpret_cast<int2*>(ws + WsLayout::ranges_off(a.B, a.H));
  p.partials = reinterpret_cast<float*>(ws + WsLayout::partials_off(a.B, a.H));
  p.B = a.B; p.H = a.H; p.S_cap = a.S_cap; p.max_kv_len = a.max_kv_len; p.n = a.nq;
  p.Hkv = a.Hkv; p.group = group; p.rows = p.n * group; p.R = R; p.tree = a.tree;
  p.ns = ns;
  p.scale_log2 = a.scale * kLog2e;
  cudaError_t e = launch_pdl(tree_attn_tc_kernel<D>, dim3((unsigned)(G * R)), dim3(kThreads), C::smem_bytes(a.B, ns),
                             st, mk, mv, p);
  if (e != cudaSuccess) return e;
  return launch_tree_merge<D>(p.ranges, p.partials, p.out, a.B * a.Hkv, p.rows, group, a.H, a.Hkv, st);
}

}  // namespace

cudaError_t launch_tree_attn_tc(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype != 0 || (a.D != 128 && a.D != 64)) return cudaErrorNotSupported;
  if ((long long)a.B * a.Hkv * a.S_cap > 0x7fffffffLL) return cudaErrorNotSupported;  // 32-bit TMA row coordinate
  if (a.nq * (a.H / a.Hkv) > kMaxRows) return cudaErrorNotSupported;  // the abi rejects this first
  if (a.D == 128) return launch_typed<128>(a, st);
  return launch_typed<64>(a, st);
}

}  // namespace glide
