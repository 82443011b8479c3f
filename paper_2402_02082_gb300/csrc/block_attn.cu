// The draft's cross-attention at training time under the block-wise mask
// (Section 3.1, "Block-wise Attention Mask") on the tcgen05 tensor cores.
//
// Position j of a training sequence attends to the target's keys and values
// of the positions k < L * (j / L), the blocks before its own.  Over T
// positions that is a lower-triangular attention of about T^2 / 2 (query,
// key) pairs at 4 D flops each: a compute-bound product, unlike the
// memory-bound decoding kernels.  Both products run on the tensor cores:
//   S = Q K^T   : M = 128 positions, N = 128 keys, K = D, operands in shared memory
//   O += P V    : M = 128, N = D, K = 64 keys per key half, P in tensor memory, V in shared memory
// Q and K sit in shared memory in the 128-byte-swizzled K-major layout, V in
// the M/N-major layout.  Tensor memory (TMEM, 512 columns) holds three S
// buffers of 128 columns and the O accumulator (D columns).  Two softmax
// groups take the two 64-key halves of every tile, so every SM sub-partition
// runs two softmax warps and one warp's loads, maxima and stores overlap the
// other's exponentials (the softmax is latency-bound: at 32 exponentials per
// clock per SM the MUFU unit is busy about a third of a tile).  The partners
// of a lane quarter agree on each tile's row max through one TMEM column of
// their halves, so both halves share one reference max and accumulate into
// the one O; each group rescales, and at the end writes, its half of O's
// columns.  A group overwrites the first 32 columns of its half of the S
// buffer with P as bf16 pairs and the P.V product reads P from there: P never
// passes through shared memory, whose bandwidth the MMA operand reads and the
// TMA writes already share.  S of tile i + 3 reuses the buffer of tile i, so
// it waits for the completion of P.V of tile i; three buffers keep that wait
// off the softmax's path.
//
// The K and V rings have separate depths, the keys' deeper (S runs up to
// three tiles ahead of P.V): 3 and 2 stages of 32 KB for D = 128, what the
// shared memory holds next to Q and the epilogue staging.  The epilogue stages
// O / l in 4 KB boxes of shared memory (the 128-byte swizzle) and writes them
// with bulk tensor stores, which drain while the warps go on.
//
// Work item: (sequence b, query head h, tile of 128 positions).  Tile x of a
// (b, h) sees about x + 1 key tiles, so tile x is paired with tile
// T/128 - 1 - x and every pair carries the same number of key tiles.  CTA c
// runs pairs c, c + G, c + 2G, ... in (b, h)-major order: the CTAs that run at
// the same time read the keys and values of a few heads, which stay in L2.
//
// Roles (512 threads, one CTA per SM; setmaxnreg gives the softmax warps 168
// registers a thread and the others 88):
//   warps 0-7   softmax, two groups of four: warp w reads TMEM lane quarter
//               w % 4 (one thread per position) and key half w / 4 of every
//               tile, with packed f32x2 arithmetic; at the end of an item it
//               hands its row sums to the epilogue warps.
//   warp 8      producer: lane 0 loads the Q tile and feeds the K and V rings
//               with 2-D TMA, polling the free slots of both.
//   warp 9      S issue (lane 0) and the TMEM allocation.
//   warp 10     P.V issue (lane 0).  Separate issuers keep S of later tiles
//               from queueing behind the wait for this tile's P.
//   warp 11     idle (completes the register split's warpgroup).
//   warps 12-15 epilogue: warp 12 + q reads lane quarter q of O once the
//               item's last P.V is done, frees O for the next item and writes
//               O / l with bulk tensor stores, while the softmax warps are
//               already on the next item.
//
// Online softmax in the log2 domain with a lazy reference max: O is rescaled
// in TMEM only when a tile's max exceeds the reference by more than 8 (factor
// 256); the final division by the sum taken against the same reference makes
// the result exact up to rounding.  Keys past the item's last visible key are
// masked, and their V rows are zeroed in shared memory before P.V (the cache
// beyond a sequence may hold anything, even NaN); positions at or past the
// sequence's length are written as zeros whatever their queries hold.
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

constexpr int kBM = 128;          // positions per work item (MMA rows, TMEM lanes)
constexpr int kBN = 128;          // keys per tile
constexpr int kMaxStages = 4;     // K/V ring stages (the launch picks as many as fit)
constexpr int kSoftWarps = 8;     // two groups of four: the key halves of every tile
constexpr int kProdWarp = 8;
constexpr int kSWarp = 9;
constexpr int kPVWarp = 10;      // warp 11 only completes warpgroup 2
constexpr int kEpiWarp0 = 12;    // warps 12-15: the item epilogues, one per TMEM lane quarter
constexpr int kEpiWarps = 4;
constexpr int kThreads = 512;
constexpr int kTmemCols = 512;
constexpr int kSBufs = 3;                   // S / P buffers at columns 0, 128, 256
constexpr uint32_t kTmemO = kSBufs * kBN;   // the O accumulator from column 384
constexpr uint32_t kAtom = 128 * 128;       // one 128-byte-swizzle atom of 128 rows
constexpr float kRescaleLog2 = 8.0f;

// ODONE has four slots (tile mod 4).  P.V completions are waited on only now
// and then (a rescale, the epilogue), when up to three products may still be
// in flight: P.V of tile i - 3 has completed once S of tile i has been read,
// but those of tiles i - 2 .. i may not have.  Four slots keep every such wait
// within one phase of its barrier; with two, a wait for tile i could pass on
// the completion of tile i - 2 (measured: the last tiles of a segment missing
// from O when the values arrived late from DRAM).
constexpr int B_KFULL = 0, B_KEMPTY = 4, B_VFULL = 8, B_VEMPTY = 12, B_QFULL = 16, B_QEMPTY = 17, B_SFULL = 18,
              B_PFULL = 21, B_BFREE = 24, B_ODONE = 27, B_OFREE = 31, B_MDONE = 32, B_LREADY = 34, B_LFREE = 35,
              kNumBars = 36;

template <int D>
struct BlkCfg {
  static constexpr int kHalves = D / 64;                // swizzle atoms across the head dim
  static constexpr uint32_t kQBytes = kHalves * kAtom;  // 128 positions x D
  static constexpr uint32_t kKV = kHalves * kAtom;      // 128 keys x D
  static constexpr uint32_t off_Q = 0;
  // epilogue staging: per epilogue warp two boxes of 32 positions x 32 fp32
  // outputs (4 KB each, 128-byte swizzle): the D/32 chunks go through them in
  // rounds of two
  static constexpr uint32_t kStage = kEpiWarps * 2 * 4096;
  static constexpr uint32_t off_stg = off_Q + kQBytes;
  static constexpr uint32_t off_K = off_stg + kStage;
  // K ring of nk stages, then the V ring of nv
  static __host__ __device__ uint32_t off_V(int nk) { return off_K + nk * kKV; }
  static __host__ __device__ uint32_t off_bar(int nk, int nv) { return off_V(nk) + nv * kKV; }
  static __host__ __device__ uint32_t off_misc(int nk, int nv) { return off_bar(nk, nv) + 512; }
  // the item's row sums, [key half][position], from the softmax to the epilogue warps
  static __host__ __device__ uint32_t off_lsum(int nk, int nv) { return off_misc(nk, nv) + 16; }
  static size_t smem_bytes(int nk, int nv) { return 1024 + off_lsum(nk, nv) + 2 * kBM * 4; }
  static_assert(kTmemO + D <= kTmemCols, "TMEM columns");
  static_assert(kNumBars * 8 <= 512, "barrier area");
};

// Division of a non-negative int below 2^31 by a fixed positive divisor d as
// one multiply and shift (Granlund and Montgomery, "Division by invariant
// integers using multiplication", 1994): with l = ceil(log2 d) and
// m = ceil(2^(31+l) / d) < 2^32, n / d = (m n) >> (31 + l) for 0 <= n < 2^31.
struct FastDiv {
  uint32_t m, s;
  int d;
  __device__ __forceinline__ int div(int n) const { return (int)(((uint64_t)m * (uint32_t)n) >> s); }
  static FastDiv make(int d) {
    int l = 0;
    while ((1ll << l) < d) ++l;
    FastDiv f;
    f.m = (uint32_t)(((1ull << (31 + l)) + (uint64_t)d - 1) / (uint64_t)d);
    f.s = 31 + l;
    f.d = d;
    return f;
  }
};

struct BlkParams {
  const int* seq_len;
  unsigned* status;
  int B, H, Hkv, T, S_cap, L;
  FastDiv by_L, by_H, by_group, by_npb;
  int nqt;             // position tiles per sequence
  int npb;             // tile pairs per (b, h)
  int npairs;          // B * H * npb (below 2^31)
  int nk, nv;          // K and V ring stages
  float scale_log2;
};

// One work item and its keys: positions j0 .. j0+127 of sequence b, query head
// h; keys [0, klen) are visible to some position of the tile, keys [0, mlim)
// to every position below the sequence's length n; nt key tiles.
struct Item {
  int b, h, j0, n, klen, mlim, nt;
};

// The items of this CTA in order: pairs blockIdx.x, +G, ...; in each pair the
// later (larger) tile first.  Items with no visible key are included.
struct Walker {
  int pair, e;
  int cb, cn;  // the last sequence looked up and its clamped length
  __device__ void start() {
    pair = blockIdx.x;
    e = 0;
    cb = -1;
    cn = 0;
  }
  __device__ bool next(const BlkParams& p, Item& it) {
    while (pair < p.npairs) {
      const int bh = p.by_npb.div(pair);
      const int k = pair - bh * p.npb;
      const int qa = p.nqt - 1 - k, qb = k;
      const int e0 = e;
      if (e == 0) {
        e = 1;
      } else {
        e = 0;
        pair += gridDim.x;
      }
      if (e0 == 1 && qb >= qa) continue;  // a pair of one tile (the middle of an odd count)
      it.b = p.by_H.div(bh);
      it.h = bh - it.b * p.H;
      if (it.b != cb) {  // consecutive pairs mostly share the sequence: one load per change
        const int n = p.seq_len[it.b];
        cb = it.b;
        cn = n < 0 ? 0 : (n > p.T ? p.T : n);
      }
      const int n = cn;
      it.n = n;
      it.j0 = (e0 == 0 ? qa : qb) * kBM;
      if (it.j0 < n) {
        const int jl = (it.j0 + kBM < n ? it.j0 + kBM : n) - 1;
        it.klen = p.L * p.by_L.div(jl);
        it.mlim = p.L * p.by_L.div(it.j0);
      } else {
        it.klen = 0;
        it.mlim = 0;
      }
      it.nt = (it.klen + kBN - 1) / kBN;
      return true;
    }
    return false;
  }
};


// One 32 x 32 fp32 box of this warp's staging (rows of 128 bytes, 16-byte
// chunk e of row r at chunk e ^ (r & 7): the 128-byte swizzle) to the output
// at (x, y, z) by a bulk tensor store from lane 0; the staging box stays in
// use until the store has read it (tc::bulk_wait_read_all).
__device__ __forceinline__ void store_box(const CUtensorMap* map, const unsigned char* box, int x, int y, int z,
                                          int lane) {
  tc::fence_async_smem();  // this lane's shared-memory writes, visible to the bulk copy
  __syncwarp();
  if (lane == 0) {
    tc::tma_store_3d(map, x, y, z, box);
    tc::bulk_commit();
  }
}

// Until the bulk store from this warp's staging box has read it.
__device__ __forceinline__ void staging_free(int lane) {
  if (lane == 0) tc::bulk_wait_read_all();
  __syncwarp();
}

// Warpgroup register split (setmaxnreg): the two softmax warpgroups take 168
// registers a thread, the producer / MMA and epilogue warpgroups give theirs
// down to 88, so that each SM sub-partition's 16384 registers hold its four
// warps (2 x 168 + 2 x 88 = 512 per lane) -- exactly the 512 x 128 the block
// is launched with.
__device__ __forceinline__ void regs_up() { asm volatile("setmaxnreg.inc.sync.aligned.u32 168;" ::: "memory"); }
__device__ __forceinline__ void regs_down() { asm volatile("setmaxnreg.dec.sync.aligned.u32 88;" ::: "memory"); }

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    block_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                      const BlkParams p) {
  using C = BlkCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int k_stages = p.nk, v_stages = p.nv;  // K and V ring depths
  const uint32_t off_V = C::off_V(k_stages);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::off_bar(k_stages, v_stages));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + C::off_misc(k_stages, v_stages));
  float* lsum = reinterpret_cast<float*>(base + C::off_lsum(k_stages, v_stages));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::off_misc(k_stages, v_stages) + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int b = 0; b < kNumBars; ++b) {
      const bool soft = (b >= B_PFULL && b < B_PFULL + kSBufs) || b == B_LREADY;
      const bool epi = b == B_OFREE || b == B_LFREE;
      mbar_init(&bars[b], soft ? kSoftWarps : (epi ? kEpiWarps : 1));
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kSWarp) {
    tc::tmem_alloc(tmem_slot, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;
  if (warp >= kSoftWarps) {
  regs_down();
  if (warp == kProdWarp) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::prefetch_tmap(&tmV);
      const uint64_t pol_q = policy_evict_first(), pol_kv = policy_evict_last();
      struct Cursor {  // next tile to load: item it, its tile t, CTA-local tile i, item kq
        Walker w;
        Item it;
        int t, i, kq;
        bool has, qdone;
      };
      auto first = [&](Cursor& c) {  // the next item with keys
        c.has = false;
        while (c.w.next(p, c.it))
          if (c.it.nt > 0) {
            c.has = true;
            c.t = 0;
            c.qdone = false;
            return;
          }
      };
      auto step = [&](Cursor& c) {
        ++c.i;
        if (++c.t == c.it.nt) {
          ++c.kq;
          first(c);
        }
      };
      auto kv_row = [&](const Cursor& c) { return (c.it.b * p.Hkv + p.by_group.div(c.it.h)) * p.S_cap + c.t * kBN; };
      Cursor ck, cv;
      ck.w.start();
      cv.w.start();
      ck.i = cv.i = ck.kq = cv.kq = 0;
      first(ck);
      first(cv);
      int q_issued = 0;
      uint64_t t_last = global_timer_ns();
      int spins = 0, seen = 0;
      while (ck.has || cv.has) {
        bool progressed = false;
        if (ck.has) {
          if (ck.t == 0 && !ck.qdone) {
            if (mbar_test_wait(&bars[B_QEMPTY], (ck.kq & 1) ^ 1)) {
              mbar_arrive_expect_tx(&bars[B_QFULL], C::kQBytes);
              for (int hd = 0; hd < C::kHalves; ++hd)
                tc::tma_load_2d(base + C::off_Q + hd * kAtom, &tmQ, ck.it.h * D + hd * 64, ck.it.b * p.T + ck.it.j0,
                                &bars[B_QFULL], pol_q);
              ck.qdone = true;
              ++q_issued;
              progressed = true;
              {  // the next item's Q into L2, an item ahead of its load
                Walker la = ck.w;
                Item nx;
                while (la.next(p, nx))
                  if (nx.nt > 0) {
                    for (int hd = 0; hd < C::kHalves; ++hd)
                      tc::tma_prefetch_l2_2d(&tmQ, nx.h * D + hd * 64, nx.b * p.T + nx.j0);
                    break;
                  }
              }
            }
          } else if (mbar_test_wait(&bars[B_KEMPTY + ck.i % k_stages], ((ck.i / k_stages) & 1) ^ 1)) {
            const int st = ck.i % k_stages;
            mbar_arrive_expect_tx(&bars[B_KFULL + st], C::kKV);
            for (int hd = 0; hd < C::kHalves; ++hd)
              tc::tma_load_2d(base + C::off_K + st * C::kKV + hd * kAtom, &tmK, hd * 64, kv_row(ck),
                              &bars[B_KFULL + st], pol_kv);
            step(ck);
            progressed = true;
          }
        }
        if (cv.has && mbar_test_wait(&bars[B_VEMPTY + cv.i % v_stages], ((cv.i / v_stages) & 1) ^ 1)) {
          const int st = cv.i % v_stages;
          mbar_arrive_expect_tx(&bars[B_VFULL + st], C::kKV);
          for (int hd = 0; hd < C::kHalves; ++hd)
            tc::tma_load_2d(base + off_V + st * C::kKV + hd * kAtom, &tmV, hd * 64, kv_row(cv), &bars[B_VFULL + st],
                            pol_kv);
          step(cv);
          progressed = true;
        }
        if (progressed) continue;
        // Nothing to do: back off so that this warp leaves its scheduler's
        // issue slots to the softmax warp beside it.
        __nanosleep(32);
        if (++spins < 32) continue;
        spins = 0;  // every 32 idle polls: check for an abort or a stall of more than kWaitLimitNs
        const uint64_t now = global_timer_ns();
        if (ck.i + cv.i + q_issued != seen) {
          seen = ck.i + cv.i + q_issued;
          t_last = now;
        }
        if (*abort_flag) break;
        if (now - t_last > kWaitLimitNs) {
          *abort_flag = 1;
          record_status(p.status, kStatusTimeout);
          break;
        }
      }
      if (ck.has || cv.has) {  // aborted: let issued loads land before the CTA exits
        for (int j = (ck.i > k_stages ? ck.i - k_stages : 0); j < ck.i; ++j)
          mbar_drain(&bars[B_KFULL + j % k_stages], (j / k_stages) & 1);
        for (int j = (cv.i > v_stages ? cv.i - v_stages : 0); j < cv.i; ++j)
          mbar_drain(&bars[B_VFULL + j % v_stages], (j / v_stages) & 1);
        if (q_issued > 0) mbar_drain(&bars[B_QFULL], (q_issued - 1) & 1);
      }
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
      Walker w;
      w.start();
      Item it;
      int i = 0, kq = 0;
      while (ok && w.next(p, it)) {
        if (it.nt == 0) continue;
        for (int t = 0; t < it.nt; ++t, ++i) {
          const int bi = i % kSBufs;
          if (s_role) {
            // S(i) = Q K(i)^T into buffer i % 3, once P.V of tile i - 3 has read that buffer
            if ((t == 0 && !mbar_wait(&bars[B_QFULL], kq & 1, abort_flag, p.status)) ||
                !mbar_wait(&bars[B_KFULL + i % k_stages], (i / k_stages) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_BFREE + bi], ((i / kSBufs) & 1) ^ 1, abort_flag, p.status)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint64_t dK = tc::sw128_desc(sK + (i % k_stages) * C::kKV, 16, 1024);
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint64_t step = desc_step((ks >> 2) * kAtom + (ks & 3) * 32);
              tc::mma_bf16(tmem + bi * kBN, dQ + step, dK + step, idS, ks > 0 ? 1u : 0u);
            }
            tc::mma_commit(&bars[B_SFULL + bi]);
            tc::mma_commit(&bars[B_KEMPTY + i % k_stages]);
            if (t == it.nt - 1) tc::mma_commit(&bars[B_QEMPTY]);
          } else {
            // O (+)= P_0(i) V_0(i) + P_1(i) V_1(i) over the key halves h = 0, 1: P_h in
            // columns 64h .. 64h+31 of buffer i % 3
            const bool first = t == 0;
            if (!mbar_wait(&bars[B_PFULL + bi], (i / kSBufs) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_VFULL + i % v_stages], (i / v_stages) & 1, abort_flag, p.status) ||
                (first && kq > 0 && !mbar_wait(&bars[B_OFREE], (kq - 1) & 1, abort_flag, p.status))) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint64_t dV = tc::sw128_desc(sV + (i % v_stages) * C::kKV, kAtom, 1024);
            const uint32_t pcol = tmem + bi * kBN;
            if (first) {
              tc::mma_bf16_ts(tmem + kTmemO, pcol, dV, idO, 0u);
            } else {
              tc::mma_bf16_ts(tmem + kTmemO, pcol, dV, idO, 1u);
            }
#pragma unroll
            for (int ks = 1; ks < kBN / 16; ++ks)
              tc::mma_bf16_ts(tmem + kTmemO, pcol + (ks >> 2) * 64 + (ks & 3) * 8, dV + desc_step(ks * 16 * 128), idO, 1u);
            tc::mma_commit(&bars[B_VEMPTY + i % v_stages]);
            tc::mma_commit(&bars[B_ODONE + (i & 3)]);
            tc::mma_commit(&bars[B_BFREE + bi]);
          }
        }
        ++kq;
      }
      const int role = s_role ? 0 : 1;
      tc::mma_commit(&bars[B_MDONE + role]);  // every MMA finished before TMEM is released
      mbar_drain(&bars[B_MDONE + role], 0);
    }
  } else if (warp >= kEpiWarp0) {
    // ------------------------------------------------------------ epilogue
    // Warp 12 + q writes positions 32q .. 32q+31 of every item: O / (l_0 + l_1)
    // from TMEM lane quarter q, staged in D/32 boxes and written with bulk
    // tensor stores.  The softmax warps go on with the next item meanwhile; its
    // first P.V waits until O has been read here.
    const int quarter = warp - kEpiWarp0;
    const int r = quarter * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    unsigned char* stg = base + C::off_stg + quarter * 2 * 4096;  // this warp's two boxes
    bool dead = false;
    Walker w;
    w.start();
    Item it;
    int i = 0, ke = 0;
    while (w.next(p, it)) {
      staging_free(lane);  // the previous item's stores have read the boxes
      if (it.nt == 0) {  // no visible key anywhere in the tile: zeros, every chunk from the first box
#pragma unroll
        for (int e = 0; e < 8; ++e)
          *reinterpret_cast<float4*>(stg + lane * 128 + (e << 4)) = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) store_box(&tmO, stg, it.h * D + c * 32, it.j0 + quarter * 32, it.b, lane);
        continue;
      }
      i += it.nt;
      const int jl = i - 1;  // the item's last tile
      const int j = it.j0 + r;
      // a position that saw no key, or past the sequence: zeros
      const bool has_value = j < it.n && p.L * p.by_L.div(j) > 0;
      if (!dead) dead = !warp_wait(&bars[B_LREADY], ke & 1, abort_flag, p.status);
      const float l0 = lsum[r], l1 = lsum[kBM + r];
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_LFREE]);
      ++ke;
      const float inv = has_value ? 1.f / (l0 + l1) : 0.f;
      if (!dead) dead = !warp_wait(&bars[B_ODONE + (jl & 3)], (jl >> 2) & 1, abort_flag, p.status);
      // rounds of two chunks: read from TMEM into the two boxes, then their stores
#pragma unroll 1
      for (int c2 = 0; c2 < D / 32; c2 += 2) {
        if (c2 > 0) staging_free(lane);  // the previous round's stores have read the boxes
        if (!dead) {
          tc::fence_after_sync();
#pragma unroll 1
          for (int c = c2; c < c2 + 2; ++c) {
            uint32_t a[32];
            tc::tmem_ld32(lane_base + kTmemO + c * 32, a);
            tc::tmem_wait_ld();
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
              if (has_value)
                v = make_float4(__uint_as_float(a[4 * q]) * inv, __uint_as_float(a[4 * q + 1]) * inv,
                                __uint_as_float(a[4 * q + 2]) * inv, __uint_as_float(a[4 * q + 3]) * inv);
              *reinterpret_cast<float4*>(stg + (c - c2) * 4096 + lane * 128 + ((q ^ (lane & 7)) << 4)) = v;
            }
          }
        }
        if (c2 + 2 == D / 32) {  // O is read: the next item's P.V may overwrite it
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars[B_OFREE]);
        }
        if (!dead)
#pragma unroll 1
          for (int c = c2; c < c2 + 2; ++c)
            store_box(&tmO, stg + (c - c2) * 4096, it.h * D + c * 32, it.j0 + quarter * 32, it.b, lane);
      }
    }
    if (lane == 0) tc::bulk_wait_all();  // the output stores have landed
  }
  } else {
  regs_up();
    // ------------------------------------------------------------- softmax
    const int kh = warp >> 2, quarter = warp & 3;
    const int r = quarter * 32 + lane;  // this thread's position in the tile (its TMEM lane)
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    const uint32_t o_col = kTmemO + kh * (D / 2);  // this group's half of the O columns
    const int sid = threadIdx.x;        // 0..255 among the softmax threads
    const float sl2 = p.scale_log2;
    bool dead = false;
    Walker w;
    w.start();
    Item it;
    int i = 0, ke = 0;  // CTA-local tile, items with keys
    while (w.next(p, it)) {
      if (it.nt == 0) continue;  // no visible key anywhere in the tile: the epilogue warps write zeros
      const int j = it.j0 + r;
      const bool valid = j < it.n;
      const int rowlim = valid ? p.L * p.by_L.div(j) : 0;  // keys below it are visible to this position
      float m_used = -CUDART_INF_F, l = 0.f;
      for (int t = 0; t < it.nt; ++t, ++i) {
        const int bi = i % kSBufs;
        uint32_t s[64];
        if (!dead) dead = !warp_wait(&bars[B_SFULL + bi], (i / kSBufs) & 1, abort_flag, p.status);
        if (!dead) {
          tc::fence_after_sync();
          tc::tmem_ld32(lane_base + bi * kBN + kh * 64, *reinterpret_cast<uint32_t(*)[32]>(s));
          tc::tmem_ld32(lane_base + bi * kBN + kh * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(s + 32));
          tc::tmem_wait_ld();
        } else {
#pragma unroll
          for (int e = 0; e < 64; ++e) s[e] = 0u;
        }
        // keys at or past this position's limit: -inf (a suffix of the tile)
        const int nv = rowlim - t * kBN - kh * 64;
        if ((t + 1) * kBN > it.mlim && __any_sync(0xffffffffu, nv < 64)) {
#pragma unroll
          for (int e = 0; e < 64; ++e) s[e] = e < nv ? s[e] : 0xff800000u;
        }
        float mx[4] = {__uint_as_float(s[0]), __uint_as_float(s[1]), __uint_as_float(s[2]), __uint_as_float(s[3])};
#pragma unroll
        for (int e = 4; e < 64; e += 8) {
          mx[0] = fmax3(mx[0], __uint_as_float(s[e]), __uint_as_float(s[e + 1]));
          mx[1] = fmax3(mx[1], __uint_as_float(s[e + 2]), __uint_as_float(s[e + 3]));
          if (e + 4 < 64) {
            mx[2] = fmax3(mx[2], __uint_as_float(s[e + 4]), __uint_as_float(s[e + 5]));
            mx[3] = fmax3(mx[3], __uint_as_float(s[e + 6]), __uint_as_float(s[e + 7]));
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
          if (t > 0 && !dead) {  // O holds the P.V of this item's earlier tiles: rescale this group's half
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
          unf2(ffma2(f2(__uint_as_float(s[2 * e]), __uint_as_float(s[2 * e + 1])), sc2, nm2), x0, x1);
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
        const int vrows = it.klen - t * kBN;
        if (vrows < kBN) {  // the item's last tile: clear V rows past its last visible key
          const int st = i % v_stages;
          if (!dead) dead = !warp_wait(&bars[B_VFULL + st], (i / v_stages) & 1, abort_flag, p.status);
          if (!dead)
            for (int idx = sid; idx < (kBN - vrows) * C::kHalves * 8; idx += kSoftWarps * 32) {
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

      // The item's sums to the epilogue warps (the buffer is free once they
      // have read the previous item's).
      if (!dead) dead = !warp_wait(&bars[B_LFREE], (ke & 1) ^ 1, abort_flag, p.status);
      lsum[kh * kBM + r] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_LREADY]);
      ++ke;
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

template <int D>
cudaError_t launch_typed(const AttnArgs& a, cudaStream_t st) {
  using C = BlkCfg<D>;
  static bool configured = false;
  const int limit = smem_optin_bytes();
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(block_attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  // As many stages as fit, the K ring first: S runs up to three tiles ahead of
  // P.V, so the keys are needed earlier than the values.
  int nk = kMaxStages, nv = kMaxStages;
  while ((nk > 2 || nv > 2) && C::smem_bytes(nk, nv) > (size_t)limit) {
    if (nv >= nk && nv > 2)
      --nv;
    else
      --nk;
  }
  if (C::smem_bytes(nk, nv) > (size_t)limit) return cudaErrorNotSupported;
  CUtensorMap mq, mk, mv, mo;
  const long long kv_rows = (long long)a.B * a.Hkv * a.S_cap;
  if (!make_bf16_map(&mq, a.q, (long long)a.B * a.T, (long long)a.H * D, (long long)a.H * D, kBM) ||
      !make_bf16_map(&mk, a.K, kv_rows, D, D, kBN) || !make_bf16_map(&mv, a.V, kv_rows, D, D, kBN) ||
      !make_f32_seq_map(&mo, a.out, a.B, a.T, (long long)a.H * D))
    return cudaErrorNotSupported;
  BlkParams p;
  p.seq_len = a.kv_len;
  p.status = reinterpret_cast<unsigned*>(a.ws);
  p.B = a.B; p.H = a.H; p.Hkv = a.Hkv; p.T = a.T; p.S_cap = a.S_cap; p.L = a.block_L;
  p.by_L = FastDiv::make(a.block_L);
  p.by_H = FastDiv::make(a.H);
  p.by_group = FastDiv::make(a.H / a.Hkv);
  p.nqt = (a.T + kBM - 1) / kBM;
  p.npb = (p.nqt + 1) / 2;
  if ((long long)a.B * a.H * p.npb > 0x7fffffffLL) return cudaErrorNotSupported;
  p.npairs = a.B * a.H * p.npb;
  p.by_npb = FastDiv::make(p.npb);
  p.nk = nk;
  p.nv = nv;
  p.scale_log2 = a.scale * kLog2e;
  int G = a.max_ctas > 0 ? a.max_ctas : sm_count();
  if (G > p.npairs) G = p.npairs;
  if (G < 1) G = 1;
  if ((long long)p.npairs + G > 0x7fffffffLL) return cudaErrorNotSupported;  // a CTA's pair index steps by G
  block_attn_kernel<D><<<(unsigned)G, kThreads, C::smem_bytes(nk, nv), st>>>(mq, mk, mv, mo, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_block_attn(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype != 0 || (a.D != 128 && a.D != 64) || a.block_L < 1 || a.T < 1) return cudaErrorNotSupported;
  if (reinterpret_cast<uintptr_t>(a.out) & 15) return cudaErrorNotSupported;  // bulk tensor stores
  // 32-bit TMA row coordinates, including a tile's reach past the last row
  if ((long long)a.B * a.T + kBM > 0x7fffffffLL || (long long)a.B * a.Hkv * a.S_cap + kBN > 0x7fffffffLL)
    return cudaErrorNotSupported;
  if (a.D == 128) return launch_typed<128>(a, st);
  return launch_typed<64>(a, st);
}

}  // namespace glide
