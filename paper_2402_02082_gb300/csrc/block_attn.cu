// The draft's cross-attention at training time under the block-wise mask
// (Section 3.1, "Block-wise Attention Mask") on the tcgen05 tensor cores.
//
// Position j of a training sequence attends to the target's keys and values
// of the positions k < L * (j / L), the blocks before its own.  Over T
// positions that is a lower-triangular attention of about T^2 / 2 (query,
// key) pairs at 4 D flops each: a compute-bound product, unlike the
// memory-bound decoding kernels.  Both products run on the tensor cores:
//   S = Q K^T   : M = 128 positions, N = 128 keys, K = D, operands in shared memory
//   O += P V    : M = 128, N = D, K = 128 keys, P in tensor memory, V in shared memory
// Q and K sit in shared memory in the 128-byte-swizzled K-major layout, V in
// the M/N-major layout.  Tensor memory (TMEM, 512 columns) holds three S
// buffers of 128 columns and the O accumulator (D columns).  The softmax
// overwrites the first 64 columns of its S buffer with P as bf16 pairs, and
// the P.V product reads P from there: P never passes through shared memory,
// whose bandwidth the MMA operand reads, the TMA writes and P stores would
// otherwise share.  S of tile i + 3 reuses the buffer of tile i, so it waits
// for the completion of P.V of tile i.
//
// Work item: (sequence b, query head h, tile of 128 positions).  Tile x of a
// (b, h) sees about x + 1 key tiles, so tile x is paired with tile
// T/128 - 1 - x and every pair carries the same number of key tiles.  CTA c
// runs pairs c, c + G, c + 2G, ... in (b, h)-major order: the CTAs that run at
// the same time read the keys and values of a few heads, which stay in L2.
//
// Roles (224 threads, one CTA per SM):
//   warps 0-3  softmax: one thread per position (TMEM lane), 128 keys per
//              tile, packed f32x2 arithmetic; then the item's epilogue.
//   warp 4     producer: lane 0 loads the Q tiles (two buffers) and feeds the
//              K and V rings with 2-D TMA, polling the free slots of both.
//   warp 5     S issue (lane 0) and the TMEM allocation.
//   warp 6     P.V issue (lane 0).  Separate issuers keep S of later tiles
//              from queueing behind the wait for this tile's P.
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
#include "tc_ptx.cuh"
#include "tensor_map.h"

namespace glide {
namespace {

constexpr int kBM = 128;          // positions per work item (MMA rows, TMEM lanes)
constexpr int kBN = 128;          // keys per tile
constexpr int kMaxStages = 4;     // K/V ring stages (the launch picks as many as fit)
constexpr int kSoftWarps = 4;
constexpr int kProdWarp = 4;
constexpr int kSWarp = 5;
constexpr int kPVWarp = 6;
constexpr int kThreads = 224;
constexpr int kTmemCols = 512;
constexpr int kSBufs = 3;                   // S / P buffers at columns 0, 128, 256
constexpr uint32_t kTmemO = kSBufs * kBN;   // O accumulator from column 384
constexpr uint32_t kAtom = 128 * 128;       // one 128-byte-swizzle atom of 128 rows
constexpr uint32_t kStage = 4 * 32 * 128;   // epilogue staging: 32 rows x 128 B per softmax warp
constexpr float kRescaleLog2 = 8.0f;
// Every kPolyEvery-th pair of exponentials runs on the FMA pipe (exp2_poly2)
// instead of the MUFU unit, which alone would bound the softmax.
constexpr int kPolyEvery = 6;

constexpr int B_KFULL = 0, B_KEMPTY = 4, B_VFULL = 8, B_VEMPTY = 12, B_QFULL = 16, B_QEMPTY = 18, B_SFULL = 20,
              B_PFULL = 23, B_BFREE = 26, B_ODONE = 29, B_OFREE = 31, B_MDONE = 32, kNumBars = 34;

template <int D>
struct BlkCfg {
  static constexpr int kHalves = D / 64;                // swizzle atoms across the head dim
  static constexpr uint32_t kQBytes = kHalves * kAtom;  // 128 positions x D
  static constexpr uint32_t kKV = kHalves * kAtom;      // 128 keys x D
  static constexpr uint32_t off_Q = 0;                  // two Q buffers
  static constexpr uint32_t off_stg = off_Q + 2 * kQBytes;
  static constexpr uint32_t off_K = off_stg + kStage;
  static __host__ __device__ uint32_t off_V(int ns) { return off_K + ns * kKV; }
  static __host__ __device__ uint32_t off_bar(int ns) { return off_V(ns) + ns * kKV; }
  static __host__ __device__ uint32_t off_misc(int ns) { return off_bar(ns) + 512; }
  static size_t smem_bytes(int ns) { return 1024 + off_misc(ns) + 16; }
  static_assert(kTmemO + D <= kTmemCols, "TMEM columns");
  static_assert(kNumBars * 8 <= 512, "barrier area");
};

struct BlkParams {
  float* out;
  const int* seq_len;
  unsigned* status;
  int B, H, Hkv, group, T, S_cap, L;
  int nqt;             // position tiles per sequence
  int npb;             // tile pairs per (b, h)
  long long npairs;    // B * H * npb
  int ns;              // K/V stages
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
  long long pair;
  int e;
  __device__ void start() {
    pair = blockIdx.x;
    e = 0;
  }
  __device__ bool next(const BlkParams& p, Item& it) {
    while (pair < p.npairs) {
      const int k = (int)(pair % p.npb);
      const long long bh = pair / p.npb;
      const int qa = p.nqt - 1 - k, qb = k;
      const int e0 = e;
      if (e == 0) {
        e = 1;
      } else {
        e = 0;
        pair += gridDim.x;
      }
      if (e0 == 1 && qb >= qa) continue;  // a pair of one tile (the middle of an odd count)
      it.b = (int)(bh / p.H);
      it.h = (int)(bh - (long long)it.b * p.H);
      int n = p.seq_len[it.b];
      n = n < 0 ? 0 : (n > p.T ? p.T : n);
      it.n = n;
      it.j0 = (e0 == 0 ? qa : qb) * kBM;
      if (it.j0 < n) {
        const int jl = (it.j0 + kBM < n ? it.j0 + kBM : n) - 1;
        it.klen = p.L * (jl / p.L);
        it.mlim = p.L * (it.j0 / p.L);
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

// 2^x for a pair of x <= 8 (the lazy reference max keeps every exponent
// there) on the FMA pipe: x = n + f with n = round(x), read from the low
// mantissa bits of x + 1.5 * 2^23, and f in [-1/2, 1/2]; 2^f from a degree-3
// polynomial (relative-error minimax fit by Remez exchange, written by
// exp2_poly.py; max relative error 7.5e-5, far below the bf16 rounding of P);
// n is added to the exponent field.  x is clamped at -126 so the exponent
// cannot wrap: a masked key (-inf) gets 2^-126 instead of 0, which no sum of
// a position with a visible key can notice.
constexpr float kExpC0 = 0.999928074f, kExpC1 = 0.693260985f, kExpC2 = 0.242611122f, kExpC3 = 0.0551716691f;
constexpr float kRound = 12582912.0f;  // 1.5 * 2^23
__device__ __forceinline__ uint64_t exp2_poly2(uint64_t x2) {
  float x0, x1;
  unf2(x2, x0, x1);
  const uint64_t xc = f2(fmaxf(x0, -126.f), fmaxf(x1, -126.f));
  const uint64_t j = fadd2(xc, f2(kRound, kRound));
  const uint64_t n = fadd2(j, f2(-kRound, -kRound));
  const uint64_t f = ffma2(n, f2(-1.f, -1.f), xc);
  uint64_t q = ffma2(f2(kExpC3, kExpC3), f, f2(kExpC2, kExpC2));
  q = ffma2(q, f, f2(kExpC1, kExpC1));
  q = ffma2(q, f, f2(kExpC0, kExpC0));
  float j0, j1, q0, q1;
  unf2(j, j0, j1);
  unf2(q, q0, q1);
  return f2(__uint_as_float(__float_as_uint(q0) + (__float_as_uint(j0) << 23)),
            __uint_as_float(__float_as_uint(q1) + (__float_as_uint(j1) << 23)));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    block_attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const BlkParams p) {
  using C = BlkCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int ns = p.ns;
  const uint32_t off_V = C::off_V(ns);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::off_bar(ns));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + C::off_misc(ns));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::off_misc(ns) + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int b = 0; b < kNumBars; ++b) {
      const bool soft = (b >= B_PFULL && b < B_PFULL + kSBufs) || b == B_OFREE;
      mbar_init(&bars[b], soft ? kSoftWarps : 1);
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
      auto kv_row = [&](const Cursor& c) { return (c.it.b * p.Hkv + c.it.h / p.group) * p.S_cap + c.t * kBN; };
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
            const int qs = ck.kq & 1;
            if (mbar_test_wait(&bars[B_QEMPTY + qs], ((ck.kq >> 1) & 1) ^ 1)) {
              mbar_arrive_expect_tx(&bars[B_QFULL + qs], C::kQBytes);
              for (int hd = 0; hd < C::kHalves; ++hd)
                tc::tma_load_2d(base + C::off_Q + qs * C::kQBytes + hd * kAtom, &tmQ, ck.it.h * D + hd * 64,
                                ck.it.b * p.T + ck.it.j0, &bars[B_QFULL + qs], pol_q);
              ck.qdone = true;
              ++q_issued;
              progressed = true;
            }
          } else if (mbar_test_wait(&bars[B_KEMPTY + ck.i % ns], ((ck.i / ns) & 1) ^ 1)) {
            const int st = ck.i % ns;
            mbar_arrive_expect_tx(&bars[B_KFULL + st], C::kKV);
            for (int hd = 0; hd < C::kHalves; ++hd)
              tc::tma_load_2d(base + C::off_K + st * C::kKV + hd * kAtom, &tmK, hd * 64, kv_row(ck),
                              &bars[B_KFULL + st], pol_kv);
            step(ck);
            progressed = true;
          }
        }
        if (cv.has && mbar_test_wait(&bars[B_VEMPTY + cv.i % ns], ((cv.i / ns) & 1) ^ 1)) {
          const int st = cv.i % ns;
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
        for (int j = (ck.i > ns ? ck.i - ns : 0); j < ck.i; ++j) mbar_drain(&bars[B_KFULL + j % ns], (j / ns) & 1);
        for (int j = (cv.i > ns ? cv.i - ns : 0); j < cv.i; ++j) mbar_drain(&bars[B_VFULL + j % ns], (j / ns) & 1);
        for (int q = (q_issued > 2 ? q_issued - 2 : 0); q < q_issued; ++q)
          mbar_drain(&bars[B_QFULL + (q & 1)], (q >> 1) & 1);
      }
    }
  } else if (warp == kSWarp || warp == kPVWarp) {
    // ----------------------------------------------------------- MMA issue
    if (lane == 0) {
      const bool s_role = warp == kSWarp;
      constexpr uint32_t idS = tc::idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t idO = tc::idesc_bf16_f32(kBM, D, false, true);
      const uint32_t sQ = smem_u32(base + C::off_Q);
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
            if ((t == 0 && !mbar_wait(&bars[B_QFULL + (kq & 1)], (kq >> 1) & 1, abort_flag, p.status)) ||
                !mbar_wait(&bars[B_KFULL + i % ns], (i / ns) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_BFREE + bi], ((i / kSBufs) & 1) ^ 1, abort_flag, p.status)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t qb = sQ + (kq & 1) * C::kQBytes, kb = sK + (i % ns) * C::kKV;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint64_t a = tc::sw128_desc(qb + (ks >> 2) * kAtom + (ks & 3) * 32, 16, 1024);
              const uint64_t bdesc = tc::sw128_desc(kb + (ks >> 2) * kAtom + (ks & 3) * 32, 16, 1024);
              tc::mma_bf16(tmem + bi * kBN, a, bdesc, idS, ks > 0 ? 1u : 0u);
            }
            tc::mma_commit(&bars[B_SFULL + bi]);
            tc::mma_commit(&bars[B_KEMPTY + i % ns]);
            if (t == it.nt - 1) tc::mma_commit(&bars[B_QEMPTY + (kq & 1)]);
          } else {
            // O (+)= P(i) V(i), P from the first 64 columns of buffer i % 3
            const bool first = t == 0;
            if (!mbar_wait(&bars[B_PFULL + bi], (i / kSBufs) & 1, abort_flag, p.status) ||
                !mbar_wait(&bars[B_VFULL + i % ns], (i / ns) & 1, abort_flag, p.status) ||
                (first && kq > 0 && !mbar_wait(&bars[B_OFREE], (kq - 1) & 1, abort_flag, p.status))) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t vb = sV + (i % ns) * C::kKV;
#pragma unroll
            for (int ks = 0; ks < kBN / 16; ++ks) {
              const uint64_t bdesc = tc::sw128_desc(vb + ks * 16 * 128, kAtom, 1024);
              tc::mma_bf16_ts(tmem + kTmemO, tmem + bi * kBN + ks * 8, bdesc, idO, (first && ks == 0) ? 0u : 1u);
            }
            tc::mma_commit(&bars[B_VEMPTY + i % ns]);
            tc::mma_commit(&bars[B_ODONE + (i & 1)]);
            tc::mma_commit(&bars[B_BFREE + bi]);
          }
        }
        ++kq;
      }
      const int role = s_role ? 0 : 1;
      tc::mma_commit(&bars[B_MDONE + role]);  // every MMA finished before TMEM is released
      mbar_drain(&bars[B_MDONE + role], 0);
    }
  } else {
    // ------------------------------------------------------------- softmax
    const int r = warp * 32 + lane;  // this thread's position in the tile (its TMEM lane)
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
    const int sid = threadIdx.x;     // 0..127 among the softmax threads
    const float sl2 = p.scale_log2;
    unsigned char* stg = base + C::off_stg + warp * 4096;  // this warp's 32 rows x 128 B of staging
    bool dead = false;
    Walker w;
    w.start();
    Item it;
    int i = 0, kq = 0;
    while (w.next(p, it)) {
      if (it.nt == 0) {  // no visible key anywhere in the tile: zeros, four 128-byte rows per store
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c)
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int jr = it.j0 + warp * 32 + k * 4 + (lane >> 3);
            if (jr < p.T)
              *reinterpret_cast<float4*>(p.out + (((size_t)it.b * p.T + jr) * p.H + it.h) * D + c * 32 +
                                         (lane & 7) * 4) = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        continue;
      }
      const int j = it.j0 + r;
      const bool valid = j < it.n;
      const int rowlim = valid ? p.L * (j / p.L) : 0;  // keys below it are visible to this position
      float m_used = -CUDART_INF_F, l = 0.f;
      for (int t = 0; t < it.nt; ++t, ++i) {
        const int bi = i % kSBufs;
        uint32_t s[kBN];
        if (!dead) dead = !warp_wait(&bars[B_SFULL + bi], (i / kSBufs) & 1, abort_flag, p.status);
        if (!dead) {
          tc::fence_after_sync();
#pragma unroll
          for (int c = 0; c < kBN / 32; ++c)
            tc::tmem_ld32(lane_base + bi * kBN + c * 32, *reinterpret_cast<uint32_t(*)[32]>(s + c * 32));
          tc::tmem_wait_ld();
        } else {
#pragma unroll
          for (int e = 0; e < kBN; ++e) s[e] = 0u;
        }
        // keys at or past this position's limit: -inf (a suffix of the tile)
        const int nv = rowlim - t * kBN;
        if ((t + 1) * kBN > it.mlim && __any_sync(0xffffffffu, nv < kBN)) {
#pragma unroll
          for (int e = 0; e < kBN; ++e) s[e] = e < nv ? s[e] : 0xff800000u;
        }
        // row max of the raw scores (the scale is positive), then in the log2 domain
        float mx[4] = {__uint_as_float(s[0]), __uint_as_float(s[1]), __uint_as_float(s[2]), __uint_as_float(s[3])};
#pragma unroll
        for (int e = 4; e < kBN; e += 8) {
          mx[0] = fmax3(mx[0], __uint_as_float(s[e]), __uint_as_float(s[e + 1]));
          mx[1] = fmax3(mx[1], __uint_as_float(s[e + 2]), __uint_as_float(s[e + 3]));
          if (e + 4 < kBN) {
            mx[2] = fmax3(mx[2], __uint_as_float(s[e + 4]), __uint_as_float(s[e + 5]));
            mx[3] = fmax3(mx[3], __uint_as_float(s[e + 6]), __uint_as_float(s[e + 7]));
          }
        }
        const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * sl2;

        const bool need = tmax > m_used + kRescaleLog2;
        if (__any_sync(0xffffffffu, need)) {
          const float m_new = need ? tmax : m_used;
          const float f = need ? fast_exp2(m_used - m_new) : 1.f;
          l *= f;
          if (t > 0 && !dead) {  // O holds the P.V of this item's earlier tiles
            dead = !warp_wait(&bars[B_ODONE + ((i - 1) & 1)], ((i - 1) >> 1) & 1, abort_flag, p.status);
            if (!dead) {
              tc::fence_after_sync();
#pragma unroll 1
              for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                tc::tmem_ld32(lane_base + kTmemO + c * 32, o);
                tc::tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * f);
                tc::tmem_st32(lane_base + kTmemO + c * 32, o);
              }
              tc::tmem_wait_st();
            }
          }
          m_used = m_new;
        }
        // p = 2^(s * scale * log2(e) - m), summed in fp32 and packed to bf16 pairs
        const float m_eff = m_used == -CUDART_INF_F ? 0.f : m_used;
        const uint64_t sc2 = f2(sl2, sl2), nm2 = f2(-m_eff, -m_eff);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
        uint32_t pk[kBN / 2];
#pragma unroll
        for (int e = 0; e < kBN / 2; ++e) {
          const uint64_t x2 = ffma2(f2(__uint_as_float(s[2 * e]), __uint_as_float(s[2 * e + 1])), sc2, nm2);
          float p0, p1;
          if (kPolyEvery > 0 && e % kPolyEvery == kPolyEvery - 1) {
            unf2(exp2_poly2(x2), p0, p1);
          } else {
            float x0, x1;
            unf2(x2, x0, x1);
            p0 = fast_exp2(x0);
            p1 = fast_exp2(x1);
          }
          acc[e & 3] = fadd2(acc[e & 3], f2(p0, p1));
          pk[e] = pack_bf16x2(p0, p1);
        }
        {
          float a0, a1, b0, b1;
          unf2(fadd2(acc[0], acc[1]), a0, a1);
          unf2(fadd2(acc[2], acc[3]), b0, b1);
          l += (a0 + a1) + (b0 + b1);
        }
        if (!dead) {  // P over the first 64 columns of this tile's S buffer
          tc::tmem_st32(lane_base + bi * kBN, *reinterpret_cast<const uint32_t(*)[32]>(pk));
          tc::tmem_st32(lane_base + bi * kBN + 32, *reinterpret_cast<const uint32_t(*)[32]>(pk + 32));
          tc::tmem_wait_st();
        }
        const int vrows = it.klen - t * kBN;
        if (vrows < kBN) {  // the item's last tile: clear V rows past its last visible key
          const int st = i % ns;
          if (!dead) dead = !warp_wait(&bars[B_VFULL + st], (i / ns) & 1, abort_flag, p.status);
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

      // ---- item epilogue: O / l, 32 columns at a time, staged so that every
      // store writes four whole 128-byte rows.  O is released at the end: the
      // next item's first P.V also waits for its P, which these warps write
      // only after this epilogue.
      const int jl = i - 1;
      const bool has_value = rowlim > 0;  // a position that saw no key, or past the sequence: zeros
      const float inv = has_value ? 1.f / l : 0.f;
      if (!dead) dead = !warp_wait(&bars[B_ODONE + (jl & 1)], (jl >> 1) & 1, abort_flag, p.status);
      if (!dead) {
        tc::fence_after_sync();
        // the load of chunk c + 1 is in flight while chunk c is staged and stored
        uint32_t o[2][32];
        tc::tmem_ld32(lane_base + kTmemO, o[0]);
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          tc::tmem_wait_ld();
          if (c + 1 < D / 32) tc::tmem_ld32(lane_base + kTmemO + (c + 1) * 32, o[(c + 1) & 1]);
          const uint32_t* oc = o[c & 1];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (has_value)
              v = make_float4(__uint_as_float(oc[4 * e]) * inv, __uint_as_float(oc[4 * e + 1]) * inv,
                              __uint_as_float(oc[4 * e + 2]) * inv, __uint_as_float(oc[4 * e + 3]) * inv);
            *reinterpret_cast<float4*>(stg + lane * 128 + ((e ^ (lane & 7)) << 4)) = v;
          }
          __syncwarp();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int rr = k * 4 + (lane >> 3), cc = lane & 7;
            const float4 v = *reinterpret_cast<const float4*>(stg + rr * 128 + ((cc ^ (rr & 7)) << 4));
            const int jr = it.j0 + warp * 32 + rr;
            if (jr < p.T)
              *reinterpret_cast<float4*>(p.out + (((size_t)it.b * p.T + jr) * p.H + it.h) * D + c * 32 + cc * 4) = v;
          }
          __syncwarp();
        }
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_OFREE]);
      ++kq;
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
  int ns = kMaxStages;
  while (ns > 2 && C::smem_bytes(ns) > (size_t)limit) --ns;
  if (C::smem_bytes(ns) > (size_t)limit) return cudaErrorNotSupported;
  CUtensorMap mq, mk, mv;
  const long long kv_rows = (long long)a.B * a.Hkv * a.S_cap;
  if (!make_bf16_map(&mq, a.q, (long long)a.B * a.T, (long long)a.H * D, (long long)a.H * D, kBM) ||
      !make_bf16_map(&mk, a.K, kv_rows, D, D, kBN) || !make_bf16_map(&mv, a.V, kv_rows, D, D, kBN))
    return cudaErrorNotSupported;
  BlkParams p;
  p.out = a.out;
  p.seq_len = a.kv_len;
  p.status = reinterpret_cast<unsigned*>(a.ws);
  p.B = a.B; p.H = a.H; p.Hkv = a.Hkv; p.group = a.H / a.Hkv; p.T = a.T; p.S_cap = a.S_cap; p.L = a.block_L;
  p.nqt = (a.T + kBM - 1) / kBM;
  p.npb = (p.nqt + 1) / 2;
  p.npairs = (long long)a.B * a.H * p.npb;
  p.ns = ns;
  p.scale_log2 = a.scale * kLog2e;
  long long G = a.max_ctas > 0 ? a.max_ctas : sm_count();
  if (G > p.npairs) G = p.npairs;
  if (G < 1) G = 1;
  block_attn_kernel<D><<<(unsigned)G, kThreads, C::smem_bytes(ns), st>>>(mq, mk, mv, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_block_attn(const AttnArgs& a, cudaStream_t st) {
  if (a.dtype != 0 || (a.D != 128 && a.D != 64) || a.block_L < 1 || a.T < 1) return cudaErrorNotSupported;
  // 32-bit TMA row coordinates, including a tile's reach past the last row
  if ((long long)a.B * a.T + kBM > 0x7fffffffLL || (long long)a.B * a.Hkv * a.S_cap + kBN > 0x7fffffffLL)
    return cudaErrorNotSupported;
  if (a.D == 128) return launch_typed<128>(a, st);
  return launch_typed<64>(a, st);
}

}  // namespace glide
