// Dirty-query attention on the tensor cores (Section 3.3, Region-Level Sparse
// Attention): the queries of the active tokens attend over every token's keys
// and values.  In the self-attention K/V come from the (layer, timestep) cache
// whose dirty rows the QKV GEMM has just refreshed; in the text cross-
// attention they are the per-layer text keys / values.
//
// One work unit = 128 queries of one head over one split of the keys.  CTAs
// are persistent and warp-specialised:
//   warp 0     TMA: Q once per unit, then K/V blocks of 64 keys (4 stages).
//              Every operand comes through 3-D tensor maps (head_dim, head,
//              row) as a 64-wide 128B-swizzled tile plus a 16-wide 32B-
//              swizzled tail; the head_dim extent is the true 72, so the pad
//              to 80 reads as zero and adds nothing to Q K^T.
//   warp 1     TMEM owner and MMA issuer, polling its inputs: O += P V
//              (M=128, N=80, 4 K-steps of 16 keys; P read from TMEM as the A
//              operand, V from shared memory as an MN-major B operand) as
//              soon as P is ready, and S = Q K^T (M=128, N=64, 5 K-steps of
//              16) into one of two TMEM S buffers as soon as the block's K/V
//              have landed and the softmax has read that buffer's last S
//              (so S runs up to two blocks ahead of the softmax).
//   warps 2-5  softmax, one thread per query row: reads its S row from TMEM
//              (freeing the buffer), online softmax in base 2 with lazy
//              rescaling (O in TMEM is rescaled only when the running max
//              grows by more than 2^8), and writes its P row (bf16 pairs) to
//              the TMEM P buffer once the previous P V has read it.  At the
//              end it normalises O.
// Two CTAs share an SM (256 TMEM columns and ~100 KB of shared memory each),
// so the softmax of one overlaps the MMAs and exponentials of the other.
// Key splits of the same (query tile, head) leave their unnormalised O and
// row max / sum in a workspace (as column planes, so that the softmax
// threads' stores are whole 512-byte runs); a small combine kernel, launched
// right after, merges them (one lane per row).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace rc {

namespace {

using namespace rc::tc;

constexpr int BQ = 128, BKV = 64, THREADS = 192;
constexpr int TMEM_COLS = 256;     // S0 | S1 (64 columns each) | O (80) | P (32)
constexpr int CTAS_PER_SM = 2;
// floats per row of a workspace slot: a piece's DH columns, its row max and
// sum (stored as column planes, see attn_combine_kernel)
constexpr int PART_STRIDE = 76;
static_assert(72 + 2 <= PART_STRIDE, "a slot holds DH + 2 floats per row");
constexpr float LAZY_RESCALE = 8.f;
constexpr int MIN_KB_PER_SPLIT = 4;  // key blocks per CTA range, at least

// Packed f32x2 arithmetic (two lanes of f32 per 64-bit register pair).
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack_f32x2(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma_f32x2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add_f32x2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// 2^x on the special-function unit (flushes subnormal results to zero; the
// argument is at most 8 here).
__device__ __forceinline__ float ex2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int DH>
struct ACfg {
  static_assert(DH == 64 || DH == 72, "head_dim 64 or 72");
  static constexpr bool TAIL = DH > 64;          // head dims 64..79 (72..79 read as zero)
  static constexpr int DHP = TAIL ? 80 : 64;     // padded head dim of the PV accumulator
  // shared-memory operand tiles: a 64-wide 128B-swizzled part, a 16-wide
  // 32B-swizzled tail
  static constexpr int Q128 = BQ * 128, Q32 = TAIL ? BQ * 32 : 0;
  static constexpr int K128 = BKV * 128, K32 = TAIL ? BKV * 32 : 0;
  // K: 64-wide SW128 tile + 16-wide SW32 tail (the S MMA reads them as two
  // K-major operands); V: one SW128 atom per 64 head-dim columns, so that P V
  // is a single MMA of N = DHP per 16 keys (MN-major B spanning the atoms)
  static constexpr int K_BYTES = K128 + K32;
  static constexpr int V_BYTES = TAIL ? 2 * K128 : K128;
  // separate rings: K (read by the S MMAs, refilled by the thread that
  // issues them) and V (read by the P V MMAs, refilled by their issuer)
  static constexpr int K_STAGES = TAIL ? 4 : 5;
  static constexpr int V_STAGES = TAIL ? 3 : 4;
  static constexpr int Q_BYTES = Q128 + Q32;
  static constexpr size_t SMEM =
      size_t(Q_BYTES) + K_STAGES * K_BYTES + V_STAGES * V_BYTES + 1024 + 256;
  // kind::f16, D f32, A/B bf16; S: both K-major; PV: B (V) MN-major (bit 16)
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) |
                                      (uint32_t(BKV >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_PV = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) |
                                       (uint32_t(DHP >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
};

// Query tile qt of a launch: its item, first compact row and live rows.
struct TileLoc {
  int item, row0, rows;
};
__device__ __forceinline__ TileLoc locate_tile(const RowMap& rm, int n_items, int D, int qt) {
  if (!rm.meta) return TileLoc{0, qt * BQ, min(BQ, D - qt * BQ)};
  int i = 0;
  while (i + 1 < n_items && __ldg(rm.meta + META_TILE + i + 1) <= qt) ++i;
  const int j = qt - __ldg(rm.meta + META_TILE + i);
  return TileLoc{i, __ldg(rm.meta + META_OFF + i) + j * BQ,
                 min(BQ, __ldg(rm.meta + META_CNT + i) - j * BQ)};
}

// Query tiles of a launch: 128-row tiles of each item's rows.
__device__ __forceinline__ int query_tiles(const RowMap& rm, int n_items, int D) {
  return rm.meta ? __ldg(rm.meta + META_TILE + n_items) : (D + BQ - 1) / BQ;
}

// Work list of one launch, identical in every thread.  A pair = one query
// tile of one head (heads outermost).  With at least 2 MIN_KB_PER_SPLIT key
// blocks (the self-attention) the (pair, key block) sequence is cut into G
// equal contiguous ranges, one per CTA (stream-K): every CTA does the same
// number of key blocks, and a pair cut by a range boundary leaves partial
// results (unnormalised O, row max and sum) that the combine kernel merges.
// With fewer key blocks (the text cross-attention) every pair is one unit,
// handed out round-robin.
//
// G: as many CTAs as the grid holds (at least MIN_KB_PER_SPLIT key blocks
// each), unless ranges of r key blocks, r a power of two dividing the pair's
// count, cost less: then every CTA holds exactly one piece of one pair.  The
// estimate is the busiest CTA's key blocks plus PIECE_COST per piece it
// holds (a piece costs a Q load, a drained O and a stored partial; the equal
// cut leaves most CTAs two).  Measured on the 4096-token step: at 205 dirty
// queries (2048 key blocks) 304 ranges of 6-7 blocks gave 441 steps/s, 256
// of 8 blocks 460; at 410 (4096 key blocks) 304 of 13-14 gave 363, 256 of 16
// gave 389; from 831 queries on, the equal cut stays.
struct AttnSched {
  int qtiles, pairs, nkb, G, total;
  bool streamk;
  static constexpr int PIECE_COST = 4;  // key blocks
  __device__ void init(int tiles, int heads, int Nk, int grid) {
    qtiles = tiles;
    pairs = qtiles * heads;
    nkb = (Nk + BKV - 1) / BKV;
    total = pairs * nkb;
    streamk = nkb >= 2 * MIN_KB_PER_SPLIT;
    G = grid;
    if (!streamk) return;
    G = pick_ctas(total, nkb, grid);
  }
  // (powers of two only, found with shifts: every thread of the attention
  // and combine kernels runs this before its first load, and a search with
  // run-time divisors cost more than the better ranges saved; not inlined,
  // so that its temporaries do not raise the kernels' register counts)
  static __device__ __noinline__ int pick_ctas(int total, int nkb, int grid) {
    const int G = max(1, min(grid, total / MIN_KB_PER_SPLIT));
    if (nkb & (nkb - 1)) return G;
    int lg = 0;
    while ((1 << lg) < MIN_KB_PER_SPLIT) ++lg;
    while ((1 << lg) < nkb && (total >> lg) > grid) ++lg;
    if ((1 << lg) > nkb || (total >> lg) > grid) return G;
    const int r0 = (total + G - 1) / G;
    const bool one_piece = total % G == 0 && nkb % r0 == 0;
    return (1 << lg) + PIECE_COST < r0 + PIECE_COST * (one_piece ? 1 : 2) ? total >> lg : G;
  }
  // unsigned 32-bit arithmetic: the launcher checks total * G < 2^32
  __device__ int bound(int c) const { return int(unsigned(total) * unsigned(c) / unsigned(G)); }
  // the CTA whose range holds key-block position pos (0 <= pos < total)
  __device__ int cta_of(int pos) const {
    int c = int(unsigned(pos) * unsigned(G) / unsigned(total));
    while (c > 0 && bound(c) > pos) --c;
    while (c + 1 < G && bound(c + 1) <= pos) ++c;
    return c;
  }
};

// One CTA's segments in order: (pair, key blocks [kb0, kb1), slot), slot -1
// for a whole pair (its normalised output is written directly), 0 / 1 for
// the CTA's first / last partial piece (workspace slot 2 c + slot).
struct AttnSeg {
  const AttnSched* sc;
  int cur, end;
  bool first;
  __device__ void init(const AttnSched& s, int c) {
    sc = &s;
    first = true;
    if (s.streamk) {
      cur = c < s.G ? s.bound(c) : 0;
      end = c < s.G ? s.bound(c + 1) : 0;
    } else {
      cur = c;  // next pair
      end = s.pairs;
    }
  }
  __device__ bool next(int& pair, int& kb0, int& kb1, int& slot) {
    if (cur >= end) return false;
    if (!sc->streamk) {
      pair = cur;
      kb0 = 0;
      kb1 = sc->nkb;
      slot = -1;
      cur += sc->G;
      return true;
    }
    pair = cur / sc->nkb;
    kb0 = cur - pair * sc->nkb;
    kb1 = min(sc->nkb, kb0 + (end - cur));
    cur += kb1 - kb0;
    slot = (kb0 == 0 && kb1 == sc->nkb) ? -1 : (first ? 0 : 1);
    first = false;
    return true;
  }
};

template <int DH>
__global__ void __launch_bounds__(THREADS, CTAS_PER_SM)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQt,
               const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmKt,
               const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnItems ai, int Nk, bf16* __restrict__ O, int ldo,
               int heads, RowMap rm, float scale_log2, unsigned* err, float* __restrict__ part,
               const __grid_constant__ AttnCapture cap) {
  using C = ACfg<DH>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  constexpr int KS = C::K_STAGES, VS = C::V_STAGES;
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + KS * C::K_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + VS * C::V_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 30);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // barrier addresses
  const uint32_t b0 = saddr(bars);
  const uint32_t q_full = b0, q_empty = b0 + 8;
  const uint32_t k_full = b0 + 16, k_empty = k_full + 8 * KS;
  const uint32_t v_full = k_empty + 8 * KS;
  const uint32_t s_full = v_full + 8 * VS;           // [2]: S of a block is in TMEM
  const uint32_t s_free = s_full + 16;               // [2]: the softmax has read it
  const uint32_t p_ready = s_free + 16;              // P of the next block is in TMEM
  const uint32_t pv_done = p_ready + 8;              // one phase per completed P V
  const uint32_t o_full = pv_done + 8, o_free = o_full + 8;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int s = 0; s < KS; ++s) {
      mbar_init(k_full + 8 * s, 1);
      mbar_init(k_empty + 8 * s, 1);
    }
    for (int s = 0; s < VS; ++s) mbar_init(v_full + 8 * s, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full + 8 * b, 1);
      mbar_init(s_free + 8 * b, 128);
    }
    mbar_init(p_ready, 128);
    mbar_init(pv_done, 1);
    mbar_init(o_full, 1);
    mbar_init(o_free, 128);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(saddr(tmem_slot), TMEM_COLS);
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
    if (C::TAIL) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQt)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmKt)) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t tS0 = tmem_base, tO = tmem_base + 2 * BKV, tP = tO + 80;

  // the live row count (and, for several items, the row table) was written
  // two or more launches earlier: read before the programmatic-dependency
  // wait (every kernel of the library waits for its predecessor before
  // letting its successor start); Q and the fresh K / V rows come from the
  // predecessor
  const int D = live_count(rm.count, rm.bound, err);
  AttnSched sc;
  sc.init(query_tiles(rm, ai.n, D), heads, Nk, gridDim.x);
  pdl_wait();
  pdl_trigger();

  // Two issuing threads, so that neither MMA stream waits behind the other's
  // instruction issue: warp 0 loads Q and K and issues the S MMAs, warp 1
  // loads V and issues the P V MMAs.  Each refills its own ring.
  if (warp == 0) {
    // ------------------------------------------------- Q, K loads and S = Q K^T
    // K runs KS - 2 key blocks ahead of the S MMAs: the K stage of block
    // g + KS - 2 is the one block g - 2 used, whose S has long completed, so
    // the refill never waits on the MMA just issued.  S(g) goes into the S
    // buffer the softmax of block g - 2 has read.
    if (lane == 0) {
      const uint32_t qb = saddr(sQ), kb_0 = saddr(sK);
      const uint64_t dq = sw128_desc(qb), dqt = sw32_kmajor_desc(qb + C::Q128);
      // stage descriptors differ only in the start address field (address >>
      // 4, which never carries out of its 14 bits here)
      const uint64_t dk = sw128_desc(kb_0), dkt = sw32_kmajor_desc(kb_0 + C::K128);
      int gl = 0, gs = 0, uc = 0;
      AttnSeg itl;
      itl.init(sc, blockIdx.x);
      int l_kb = 0, l_kb1 = 0, l_h = 0, l_row = 0;
      bool l_more = true;
      // requests K of the next key block to load (false: a wait gave up)
      auto load_k = [&]() -> bool {
        while (l_kb >= l_kb1) {
          int pair, kb0, kb1, slot;
          if (!itl.next(pair, kb0, kb1, slot)) {
            l_more = false;
            return true;
          }
          const TileLoc tl = locate_tile(rm, ai.n, D, pair % sc.qtiles);
          l_h = pair / sc.qtiles;
          l_row = ai.krow[tl.item];
          l_kb = kb0;
          l_kb1 = kb1;
        }
        const int st = gl % KS;
        if (!mbar_sleep(k_empty + 8 * st, ((gl / KS) & 1) ^ 1, abort_flag)) return false;
        mbar_expect_tx(k_full + 8 * st, C::K_BYTES);
        uint8_t* base = sK + st * C::K_BYTES;
        tma_load_3d(saddr(base), &tmK, k_full + 8 * st, 0, l_h, l_row + l_kb * BKV);
        if (C::TAIL)
          tma_load_3d(saddr(base + C::K128), &tmKt, k_full + 8 * st, 64, l_h, l_row + l_kb * BKV);
        ++l_kb;
        ++gl;
        return true;
      };
      AttnSeg it;
      it.init(sc, blockIdx.x);
      int pair, kb0, kb1, slot;
      for (; it.next(pair, kb0, kb1, slot); ++uc) {
        const int qt = pair % sc.qtiles, h = pair / sc.qtiles;
        const TileLoc tl = locate_tile(rm, ai.n, D, qt);
        const int n = kb1 - kb0;
        // Q of the unit, once the previous unit's S MMAs have read the buffer
        if (!mbar_sleep(q_empty, (uc + 1) & 1, abort_flag)) goto timeout;
        mbar_expect_tx(q_full, C::Q_BYTES);
        tma_load_3d(saddr(sQ), &tmQ, q_full, 0, h, tl.row0);
        if (C::TAIL) tma_load_3d(saddr(sQ + C::Q128), &tmQt, q_full, 64, h, tl.row0);
        for (int ns = 0; ns < n; ++ns, ++gs) {
          while (l_more && gl < gs + KS - 1) {
            if (!load_k()) goto timeout;
          }
          if (ns == 0 && !mbar_sleep(q_full, uc & 1, abort_flag)) goto timeout;
          const int st = gs % KS;
          if (!mbar_sleep(k_full + 8 * st, (gs / KS) & 1, abort_flag) ||
              !mbar_sleep(s_free + 8 * (gs & 1), ((gs >> 1) + 1) & 1, abort_flag))
            goto timeout;
          tc_fence_after();
          const uint64_t so = uint64_t(st * (C::K_BYTES >> 4));
          const uint32_t sd = tS0 + uint32_t(BKV) * uint32_t(gs & 1);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            umma_bf16(sd, dq + 2 * kk, dk + so + 2 * kk, C::IDESC_S, kk > 0 ? 1u : 0u);
          if (C::TAIL) umma_bf16(sd, dqt, dkt + so, C::IDESC_S, 1u);
          umma_commit(k_empty + 8 * st);
          umma_commit(s_full + 8 * (gs & 1));
          if (ns == n - 1) umma_commit(q_empty);  // last S of the unit issued
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------ V loads and O += P V
    // V runs VS key blocks ahead: after P V(g) the thread waits for it to
    // complete (pv_done, which the softmax waits for too; the thread has time:
    // P(g + 1) takes a whole softmax) and refills the stage with V(g + VS).
    if (lane == 0) {
      const uint64_t dv = sw128_mnmajor_desc_lbo(saddr(sV), C::K128);
      int gv = 0, g = 0, uc = 0;
      AttnSeg itl;
      itl.init(sc, blockIdx.x);
      int l_kb = 0, l_kb1 = 0, l_h = 0, l_row = 0;
      bool l_more = true;
      auto load_v = [&]() -> bool {
        while (l_kb >= l_kb1) {
          int pair, kb0, kb1, slot;
          if (!itl.next(pair, kb0, kb1, slot)) {
            l_more = false;
            return true;
          }
          const TileLoc tl = locate_tile(rm, ai.n, D, pair % sc.qtiles);
          l_h = pair / sc.qtiles;
          l_row = ai.vrow[tl.item];
          l_kb = kb0;
          l_kb1 = kb1;
        }
        const int st = gv % VS;
        // the stage's previous block, gv - VS, is the P V just issued
        if (gv >= VS && !mbar_sleep(pv_done, (gv - VS) & 1, abort_flag)) return false;
        mbar_expect_tx(v_full + 8 * st, C::V_BYTES);
        uint8_t* base = sV + st * C::V_BYTES;
        tma_load_3d(saddr(base), &tmV, v_full + 8 * st, 0, l_h, l_row + l_kb * BKV);
        if (C::TAIL)
          tma_load_3d(saddr(base + C::K128), &tmV, v_full + 8 * st, 64, l_h, l_row + l_kb * BKV);
        ++l_kb;
        ++gv;
        return true;
      };
      while (l_more && gv < VS) {
        if (!load_v()) goto timeout;
      }
      AttnSeg it;
      it.init(sc, blockIdx.x);
      int pair, kb0, kb1, slot;
      for (; it.next(pair, kb0, kb1, slot); ++uc) {
        const int n = kb1 - kb0;
        for (int np = 0; np < n; ++np, ++g) {
          if (np == 0 && !mbar_sleep(o_free, (uc + 1) & 1, abort_flag)) goto timeout;
          const int st = g % VS;
          if (!mbar_sleep(p_ready, g & 1, abort_flag) ||
              !mbar_sleep(v_full + 8 * st, (g / VS) & 1, abort_flag))
            goto timeout;
          tc_fence_after();
          const uint64_t vd = dv + uint64_t(st * (C::V_BYTES >> 4));
          // 16 keys per MMA: P columns 8 kk .., V rows 16 kk .. (2 KB)
#pragma unroll
          for (int kk = 0; kk < BKV / 16; ++kk)
            umma_bf16_ta(tO, tP + 8 * kk, vd + 128 * kk, C::IDESC_PV,
                         (np > 0 || kk > 0) ? 1u : 0u);
          umma_commit(pv_done);
          if (np == n - 1) umma_commit(o_full);
          if (l_more && !load_v()) goto timeout;  // V(g + VS) into this stage
        }
      }
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int sp4 = warp & 3;
    const int row = sp4 * 32 + lane;
    const uint32_t lane_off = uint32_t(sp4 * 32) << 16;
    int g = 0, uc = 0;
    AttnSeg it;
    it.init(sc, blockIdx.x);
    int pair, kb0, kb1, slot;
    for (; it.next(pair, kb0, kb1, slot); ++uc) {
      const int qt = pair % sc.qtiles, h = pair / sc.qtiles;
      const int n = kb1 - kb0;
      float m = -INFINITY, l = 0.f;
      float cap_s[8];  // scaled scores of the captured key columns
#pragma unroll
      for (int q = 0; q < 8; ++q) cap_s[q] = -INFINITY;
      for (int j = 0; j < n; ++j, ++g) {
        if (!mbar_sleep_warp(s_full + 8 * (g & 1), (g >> 1) & 1, abort_flag)) goto timeout;
        tc_fence_after();
        uint32_t r[BKV];
#pragma unroll
        for (int i = 0; i < BKV / 16; ++i)
          tmem_ld16_nowait(tS0 + uint32_t(BKV) * uint32_t(g & 1) + lane_off + 16u * i, r + 16 * i);
        tmem_wait_ld();
        if (cap.n) {  // (warp-uniform) the captured columns that fall in this block
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (q < cap.n && cap.id[q] / BKV == kb0 + j)
              cap_s[q] = __uint_as_float(tmem_ld1_nowait(tS0 + uint32_t(BKV) * uint32_t(g & 1) +
                                                         lane_off + uint32_t(cap.id[q] % BKV))) *
                         scale_log2;
          tmem_wait_ld();
        }
        tc_fence_before();
        mbar_arrive(s_free + 8 * (g & 1));
        // raw scores: the running max m is kept in scaled base-2 units; the
        // scale (log2 e / sqrt(dh) > 0) commutes with the max, and
        // p = 2^(s * scale - m) is one FFMA + ex2 per element
        const int valid = Nk - (kb0 + j) * BKV;
        if (valid < BKV) {  // the last, partial key block (warp-uniform)
#pragma unroll
          for (int c = 0; c < BKV; ++c)
            if (c >= valid) r[c] = __float_as_uint(-INFINITY);
        }
        float mx8[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) mx8[q] = __uint_as_float(r[q]);
#pragma unroll
        for (int c = 8; c < BKV; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(r[c]));
        float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                         fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]))) * scale_log2;
        // lazy rescale (warp-uniform decision: the TMEM accesses are
        // warp-wide); O itself is rescaled below, once P V of the previous
        // block has completed
        bool rescale = false;
        float alpha = 1.f;
        if (j == 0) {
          m = mx;
        } else if (__any_sync(0xffffffffu, mx > m + LAZY_RESCALE)) {
          rescale = true;
          mx = fmaxf(mx, m);
          alpha = ex2_ftz(m - mx);
          l *= alpha;
          m = mx;
        }
        // p = 2^(s scale - m): the scaling FMA and the row sum run two
        // columns per instruction (packed f32x2)
        const uint64_t sc2 = f32x2(scale_log2, scale_log2), nm2 = f32x2(-m, -m);
        uint64_t sum2[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) sum2[q] = f32x2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < BKV; c += 2) {
          float a, b;
          unpack_f32x2(fma_f32x2(f32x2(__uint_as_float(r[c]), __uint_as_float(r[c + 1])), sc2, nm2),
                       a, b);
          a = ex2_ftz(a);
          b = ex2_ftz(b);
          r[c] = __float_as_uint(a);
          r[c + 1] = __float_as_uint(b);
          sum2[(c >> 1) & 3] = add_f32x2(sum2[(c >> 1) & 3], f32x2(a, b));
        }
        float s0, s1, s2, s3, s4, s5, s6, s7;
        unpack_f32x2(sum2[0], s0, s1);
        unpack_f32x2(sum2[1], s2, s3);
        unpack_f32x2(sum2[2], s4, s5);
        unpack_f32x2(sum2[3], s6, s7);
        l += ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
        // the P buffer and O are free once P V of the previous block is done
        if (g > 0 && !mbar_sleep_warp(pv_done, (g - 1) & 1, abort_flag)) goto timeout;
        tc_fence_after();
        if (rescale) {
#pragma unroll
          for (int i = 0; i < C::DHP / 16; ++i) {
            uint32_t o16[16];
            tmem_ld16_nowait(tO + lane_off + 16u * i, o16);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) o16[e] = __float_as_uint(__uint_as_float(o16[e]) * alpha);
            tmem_st16(tO + lane_off + 16u * i, o16);
          }
        }
        // P row (64 keys as 32 bf16 pairs): the A operand of P V
        const uint32_t tp = tP + lane_off;
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          uint32_t w[16];
#pragma unroll
          for (int c = 0; c < 16; ++c)
            w[c] = pack_bf16x2(__uint_as_float(r[32 * h2 + 2 * c]),
                               __uint_as_float(r[32 * h2 + 2 * c + 1]));
          tmem_st16(tp + 16u * h2, w);
        }
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(p_ready);
      }
      // ---- unit epilogue
      if (!mbar_sleep_warp(o_full, uc & 1, abort_flag)) goto timeout;
      tc_fence_after();
      uint32_t o[C::DHP];
#pragma unroll
      for (int i = 0; i < C::DHP / 16; ++i) tmem_ld16_nowait(tO + lane_off + 16u * i, o + 16 * i);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(o_free);
      if (slot < 0) {
        const TileLoc tl = locate_tile(rm, ai.n, D, qt);
        const int qrow = tl.row0 + row;
        if (cap.n && row < tl.rows) {
          const int tok = rm.tok ? __ldg(rm.tok + qrow) : qrow;
          const float inv_l = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (q < cap.n)
              atomicAdd(cap.out + size_t(tok) * cap.ldo + cap.id[q],
                        cap.w * ex2_ftz(cap_s[q] - m) * inv_l);
        }
        if (row < tl.rows) {
          const float inv = l > 0.f ? 1.f / l : 0.f;
          uint4* dst = reinterpret_cast<uint4*>(O + size_t(qrow) * ldo + h * DH);
#pragma unroll
          for (int c8 = 0; c8 < DH / 8; ++c8) {
            uint4 w;
            w.x = pack_bf16x2(__uint_as_float(o[8 * c8 + 0]) * inv, __uint_as_float(o[8 * c8 + 1]) * inv);
            w.y = pack_bf16x2(__uint_as_float(o[8 * c8 + 2]) * inv, __uint_as_float(o[8 * c8 + 3]) * inv);
            w.z = pack_bf16x2(__uint_as_float(o[8 * c8 + 4]) * inv, __uint_as_float(o[8 * c8 + 5]) * inv);
            w.w = pack_bf16x2(__uint_as_float(o[8 * c8 + 6]) * inv, __uint_as_float(o[8 * c8 + 7]) * inv);
            dst[c8] = w;
          }
        }
      } else {
        // a piece of the pair's keys: unnormalised O with its row max and
        // sum; the combine kernel merges the pieces
        // (the workspace slot's planes: column group c4 of every row, then
        // the rows' (max, sum); a warp's stores are whole 512-byte runs)
        float* mine = part + (size_t(blockIdx.x) * 2 + slot) * (BQ * PART_STRIDE);
#pragma unroll
        for (int c4 = 0; c4 < DH / 4; ++c4)
          __stcg(reinterpret_cast<float4*>(mine) + c4 * BQ + row,
                 make_float4(__uint_as_float(o[4 * c4]), __uint_as_float(o[4 * c4 + 1]),
                             __uint_as_float(o[4 * c4 + 2]), __uint_as_float(o[4 * c4 + 3])));
        __stcg(reinterpret_cast<float2*>(mine + DH * BQ) + row, make_float2(m, l));
      }
    }
  }
  goto done;
timeout:
  *abort_flag = 1;
  atomicOr(err, DEVERR_TIMEOUT);
done:
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ------------------------------------------------- short keys (text cross-attention)
// All Nk <= 128 keys of a (query tile, head) in one pass, one CTA per pair:
// S = Q K^T (M = 128, N = 128) in TMEM, an exact softmax per row (no running
// max, no rescaling), P (bf16) written over S, O = P V (N = DHP, 8 MMAs of 16
// keys, P read from TMEM as the A operand), O normalised and stored.  The
// text cross-attention of a block has 120 keys: the general kernel's two
// dependent 64-key rounds become one.
constexpr int XK = 128;  // keys per pass
template <int DH>
struct XCfg {
  using C = ACfg<DH>;
  static constexpr int K128 = XK * 128, K32 = C::TAIL ? XK * 32 : 0;
  static constexpr int V_ATOM = XK * 128;  // one MN-major SW128 atom of 64 head-dim columns
  static constexpr int V_BYTES = C::TAIL ? 2 * V_ATOM : V_ATOM;
  static constexpr int BYTES = C::Q_BYTES + K128 + K32 + V_BYTES;
  // rounded up so that at most two CTAs share an SM (2 x 256 TMEM columns)
  static constexpr size_t SMEM = 100 * 1024;
  static_assert(size_t(BYTES) + 1024 + 64 <= SMEM, "cross-attention tiles exceed the request");
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) |
                                      (uint32_t(XK >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
};

template <int DH, bool CAP>
__global__ void __launch_bounds__(128, 2)
xattn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQt,
                const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmKt,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnItems ai,
                int Nk, bf16* __restrict__ O, int ldo, int heads, RowMap rm, float scale_log2,
                unsigned* err, const __grid_constant__ AttnCapture cap) {
  using C = ACfg<DH>;
  using X = XCfg<DH>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + X::K128 + X::K32;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + X::V_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t load_bar = saddr(bars), mma_bar = saddr(bars + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(load_bar, 1);
    mbar_init(mma_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  if (warp == 0) tmem_alloc(saddr(tmem_slot), 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t tS = tmem_base, tO = tmem_base + XK;  // P is written over S

  pdl_wait();
  pdl_trigger();
  const int D = live_count(rm.count, rm.bound, err);
  const int qtiles = query_tiles(rm, ai.n, D);
  const int qt = int(blockIdx.x) / heads, h = int(blockIdx.x) - (int(blockIdx.x) / heads) * heads;
  bool ok = qt < qtiles;
  TileLoc tl{0, 0, 0};
  if (ok) tl = locate_tile(rm, ai.n, D, qt);
  const int row = warp * 32 + lane;
  const uint32_t lane_off = uint32_t(warp * 32) << 16;
  if (ok && threadIdx.x == 0) {
    // ---- loads: Q (128 rows of the tile), K and V (128 keys of the item)
    const int krow = ai.krow[tl.item], vrow = ai.vrow[tl.item];
    mbar_expect_tx(load_bar, X::BYTES);
    tma_load_3d(saddr(sQ), &tmQ, load_bar, 0, h, tl.row0);
    if (C::TAIL) tma_load_3d(saddr(sQ + C::Q128), &tmQt, load_bar, 64, h, tl.row0);
    tma_load_3d(saddr(sK), &tmK, load_bar, 0, h, krow);
    if (C::TAIL) tma_load_3d(saddr(sK + X::K128), &tmKt, load_bar, 64, h, krow);
    tma_load_3d(saddr(sV), &tmV, load_bar, 0, h, vrow);
    if (C::TAIL) tma_load_3d(saddr(sV + X::V_ATOM), &tmV, load_bar, 64, h, vrow);
    // ---- S = Q K^T over the 80 (72 + zero) head dims
    if (mbar_sleep(load_bar, 0, abort_flag)) {
      tc_fence_after();
      const uint64_t dq = sw128_desc(saddr(sQ)), dk = sw128_desc(saddr(sK));
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        umma_bf16(tS, dq + 2 * kk, dk + 2 * kk, X::IDESC_S, kk > 0 ? 1u : 0u);
      if (C::TAIL)
        umma_bf16(tS, sw32_kmajor_desc(saddr(sQ + C::Q128)), sw32_kmajor_desc(saddr(sK + X::K128)),
                  X::IDESC_S, 1u);
      umma_commit(mma_bar);
    } else {
      *abort_flag = 1;
    }
  }
  // ---- exact softmax of this thread's row
  if (ok) ok = mbar_sleep_warp(mma_bar, 0, abort_flag);
  float l = 0.f;
  if (ok) {
    tc_fence_after();
    uint32_t r[XK];
#pragma unroll
    for (int i = 0; i < XK / 16; ++i) tmem_ld16_nowait(tS + lane_off + 16u * i, r + 16 * i);
    tmem_wait_ld();
#pragma unroll
    for (int c = 0; c < XK; ++c)
      if (c >= Nk) r[c] = __float_as_uint(-INFINITY);
    float mx8[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) mx8[q] = __uint_as_float(r[q]);
#pragma unroll
    for (int c = 8; c < XK; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(r[c]));
    const float m = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                          fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]))) * scale_log2;
    const uint64_t sc2 = f32x2(scale_log2, scale_log2), nm2 = f32x2(-m, -m);
    uint64_t sum2[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) sum2[q] = f32x2(0.f, 0.f);
#pragma unroll
    for (int c = 0; c < XK; c += 2) {
      float a, b;
      unpack_f32x2(fma_f32x2(f32x2(__uint_as_float(r[c]), __uint_as_float(r[c + 1])), sc2, nm2),
                   a, b);
      a = ex2_ftz(a);
      b = ex2_ftz(b);
      r[c] = __float_as_uint(a);
      r[c + 1] = __float_as_uint(b);
      sum2[(c >> 1) & 3] = add_f32x2(sum2[(c >> 1) & 3], f32x2(a, b));
    }
    float s0, s1, s2, s3, s4, s5, s6, s7;
    unpack_f32x2(sum2[0], s0, s1);
    unpack_f32x2(sum2[1], s2, s3);
    unpack_f32x2(sum2[2], s4, s5);
    unpack_f32x2(sum2[3], s6, s7);
    l = ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
    if (CAP && cap.n && row < tl.rows) {  // the localisation scores of the listed keys
      const int qrow = tl.row0 + row;
      const int tok = rm.tok ? __ldg(rm.tok + qrow) : qrow;
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        if (q < cap.n) {
          float pq = 0.f;
#pragma unroll
          for (int c = 0; c < XK; ++c)
            if (c == cap.id[q]) pq = __uint_as_float(r[c]);
          atomicAdd(cap.out + size_t(tok) * cap.ldo + cap.id[q], cap.w * pq * inv_l);
        }
    }
    // P (bf16 pairs) over the first 64 columns of S: the A operand of P V
#pragma unroll
    for (int h2 = 0; h2 < XK / 32; ++h2) {
      uint32_t w[16];
#pragma unroll
      for (int c = 0; c < 16; ++c)
        w[c] = pack_bf16x2(__uint_as_float(r[32 * h2 + 2 * c]),
                           __uint_as_float(r[32 * h2 + 2 * c + 1]));
      tmem_st16(tS + lane_off + 16u * h2, w);
    }
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();  // every row's P is in TMEM
  if (ok && threadIdx.x == 0) {
    tc_fence_after();
    const uint64_t dv = C::TAIL ? sw128_mnmajor_desc_lbo(saddr(sV), X::V_ATOM)
                                : sw128_mnmajor_desc(saddr(sV));
#pragma unroll
    for (int kk = 0; kk < XK / 16; ++kk)
      umma_bf16_ta(tO, tS + 8 * kk, dv + 128 * kk, C::IDESC_PV, kk > 0 ? 1u : 0u);
    umma_commit(mma_bar);
  }
  if (ok) ok = mbar_sleep_warp(mma_bar, 1, abort_flag);
  if (ok) {
    tc_fence_after();
    uint32_t o[C::DHP];
#pragma unroll
    for (int i = 0; i < C::DHP / 16; ++i) tmem_ld16_nowait(tO + lane_off + 16u * i, o + 16 * i);
    tmem_wait_ld();
    if (row < tl.rows) {
      const float inv = l > 0.f ? 1.f / l : 0.f;
      uint4* dst = reinterpret_cast<uint4*>(O + size_t(tl.row0 + row) * ldo + h * DH);
#pragma unroll
      for (int c8 = 0; c8 < DH / 8; ++c8) {
        uint4 w;
        w.x = pack_bf16x2(__uint_as_float(o[8 * c8 + 0]) * inv, __uint_as_float(o[8 * c8 + 1]) * inv);
        w.y = pack_bf16x2(__uint_as_float(o[8 * c8 + 2]) * inv, __uint_as_float(o[8 * c8 + 3]) * inv);
        w.z = pack_bf16x2(__uint_as_float(o[8 * c8 + 4]) * inv, __uint_as_float(o[8 * c8 + 5]) * inv);
        w.w = pack_bf16x2(__uint_as_float(o[8 * c8 + 6]) * inv, __uint_as_float(o[8 * c8 + 7]) * inv);
        dst[c8] = w;
      }
    }
  }
  if (qt < qtiles && (!ok || *abort_flag)) {
    if (threadIdx.x == 0) atomicOr(err, DEVERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, 256);
  }
}

// ------------------------------------ cross-attention with the query folded in
// The text keys and W_xq are fixed for a turn, so the query projection can be
// folded into the keys once per turn: q'_h K_h^T = (xb W_xq,h^T + b_h) K_h^T =
// xb G_h^T + kb_h, G_h = K_h W_xq,h, kb_h = K_h b_h (a reassociation of the
// same products).  The cross-query GEMM then disappears from the block.

// G and kb of one (session, layer): block (h, 8-key group), thread = 9
// columns of G, 8 keys each, f32 accumulation over the head's dh dims.
constexpr int FOLD_KEYS = 8, FOLD_THREADS = 128, FOLD_COLS = 12;  // d <= 128 * 12
__global__ void __launch_bounds__(FOLD_THREADS)
xq_fold_kernel(const bf16* __restrict__ Kt, int ldk, const bf16* __restrict__ Wq,
               const float* __restrict__ bq, int M, int dh, int d, bf16* __restrict__ G,
               float* __restrict__ kb) {
  pdl_wait();
  pdl_trigger();
  __shared__ float sk[FOLD_KEYS][80];
  const int h = blockIdx.x, r0 = blockIdx.y * FOLD_KEYS;
  for (int e = threadIdx.x; e < FOLD_KEYS * dh; e += FOLD_THREADS) {
    const int r = e / dh, j = e - (e / dh) * dh;
    sk[r][j] = r0 + r < M ? __bfloat162float(Kt[size_t(r0 + r) * ldk + h * dh + j]) : 0.f;
  }
  __syncthreads();
  const int nc = d / FOLD_THREADS;
  float acc[FOLD_KEYS][FOLD_COLS];
#pragma unroll
  for (int r = 0; r < FOLD_KEYS; ++r)
#pragma unroll
    for (int i = 0; i < FOLD_COLS; ++i) acc[r][i] = 0.f;
  for (int j = 0; j < dh; ++j) {
    const bf16* wrow = Wq + size_t(h * dh + j) * d;
    float w[FOLD_COLS];
#pragma unroll
    for (int i = 0; i < FOLD_COLS; ++i)
      w[i] = i < nc ? __bfloat162float(wrow[threadIdx.x + FOLD_THREADS * i]) : 0.f;
#pragma unroll
    for (int r = 0; r < FOLD_KEYS; ++r)
#pragma unroll
      for (int i = 0; i < FOLD_COLS; ++i) acc[r][i] = fmaf(sk[r][j], w[i], acc[r][i]);
  }
#pragma unroll
  for (int r = 0; r < FOLD_KEYS; ++r) {
    if (r0 + r >= M) break;
    bf16* grow = G + (size_t(h) * XQ_KEYS + r0 + r) * d;
#pragma unroll
    for (int i = 0; i < FOLD_COLS; ++i)
      if (i < nc) grow[threadIdx.x + FOLD_THREADS * i] = __float2bfloat16_rn(acc[r][i]);
  }
  if (threadIdx.x < FOLD_KEYS && r0 + int(threadIdx.x) < M) {
    float a = 0.f;
    for (int j = 0; j < dh; ++j) a = fmaf(sk[threadIdx.x][j], bq[h * dh + j], a);
    kb[size_t(h) * XQ_KEYS + r0 + threadIdx.x] = a;
  }
}

// One (query tile, head) per CTA: S = xb_tile G_h^T accumulated over d in
// 64-column k-blocks (TMA ring, M = 128, N = 128), then the softmax of
// (S + kb) / sqrt(dh) per row, P over S in TMEM, O = P V, O / l stored.
// Two threads issue the S MMAs, the even k-blocks into S0 and the odd ones
// into S1 (TMEM columns 0 / 128; the softmax adds them): one thread issues
// a tcgen05.mma only about every 140 cycles from a ring whose stage is known
// at run time, and the 72 MMAs of the d = 1152 loop were bound by that.
constexpr int XF_STAGES = 6;
constexpr int XF_THREADS = 224;  // TMA, MMA, 4 softmax warps, second MMA warp
template <int DH>
struct XFCfg {
  using C = ACfg<DH>;
  static constexpr int STAGE_A = BQ * 128, STAGE_G = XK * 128;
  static constexpr int STAGE = STAGE_A + STAGE_G;
  static constexpr int V_ATOM = XK * 128;
  static constexpr int V_BYTES = C::TAIL ? 2 * V_ATOM : V_ATOM;
  static constexpr size_t SMEM =
      size_t(XF_STAGES) * STAGE + V_BYTES + XK * 4 + 1024 + 256;
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) |
                                      (uint32_t(XK >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
};

template <int DH, bool CAP>
__global__ void __launch_bounds__(XF_THREADS, 1)
xfused_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmG,
                 const __grid_constant__ CUtensorMap tmV, const float* __restrict__ kb,
                 const __grid_constant__ XqItems xi, int Nk, int d, bf16* __restrict__ O,
                 int ldo, int heads, RowMap rm, float scale_log2, unsigned* err,
                 const __grid_constant__ AttnCapture cap) {
  using C = ACfg<DH>;
  using X = XFCfg<DH>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sV = smem + XF_STAGES * X::STAGE;
  float* s_kb = reinterpret_cast<float*>(sV + X::V_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_kb + XK);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * XF_STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t full0 = saddr(bars), empty0 = saddr(bars + XF_STAGES);
  const uint32_t v_full = saddr(bars + 2 * XF_STAGES), s_full = v_full + 8, p_ready = v_full + 16,
                 o_full = v_full + 24, kb_ready = v_full + 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < XF_STAGES; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, 1);
    }
    mbar_init(v_full, 1);
    mbar_init(s_full, 2);  // both MMA threads commit their half of S
    mbar_init(p_ready, 128);
    mbar_init(o_full, 1);
    mbar_init(kb_ready, 128);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // Before the programmatic-dependency wait this kernel reads only what was
  // written two or more launches earlier (every kernel of the library waits
  // for its predecessor before letting its successor start): the live row
  // count and the turn's folded keys, key biases and text values.  Only the
  // bf16 rows of x come from the predecessor.
  const int D = live_count(rm.count, rm.bound, err);
  const int qtiles = query_tiles(rm, xi.n, D);
  const int qt = int(blockIdx.x) / heads, h = int(blockIdx.x) - (int(blockIdx.x) / heads) * heads;
  // the grid covers the bound of the query tiles: CTAs past the live ones
  // leave at once, before taking tensor memory
  if (qt >= qtiles) return;
  const bool live = true;
  const TileLoc tl = locate_tile(rm, xi.n, D, qt);
  // one CTA per SM (its shared memory), so all 512 columns are there
  if (warp == 1) tmem_alloc(saddr(tmem_slot), 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // S0 | S1 | O; P is written over S0
  const uint32_t tS = tmem_base, tS1 = tmem_base + XK, tO = tmem_base + 2 * XK;
  const int nkb = d / 64;
  bool ok = live;
  if (live && warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA
    // V and the folded keys of the first stages before the wait (each stage
    // barrier expects both halves of its bytes), the x rows after it
    const int grow = xi.grow[tl.item] + h * XK;
    mbar_expect_tx(v_full, X::V_BYTES);
    tma_load_3d(saddr(sV), &tmV, v_full, 0, h, xi.vrow[tl.item]);
    if (C::TAIL) tma_load_3d(saddr(sV + X::V_ATOM), &tmV, v_full, 64, h, xi.vrow[tl.item]);
    const int pre = nkb < XF_STAGES ? nkb : XF_STAGES;
    for (int k = 0; k < pre; ++k) {
      mbar_expect_tx(full0 + 8 * k, X::STAGE);
      tma_load_3d(saddr(smem + k * X::STAGE + X::STAGE_A), &tmG, full0 + 8 * k, 0, k, grow);
    }
    pdl_wait();
    pdl_trigger();
    for (int k = 0; k < nkb; ++k) {
      const int st = k % XF_STAGES;
      uint8_t* base = smem + st * X::STAGE;
      if (k >= pre) {
        if (!mbar_wait(empty0 + 8 * st, ((k / XF_STAGES) & 1) ^ 1, abort_flag)) {
          *abort_flag = 1;
          break;
        }
        mbar_expect_tx(full0 + 8 * st, X::STAGE);
        tma_load_3d(saddr(base + X::STAGE_A), &tmG, full0 + 8 * st, 0, k, grow);
      }
      tma_load_3d(saddr(base), &tmA, full0 + 8 * st, 0, k, tl.row0);
    }
  } else if (live && (warp == 1 || warp == 6) && lane == 0) {
    // ------------------------------------------------------------ MMA
    // warp 1: the even k-blocks into S0, then P V; warp 6: the odd ones into S1
    pdl_wait();
    const int par = warp == 1 ? 0 : 1;
    const uint32_t dS = par ? tS1 : tS;
    const uint64_t da = sw128_desc(saddr(smem)), dg = sw128_desc(saddr(smem + X::STAGE_A));
    bool good = true;
    for (int k = par; k < nkb && good; k += 2) {
      const int st = k % XF_STAGES;
      if (!mbar_wait(full0 + 8 * st, (k / XF_STAGES) & 1, abort_flag)) {
        good = false;
        break;
      }
      tc_fence_after();
      const uint64_t so = uint64_t((st * X::STAGE) >> 4);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        umma_bf16(dS, da + so + 2 * kk, dg + so + 2 * kk, X::IDESC_S,
                  (k > par || kk > 0) ? 1u : 0u);
      umma_commit(empty0 + 8 * st);
    }
    if (good) umma_commit(s_full);  // (arrives at once when this half has no k-block)
    if (par) {
      if (!good) *abort_flag = 1;
      goto xf_done;
    }
    // P V once every row's P is in TMEM and V has landed
    if (good && mbar_wait(p_ready, 0, abort_flag) && mbar_wait(v_full, 0, abort_flag)) {
      tc_fence_after();
      const uint64_t dv = C::TAIL ? sw128_mnmajor_desc_lbo(saddr(sV), X::V_ATOM)
                                  : sw128_mnmajor_desc(saddr(sV));
#pragma unroll
      for (int kk = 0; kk < XK / 16; ++kk)
        umma_bf16_ta(tO, tS + 8 * kk, dv + 128 * kk, C::IDESC_PV, kk > 0 ? 1u : 0u);
      umma_commit(o_full);
    } else {
      *abort_flag = 1;
    }
  } else if (live && warp >= 2 && warp < 6) {
    // ------------------------------------------------------------ softmax
    const int sp = warp & 3;
    const int row = sp * 32 + lane;
    const uint32_t lane_off = uint32_t(sp * 32) << 16;
    const int t128 = threadIdx.x - 64;  // 0 .. 127
    s_kb[t128] = t128 < Nk ? kb[size_t(xi.grow[tl.item]) + size_t(h) * XK + t128] : 0.f;
    pdl_wait();  // (before any global write: the predecessor reads O's buffer)
    mbar_arrive(kb_ready);
    ok = mbar_sleep_warp(kb_ready, 0, abort_flag) && mbar_sleep_warp(s_full, 0, abort_flag);
    float l = 0.f;
    if (ok) {
      tc_fence_after();
      uint32_t r[XK];
#pragma unroll
      for (int i = 0; i < XK / 16; ++i) tmem_ld16_nowait(tS + lane_off + 16u * i, r + 16 * i);
      tmem_wait_ld();
      if (nkb > 1) {  // S = S0 + S1 (the odd k-blocks)
#pragma unroll
        for (int j = 0; j < XK / 32; ++j) {
          uint32_t q[32];
          tmem_ld16_nowait(tS1 + lane_off + 32u * j, q);
          tmem_ld16_nowait(tS1 + lane_off + 32u * j + 16u, q + 16);
          tmem_wait_ld();
#pragma unroll
          for (int c = 0; c < 32; ++c)
            r[32 * j + c] = __float_as_uint(__uint_as_float(r[32 * j + c]) + __uint_as_float(q[c]));
        }
      }
#pragma unroll
      for (int c = 0; c < XK; ++c)
        r[c] = c < Nk ? __float_as_uint(__uint_as_float(r[c]) + s_kb[c])
                      : __float_as_uint(-INFINITY);
      float mx8[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) mx8[q] = __uint_as_float(r[q]);
#pragma unroll
      for (int c = 8; c < XK; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(r[c]));
      const float m = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                            fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]))) * scale_log2;
      const uint64_t sc2 = f32x2(scale_log2, scale_log2), nm2 = f32x2(-m, -m);
      uint64_t sum2[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) sum2[q] = f32x2(0.f, 0.f);
#pragma unroll
      for (int c = 0; c < XK; c += 2) {
        float a, b;
        unpack_f32x2(fma_f32x2(f32x2(__uint_as_float(r[c]), __uint_as_float(r[c + 1])), sc2, nm2),
                     a, b);
        a = ex2_ftz(a);
        b = ex2_ftz(b);
        r[c] = __float_as_uint(a);
        r[c + 1] = __float_as_uint(b);
        sum2[(c >> 1) & 3] = add_f32x2(sum2[(c >> 1) & 3], f32x2(a, b));
      }
      float s0, s1, s2, s3, s4, s5, s6, s7;
      unpack_f32x2(sum2[0], s0, s1);
      unpack_f32x2(sum2[1], s2, s3);
      unpack_f32x2(sum2[2], s4, s5);
      unpack_f32x2(sum2[3], s6, s7);
      l = ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
      if (CAP && cap.n && row < tl.rows) {  // the localisation scores of the listed keys
        const int qrow = tl.row0 + row;
        const int tok = rm.tok ? __ldg(rm.tok + qrow) : qrow;
        const float inv_l = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (q < cap.n) {
            float pq = 0.f;
#pragma unroll
            for (int c = 0; c < XK; ++c)
              if (c == cap.id[q]) pq = __uint_as_float(r[c]);
            atomicAdd(cap.out + size_t(tok) * cap.ldo + cap.id[q], cap.w * pq * inv_l);
          }
      }
#pragma unroll
      for (int h2 = 0; h2 < XK / 32; ++h2) {
        uint32_t w[16];
#pragma unroll
        for (int c = 0; c < 16; ++c)
          w[c] = pack_bf16x2(__uint_as_float(r[32 * h2 + 2 * c]),
                             __uint_as_float(r[32 * h2 + 2 * c + 1]));
        tmem_st16(tS + lane_off + 16u * h2, w);
      }
      tmem_wait_st();
    }
    tc_fence_before();
    mbar_arrive(p_ready);  // arrives even on failure so that no wait is left open
    if (ok) ok = mbar_sleep_warp(o_full, 0, abort_flag);
    if (ok) {
      tc_fence_after();
      uint32_t o[C::DHP];
#pragma unroll
      for (int i = 0; i < C::DHP / 16; ++i) tmem_ld16_nowait(tO + lane_off + 16u * i, o + 16 * i);
      tmem_wait_ld();
      if (row < tl.rows) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
        uint4* dst = reinterpret_cast<uint4*>(O + size_t(tl.row0 + row) * ldo + h * DH);
#pragma unroll
        for (int c8 = 0; c8 < DH / 8; ++c8) {
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(o[8 * c8 + 0]) * inv, __uint_as_float(o[8 * c8 + 1]) * inv);
          w.y = pack_bf16x2(__uint_as_float(o[8 * c8 + 2]) * inv, __uint_as_float(o[8 * c8 + 3]) * inv);
          w.z = pack_bf16x2(__uint_as_float(o[8 * c8 + 4]) * inv, __uint_as_float(o[8 * c8 + 5]) * inv);
          w.w = pack_bf16x2(__uint_as_float(o[8 * c8 + 6]) * inv, __uint_as_float(o[8 * c8 + 7]) * inv);
          dst[c8] = w;
        }
      }
    }
  }
xf_done:
  if (live && (!ok || *abort_flag) && threadIdx.x == 64) atomicOr(err, DEVERR_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

// Merge of the pieces of the pairs that stream-K cut.  The pieces of a pair
// come from CTAs cta_of(first block) .. cta_of(last block); a CTA's piece is
// its first (slot 0) when its range starts inside the pair, else its last
// (slot 1).  A workspace slot holds its piece as DH / 4 planes of 128 float4
// (head-dim columns 4 c .. 4 c + 3 of the tile's rows), then the rows' (max,
// sum) pairs, so that the attention kernel's softmax threads (one row each)
// and this kernel's lanes (one row each) access whole 512-byte runs.  A work
// unit is 32 consecutive rows of one cut pair and COMBINE_CH of the column
// planes; units go to warps in turn.  Per row: the largest of the pieces'
// maxima M, then the pieces' columns weighted by 2^(m_q - M), over the
// weighted sums, stored as bf16.  Each of the two passes keeps several
// pieces' loads in flight.
constexpr int COMBINE_THREADS = 256, COMBINE_CH = 3;
template <int DH>
__global__ void __launch_bounds__(COMBINE_THREADS, 2)
attn_combine_kernel(const float* __restrict__ part, bf16* __restrict__ O, int ldo, int heads,
                    RowMap rm, int n_items, int Nk, int attn_grid, unsigned* err) {
  // the row count predates the attention launch (see attn_tc_kernel): read
  // before the wait; the pieces come from the predecessor
  const int D = live_count(rm.count, rm.bound, err);
  AttnSched sc;
  sc.init(query_tiles(rm, n_items, D), heads, Nk, attn_grid);
  pdl_wait();
  pdl_trigger();
  if (!sc.streamk) return;
  constexpr int C4 = DH / 4, NCH = (C4 + COMBINE_CH - 1) / COMBINE_CH;
  constexpr int PER_PAIR = (BQ / 32) * NCH;  // units of one pair
  const int lane = threadIdx.x & 31;
  const int units = sc.pairs * PER_PAIR;
  const int nwarps = int(gridDim.x) * (COMBINE_THREADS / 32);
  for (int u = int(blockIdx.x) * (COMBINE_THREADS / 32) + (int(threadIdx.x) >> 5); u < units;
       u += nwarps) {
    const int pair = u / PER_PAIR, rest = u - pair * PER_PAIR;
    const int row = (rest / NCH) * 32 + lane, c0 = (rest - (rest / NCH) * NCH) * COMBINE_CH;
    const int lo = pair * sc.nkb;
    const int c_lo = sc.cta_of(lo);
    const int np = sc.cta_of(lo + sc.nkb - 1) - c_lo + 1;
    if (np == 1) continue;  // one CTA held the whole pair (warp-uniform)
    const int slot_lo = sc.bound(c_lo) == lo ? 0 : 1;
    const TileLoc tl = locate_tile(rm, n_items, D, pair % sc.qtiles);
    const int h = pair / sc.qtiles;
    auto slot = [&](int q) {
      return part + (size_t(c_lo + q) * 2 + (q == 0 ? slot_lo : 0)) * (BQ * PART_STRIDE);
    };
    float M = -INFINITY;
#pragma unroll 8
    for (int q = 0; q < np; ++q)
      M = fmaxf(M, __ldcg(reinterpret_cast<const float2*>(slot(q) + DH * BQ) + row).x);
    float L = 0.f;
    float4 acc[COMBINE_CH];
#pragma unroll
    for (int c = 0; c < COMBINE_CH; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int q = 0; q < np; ++q) {
      const float* b = slot(q);
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(b + DH * BQ) + row);
      float4 v[COMBINE_CH];
#pragma unroll
      for (int c = 0; c < COMBINE_CH; ++c)
        if (c0 + c < C4) v[c] = __ldcg(reinterpret_cast<const float4*>(b) + (c0 + c) * BQ + row);
      const float wq = ex2_ftz(ml.x - M);
      L += wq * ml.y;
#pragma unroll
      for (int c = 0; c < COMBINE_CH; ++c)
        if (c0 + c < C4) {
          acc[c].x += wq * v[c].x;
          acc[c].y += wq * v[c].y;
          acc[c].z += wq * v[c].z;
          acc[c].w += wq * v[c].w;
        }
    }
    if (row < tl.rows) {
      const float inv = L > 0.f ? 1.f / L : 0.f;
      uint2* dst = reinterpret_cast<uint2*>(O + size_t(tl.row0 + row) * ldo + h * DH) + c0;
#pragma unroll
      for (int c = 0; c < COMBINE_CH; ++c)
        if (c0 + c < C4)
          dst[c] = make_uint2(pack_bf16x2(acc[c].x * inv, acc[c].y * inv),
                              pack_bf16x2(acc[c].z * inv, acc[c].w * inv));
    }
  }
}

// ------------------------------------------------------------------- host
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

struct HeadMapKey {
  const void* p;
  int rows, ld, heads, dh;
  bool operator==(const HeadMapKey& o) const {
    return p == o.p && rows == o.rows && ld == o.ld && heads == o.heads && dh == o.dh;
  }
};
struct HeadMapHash {
  size_t operator()(const HeadMapKey& k) const {
    return std::hash<const void*>()(k.p) ^ (size_t(k.rows) * 1000003u) ^ (size_t(k.ld) * 7919u) ^
           (size_t(k.heads) * 131u) ^ size_t(k.dh);
  }
};

// (head_dim, head, row) view of a row-major [rows][ld] bf16 matrix whose row
// holds `heads` blocks of dh; boxes of box_w x 1 x box_rows (box_w 64 with the
// 128-byte swizzle, 16 with the 32-byte swizzle); reads outside the view
// (head_dim >= dh, row >= rows) return zero.
cudaError_t head_map(const bf16* p, int rows, int ld, int heads, int dh, int box_w, int box_rows,
                     CUtensorMap* out) {
  static std::mutex mu;
  static std::unordered_map<HeadMapKey, CUtensorMap, HeadMapHash> cache;
  HeadMapKey key{p, rows, ld, heads, (dh * 1024 + box_rows) * 256 + box_w};
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *out = it->second;
      return cudaSuccess;
    }
  }
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  cuuint64_t dims[3] = {cuuint64_t(dh), cuuint64_t(heads), cuuint64_t(rows)};
  cuuint64_t strides[2] = {cuuint64_t(dh) * sizeof(bf16), cuuint64_t(ld) * sizeof(bf16)};
  cuuint32_t box[3] = {cuuint32_t(box_w), 1, cuuint32_t(box_rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<bf16*>(p), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  box_w == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_32B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, *out);
  return cudaSuccess;
}

int device_sms_attn() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (!sms[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaFuncSetAttribute(attn_tc_kernel<72>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(ACfg<72>::SMEM)) != cudaSuccess ||
        cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(ACfg<64>::SMEM)) != cudaSuccess ||
        cudaFuncSetAttribute(xattn_tc_kernel<72, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XCfg<72>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xattn_tc_kernel<72, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XCfg<72>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xattn_tc_kernel<64, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XCfg<64>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xattn_tc_kernel<64, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XCfg<64>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xfused_tc_kernel<72, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XFCfg<72>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xfused_tc_kernel<72, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XFCfg<72>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xfused_tc_kernel<64, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XFCfg<64>::SMEM)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(xfused_tc_kernel<64, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(XFCfg<64>::SMEM)) !=
            cudaSuccess)
      return 0;
    sms[dev] = v;
  }
  return sms[dev];
}

}  // namespace

size_t attention_split_floats(int Nmax, int heads, int dh) {
  (void)Nmax;
  (void)heads;
  (void)dh;
  const int sms = device_sms_attn();
  return size_t(8) * (sms > 0 ? sms : 160) * BQ * PART_STRIDE;
}


cudaError_t launch_attention(const bf16* Q, int ldq, const bf16* K, const bf16* V, int ldkv,
                             int kv_rows, const AttnItems& ai, int Nk, bf16* O, int ldo, int heads,
                             int dh, const RowMap& rm, unsigned* err, const AttnScratch& as,
                             cudaStream_t st, const AttnCapture* capture) {
  if (rm.bound <= 0) return cudaSuccess;
  if (dh != 72 && dh != 64) return cudaErrorInvalidValue;
  if (ai.n < 1 || ai.n > MAX_ITEMS || (ai.n > 1 && !rm.meta)) return cudaErrorInvalidValue;
  for (int i = 0; i < ai.n; ++i)
    if (ai.krow[i] < 0 || ai.vrow[i] < 0 || ai.krow[i] > kv_rows - Nk || ai.vrow[i] > kv_rows - Nk)
      return cudaErrorInvalidValue;
  const int sms = device_sms_attn();
  if (!sms) return cudaErrorInvalidDevice;
  // a 64-wide 128B-swizzled map and a 16-wide 32B-swizzled tail map per operand
  CUtensorMap tq, tqt, tk, tkt, tv;
  RC_TRY(head_map(Q, rm.bound, ldq, heads, dh, 64, BQ, &tq));
  RC_TRY(head_map(K, kv_rows, ldkv, heads, dh, 64, BKV, &tk));
  RC_TRY(head_map(V, kv_rows, ldkv, heads, dh, 64, BKV, &tv));
  RC_TRY(head_map(Q, rm.bound, ldq, heads, dh, 16, BQ, &tqt));
  RC_TRY(head_map(K, kv_rows, ldkv, heads, dh, 16, BKV, &tkt));
  const float scale_log2 = float(1.4426950408889634 / sqrt(double(dh)));
  AttnCapture cap{};
  if (capture && capture->n > 0) {
    // every key must sit in the one unit of its (query tile, head)
    if (capture->n > 8 || !capture->out || (Nk + BKV - 1) / BKV >= 2 * MIN_KB_PER_SPLIT)
      return cudaErrorInvalidValue;
    for (int q = 0; q < capture->n; ++q)
      if (capture->id[q] < 0 || capture->id[q] >= Nk || capture->id[q] >= capture->ldo)
        return cudaErrorInvalidValue;
    cap = *capture;
  }
  if (Nk <= XK) {
    // short key sets (the text cross-attention): one pass per (query tile,
    // head), a CTA each; tiles beyond the live count exit at once
    CUtensorMap xk, xkt, xv;
    RC_TRY(head_map(K, kv_rows, ldkv, heads, dh, 64, XK, &xk));
    RC_TRY(head_map(K, kv_rows, ldkv, heads, dh, 16, XK, &xkt));
    RC_TRY(head_map(V, kv_rows, ldkv, heads, dh, 64, XK, &xv));
    const long long xgrid = ((long long)(rm.bound + BQ - 1) / BQ + ai.n - 1) * heads;
    if (xgrid >= (1ll << 31)) return cudaErrorInvalidValue;
    auto xk_fn = dh == 72 ? (cap.n ? xattn_tc_kernel<72, true> : xattn_tc_kernel<72, false>)
                          : (cap.n ? xattn_tc_kernel<64, true> : xattn_tc_kernel<64, false>);
    RC_TRY(launch_k(xk_fn, dim3(unsigned(xgrid)), dim3(128),
                    dh == 72 ? XCfg<72>::SMEM : XCfg<64>::SMEM, st, tq, tqt, xk, xkt, xv, ai, Nk,
                    O, ldo, heads, rm, scale_log2, err, cap));
    count_launches(1);
    return cudaSuccess;
  }
  const int grid = CTAS_PER_SM * sms;
  {
    const unsigned long long tiles = (rm.bound + BQ - 1) / BQ + ai.n - 1;
    if (tiles * heads * ((Nk + BKV - 1) / BKV) * grid >= (1ull << 32)) return cudaErrorInvalidValue;
  }
  // two partial pieces per CTA at most
  if (as.part_floats < size_t(2) * grid * BQ * PART_STRIDE) return cudaErrorInvalidValue;
  if (dh == 72)
    RC_TRY(launch_k(attn_tc_kernel<72>, dim3(grid), dim3(THREADS), ACfg<72>::SMEM, st, tq, tqt,
                    tk, tkt, tv, ai, Nk, O, ldo, heads, rm, scale_log2, err, as.part, cap));
  else
    RC_TRY(launch_k(attn_tc_kernel<64>, dim3(grid), dim3(THREADS), ACfg<64>::SMEM, st, tq, tqt,
                    tk, tkt, tv, ai, Nk, O, ldo, heads, rm, scale_log2, err, as.part, cap));
  count_launches(1);
  // stream-K (and so partial pieces) only with at least 2 MIN_KB_PER_SPLIT key blocks
  if ((Nk + BKV - 1) / BKV >= 2 * MIN_KB_PER_SPLIT) {
    const int tiles = (rm.bound + BQ - 1) / BQ + ai.n - 1;  // bound of the query tiles
    // units of 32 rows and COMBINE_CH column planes of a pair
    const int units = tiles * heads * (BQ / 32) * ((dh / 4 + COMBINE_CH - 1) / COMBINE_CH);
    const int cgrid = min((units + COMBINE_THREADS / 32 - 1) / (COMBINE_THREADS / 32), 2 * sms);
    if (dh == 72)
      RC_TRY(launch_k(attn_combine_kernel<72>, dim3(cgrid), dim3(COMBINE_THREADS), 0, st,
                      as.part, O, ldo, heads, rm, ai.n, Nk, grid, err));
    else
      RC_TRY(launch_k(attn_combine_kernel<64>, dim3(cgrid), dim3(COMBINE_THREADS), 0, st,
                      as.part, O, ldo, heads, rm, ai.n, Nk, grid, err));
    count_launches(1);
  }
  return cudaSuccess;
}

cudaError_t launch_xq_fold(const bf16* Kt, int ldk, const bf16* Wq, const float* bq, int M,
                           int heads, int dh, int d, bf16* G, float* kb, cudaStream_t st) {
  if (M < 1 || M > XQ_KEYS || dh > 80 || d % FOLD_THREADS || d > FOLD_THREADS * FOLD_COLS)
    return cudaErrorInvalidValue;
  RC_TRY(launch_k(xq_fold_kernel, dim3(heads, (M + FOLD_KEYS - 1) / FOLD_KEYS),
                  dim3(FOLD_THREADS), 0, st, Kt, ldk, Wq, bq, M, dh, d, G, kb));
  count_launches(1);
  return cudaSuccess;
}

cudaError_t launch_xattn_fused(const bf16* xb, int ldx, const bf16* G, const float* kb, int g_rows,
                               const bf16* V, int ldv, int v_rows, const XqItems& xi, int Nk,
                               bf16* O, int ldo, int heads, int dh, const RowMap& rm,
                               unsigned* err, cudaStream_t st, const AttnCapture* capture) {
  if (rm.bound <= 0) return cudaSuccess;
  const int d = heads * dh;
  if ((dh != 72 && dh != 64) || Nk < 1 || Nk > XK || d % 64 || ldx % 8 || ldv % 8)
    return cudaErrorInvalidValue;
  if (xi.n < 1 || xi.n > MAX_ITEMS || (xi.n > 1 && !rm.meta)) return cudaErrorInvalidValue;
  for (int i = 0; i < xi.n; ++i)
    if (xi.grow[i] < 0 || xi.grow[i] + heads * XK > g_rows || xi.vrow[i] < 0 ||
        xi.vrow[i] > v_rows - Nk)
      return cudaErrorInvalidValue;
  if (!device_sms_attn()) return cudaErrorInvalidDevice;
  AttnCapture cap{};
  if (capture && capture->n > 0) {
    if (capture->n > 8 || !capture->out) return cudaErrorInvalidValue;
    for (int q = 0; q < capture->n; ++q)
      if (capture->id[q] < 0 || capture->id[q] >= Nk || capture->id[q] >= capture->ldo)
        return cudaErrorInvalidValue;
    cap = *capture;
  }
  // xb and G as (64 columns, column block, row) views, V as the head view
  CUtensorMap ta, tg, tv;
  RC_TRY(head_map(xb, rm.bound, ldx, d / 64, 64, 64, BQ, &ta));
  RC_TRY(head_map(G, g_rows, d, d / 64, 64, 64, XK, &tg));
  RC_TRY(head_map(V, v_rows, ldv, heads, dh, 64, XK, &tv));
  const float scale_log2 = float(1.4426950408889634 / sqrt(double(dh)));
  const long long grid = ((long long)(rm.bound + BQ - 1) / BQ + xi.n - 1) * heads;
  if (grid >= (1ll << 31)) return cudaErrorInvalidValue;
  auto fn = dh == 72 ? (cap.n ? xfused_tc_kernel<72, true> : xfused_tc_kernel<72, false>)
                     : (cap.n ? xfused_tc_kernel<64, true> : xfused_tc_kernel<64, false>);
  RC_TRY(launch_k(fn, dim3(unsigned(grid)), dim3(XF_THREADS), dh == 72 ? XFCfg<72>::SMEM : XFCfg<64>::SMEM,
                  st, ta, tg, tv, kb, xi, Nk, d, O, ldo, heads, rm, scale_log2, err, cap));
  count_launches(1);
  return cudaSuccess;
}

}  // namespace rc
