// Tensor-core GEMM of the region-sparse block on sm_103a: tcgen05.mma with
// TMEM accumulators, operands staged by TMA (128-byte swizzle), persistent
// warp-specialised CTAs, and the block's epilogues fused (bias, tanh-GELU,
// gated residual, QKV with K/V rows written straight into the cache rows of
// the dirty tokens -- Section 3.4, Kernel Fusing -- and the merged hidden
// state written into the cache's H rows).
//
// C[M][n] = A[M][k] W[n][k]^T, A and W K-major bf16, f32 accumulation.
// M (the dirty-token count) may live on the device: every CTA reads it and
// derives the same schedule.  The tile is 128 x BN with BN in {64, 128, 192,
// 256}, chosen per launch from M by a cost model (the main loop streams
// (128 + BN) x 64 bf16 operands per k-block from L2 at a fixed per-SM rate,
// and only the last tile's epilogue is exposed), so that ragged row counts
// still spread over the GPU.  Whole tiles go out in waves.  The gated
// residual (x += gate (C + b)) is written as vector reductions into x, so
// pieces of a tile simply add up: for it a small last wave is instead cut
// into equal k-block ranges (stream-K).  Its casting variant (x += ..., then
// xb = bf16(x), read-modify-write) and the other epilogues see whole tiles.
//
// CTA = 16 warps: warp 0 issues TMA loads (A), warp 14 those of W, warp 1
// owns TMEM and issues the MMAs (one thread), warps 2..13 drain the
// accumulator (one TMEM lane = one output row per thread; three warps per
// TMEM lane quarter take every third 32-column chunk; re-staged through
// shared memory so that global writes are whole row pieces), and warp 15
// is a second MMA issuer when every CTA holds one work item (the item's odd
// k-blocks into the second accumulator, see split2).  The epilogue is
// latency-bound (a CTA holds one tile at small row counts), so its width is
// worth more than a deeper ring.  Otherwise two TMEM accumulators of up to
// 256 columns let the epilogue of one tile overlap the main loop of the next.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace rc {

namespace {

using namespace rc::tc;

constexpr int BM = 128, BK = 64;
// TMA warp (A, or A and W for CTA pairs), MMA warp, 12 epilogue warps, a
// second TMA warp that loads W for unpaired CTAs (each TMA request takes long
// enough to issue that one thread issuing both operands bounds the main
// loop), and a second MMA warp
constexpr int THREADS = 512;
constexpr int W_WARP = 14;
constexpr int MMA2_WARP = 15;
constexpr int STAGE_A = BM * BK * 2;   // bytes
constexpr int MIN_KB_PER_CTA = 4;
constexpr int STAGING_WARP = 32 * 128;  // epilogue staging: 32 rows of 128 B per warp
constexpr int STAGING_BYTES = 12 * STAGING_WARP;

// Operand ring: stages of A (16 KB) + B (BN x 128 B), as many as fit.
constexpr int RING_BYTES = 168 * 1024;
constexpr int MAX_STAGES = 9;
constexpr int TMEM_COLS = 512;  // two accumulators of up to 256 columns
// per-tile column vectors of the epilogue: bias and gate of up to 256 columns
constexpr int VEC_BYTES = 2 * 256 * 4;
constexpr size_t SMEM_BYTES = size_t(RING_BYTES) + STAGING_BYTES + VEC_BYTES + 1024 + 256;
// Instruction descriptor, kind::f16: D f32, A and B bf16, both K-major,
// M >> 4 at bit 24; N >> 3 goes to bit 17 at run time.
constexpr uint32_t IDESC_BASE = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(BM >> 4) << 24);
// the same for the M = 256 MMA of a CTA pair
constexpr uint32_t IDESC_PAIR = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(256 >> 4) << 24);
// The tile width and split chosen on the host for 1 .. BN_TABLE row tiles
// (BN / 64 + 8 S), passed by value; larger row counts choose on the device.
constexpr int BN_TABLE = 64;
struct BnTable {
  uint8_t w64[BN_TABLE];
};
// W tensor maps by box height 32, 64, 96, 128, 192, 256 rows (a CTA of a
// pair loads half a tile width)
constexpr int N_BMAPS = 6;
struct BMaps {
  CUtensorMap m[N_BMAPS];
};
__host__ __device__ constexpr int bmap_index(int rows) {
  return rows == 32 ? 0 : rows == 64 ? 1 : rows == 96 ? 2 : rows == 128 ? 3 : rows == 192 ? 4 : 5;
}

// ---------------------------------------------------------------- epilogue
__device__ __forceinline__ void load32(const float* p, float* v) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    float4 a = __ldg(reinterpret_cast<const float4*>(p) + i);
    v[4 * i] = a.x; v[4 * i + 1] = a.y; v[4 * i + 2] = a.z; v[4 * i + 3] = a.w;
  }
}
__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c),
               "f"(d)
               : "memory");
}

// The mode a schedule is planned for: a gated residual held to whole tiles
// plans like any other 4-byte epilogue whose tiles are not split.
__host__ __device__ inline int sched_mode(const GemmEpi& ep) {
  return ep.mode == EPI_GATE_RES && ep.whole_tiles ? int(EPI_F32) : ep.mode;
}

__device__ __forceinline__ bool gated(const GemmEpi& ep) {
  return (ep.mode == EPI_GATE_RES || ep.mode == EPI_GATE_RES_CAST) && ep.gate_tab;
}
// The gate's per-item part comes with each row (from its item's timestep
// vector) only when the launch has several items; with one item it is
// folded into the staged gate vector.
__device__ __forceinline__ bool row_gate(const GemmEpi& ep) {
  return gated(ep) && ep.gate_off >= 0 && ep.its.n > 1;
}

// The column vectors of one tile (columns col0 .. col0 + BN - 1) in shared
// memory, written by the 384 epilogue threads before the accumulator is
// ready: sv[c] = bias (0 when absent, or when this piece of a split gated
// residual does not start at k = 0: the update is a sum over pieces, so the
// bias goes with one of them), sv[256 + c] = gate (table part, plus the
// item's timestep part when the launch has one item).
__device__ __forceinline__ void stage_vectors(const GemmEpi& ep, int col0, int BN, bool with_bias,
                                              float* sv, int etid) {
  const float* tb0 = (ep.its.n == 1 && ep.gate_off >= 0) ? ep.its.tb[0] : nullptr;
  for (int c = etid; c < BN; c += 384) {
    const int col = col0 + c;
    sv[c] = (ep.bias && with_bias) ? __ldg(ep.bias + col) : 0.f;
    if (gated(ep)) sv[256 + c] = __ldg(ep.gate_tab + col) + (tb0 ? __ldg(tb0 + ep.gate_off + col) : 0.f);
  }
}

// Epilogue values of columns c0 .. c0+31 of one output row (cl = c0 within
// the tile): bias, tanh-GELU, gate, from the staged vectors (plus the row's
// item gate when the launch has several items).
__device__ __forceinline__ void epilogue_values(const GemmEpi& ep, int c0, int cl, int item,
                                                float* v, const float* sv) {
  const float4* b4 = reinterpret_cast<const float4*>(sv + cl);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 b = b4[i];
    v[4 * i] += b.x; v[4 * i + 1] += b.y; v[4 * i + 2] += b.z; v[4 * i + 3] += b.w;
  }
  if (ep.mode == EPI_GELU_BF16) {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = gelu_tanh(v[i]);
  } else if (gated(ep)) {
    float g[32];
    const float4* g4 = reinterpret_cast<const float4*>(sv + 256 + cl);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 a = g4[i];
      g[4 * i] = a.x; g[4 * i + 1] = a.y; g[4 * i + 2] = a.z; g[4 * i + 3] = a.w;
    }
    if (row_gate(ep)) {
      const float* tb = ep.its.tb[item];
      if (tb) {
        float g2[32];
        load32(tb + ep.gate_off + c0, g2);
#pragma unroll
        for (int i = 0; i < 32; ++i) g[i] += g2[i];
      }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] *= g[i];
  }
}

// 32 consecutive f32 columns of this thread's TMEM lane, summed over the two
// accumulators at taddr and taddr + 256 (a tile whose k-blocks two MMA
// threads split between them).
__device__ __forceinline__ void tmem_ld32_sum2(uint32_t taddr, float* v) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t a[16], b[16];
    tmem_ld16_nowait(taddr + uint32_t(16 * h), a);
    tmem_ld16_nowait(taddr + 256u + uint32_t(16 * h), b);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 16; ++i) v[16 * h + i] = __uint_as_float(a[i]) + __uint_as_float(b[i]);
  }
}
// The k-blocks of parity `par` of a CTA's one work item (k-blocks [kb0, kb1),
// ring stages from 0), issued by one of two MMA threads into accumulator
// `par` (TMEM columns 256 par ..); its tfull barrier is committed at the end.
// Returns false when a bounded wait gave up.
__device__ __forceinline__ bool mma_half(int par, int kb0, int kb1, int STAGES, int STAGE,
                                         uint32_t ring, uint32_t tmem_base, uint32_t idesc,
                                         uint32_t full0, uint32_t empty0, uint32_t tfull0,
                                         uint32_t tempty0, volatile int* abort_flag) {
  if (!mbar_wait(tempty0 + 8 * par, 1, abort_flag)) return false;
  tc_fence_after();
  const uint64_t da = sw128_desc(ring), db = sw128_desc(ring + STAGE_A);
  const uint32_t dtm = tmem_base + uint32_t(par * 256);
  int stage = par;
  uint32_t phase = 0;
  for (int kb = kb0 + par; kb < kb1; kb += 2) {
    if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) return false;
    tc_fence_after();
    const uint64_t so = uint64_t((stage * STAGE) >> 4);
#pragma unroll
    for (int kk = 0; kk < BK / 16; ++kk)
      umma_bf16(dtm, da + so + 2 * kk, db + so + 2 * kk, idesc,
                (kb > kb0 + par || kk > 0) ? 1u : 0u);
    umma_commit(empty0 + 8 * stage);
    stage += 2;
    if (stage >= STAGES) {
      stage -= STAGES;
      phase ^= 1;
    }
  }
  umma_commit(tfull0 + 8 * par);
  return true;
}

// Named barrier of the 12 epilogue warps.
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, 384;" ::: "memory"); }

// Destination of columns c0 .. c0+31 of output row r, or null when the row is
// beyond the live count (or its token / item index is bad: QKV raises
// DEVERR_INDEX).  tok / item of the row are loaded once per tile.
__device__ __forceinline__ char* chunk_dst(const GemmEpi& ep, int r, int M, int tok, int item,
                                           int c0) {
  if (r >= M) return nullptr;
  switch (ep.mode) {
    case EPI_F32:
      return reinterpret_cast<char*>(ep.out_f + size_t(r) * ep.ld_out + c0);
    case EPI_GATE_RES:
    case EPI_GATE_RES_CAST:
      return reinterpret_cast<char*>(ep.xf + size_t(r) * ep.ld_xf + c0);
    case EPI_QKV: {
      const int part = c0 / ep.dsplit;
      const int cc = c0 - part * ep.dsplit;
      if (part == 0) return reinterpret_cast<char*>(ep.out_bf + size_t(r) * ep.ld_out + cc);
      if (tok < 0 || tok >= ep.n_tokens || item < 0 || item >= ep.its.n) {
        atomicOr(ep.err, DEVERR_INDEX);
        return nullptr;
      }
      return reinterpret_cast<char*>(ep.its.slice[item] + (part == 1 ? ep.k_off : ep.v_off) +
                                     size_t(tok) * ep.dsplit + cc);
    }
    default:
      return reinterpret_cast<char*>(ep.out_bf + size_t(r) * ep.ld_out + c0);
  }
}

// Writes one warp's 32 x 32 chunk (lane = row, v = its 32 columns) to global
// memory with coalesced accesses: each lane parks its row in the warp's 4 KB
// staging area, then groups of lanes write whole 128-byte (f32) or 64-byte
// (bf16) row pieces.  Staging is XOR-swizzled in 16-byte units so that both
// the row-per-lane writes and the piece-per-lane-group reads are free of bank
// conflicts.  The gated residual goes out as vector reductions (x += value);
// its casting variant reads x, adds, and writes x and bf16(x) (xb_row: the
// row's bf16 copy, columns c0 ..).
__device__ __forceinline__ void store_chunk(int mode, uint8_t* stg, int lane, const float* v,
                                            char* dst, bf16* xb_row) {
  const uint32_t s0 = saddr(stg);
  if (mode == EPI_F32 || mode == EPI_GATE_RES || mode == EPI_GATE_RES_CAST) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(
                       s0 + lane * 128 + 16 * (j ^ (lane & 7))),
                   "f"(v[4 * j]), "f"(v[4 * j + 1]), "f"(v[4 * j + 2]), "f"(v[4 * j + 3])
                   : "memory");
    __syncwarp();
    // all row pointers and pieces first (independent, so they overlap),
    // then the global writes
    const int j = lane & 7;
    char* d[8];
    bf16* xb[8];
    float4 x[8];
#pragma unroll
    for (int pass = 0; pass < 8; ++pass) {
      const int row = pass * 4 + (lane >> 3);
      d[pass] = reinterpret_cast<char*>(
          __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(dst), row));
      xb[pass] = mode == EPI_GATE_RES_CAST
                     ? reinterpret_cast<bf16*>(__shfl_sync(
                           0xffffffffu, reinterpret_cast<unsigned long long>(xb_row), row))
                     : nullptr;
      x[pass] = *reinterpret_cast<const float4*>(stg + row * 128 + 16 * (j ^ (row & 7)));
    }
    if (mode == EPI_GATE_RES_CAST) {
      // read-modify-write: all eight reads in flight before the writes
      float4 o[8];
#pragma unroll
      for (int pass = 0; pass < 8; ++pass)
        o[pass] = d[pass] ? __ldcg(reinterpret_cast<const float4*>(d[pass]) + j)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int pass = 0; pass < 8; ++pass) {
        if (!d[pass]) continue;
        float4 y = x[pass];
        y.x += o[pass].x; y.y += o[pass].y; y.z += o[pass].z; y.w += o[pass].w;
        reinterpret_cast<float4*>(d[pass])[j] = y;
        if (xb[pass])
          *reinterpret_cast<uint2*>(xb[pass] + 4 * j) =
              make_uint2(pack_bf16x2(y.x, y.y), pack_bf16x2(y.z, y.w));
      }
    } else {
#pragma unroll
      for (int pass = 0; pass < 8; ++pass) {
        if (!d[pass]) continue;
        float* q = reinterpret_cast<float*>(d[pass]) + 4 * j;
        const float4 y = x[pass];
        if (mode == EPI_GATE_RES)
          red_add_v4(q, y.x, y.y, y.z, y.w);
        else
          *reinterpret_cast<float4*>(q) = y;
      }
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                       s0 + lane * 64 + 16 * (j ^ ((lane >> 1) & 3))),
                   "r"(pack_bf16x2(v[8 * j + 0], v[8 * j + 1])),
                   "r"(pack_bf16x2(v[8 * j + 2], v[8 * j + 3])),
                   "r"(pack_bf16x2(v[8 * j + 4], v[8 * j + 5])),
                   "r"(pack_bf16x2(v[8 * j + 6], v[8 * j + 7]))
                   : "memory");
    __syncwarp();
    const int j = lane & 3;
    char* d[4];
    uint4 x[4];
#pragma unroll
    for (int pass = 0; pass < 4; ++pass) {
      const int row = pass * 8 + (lane >> 2);
      d[pass] = reinterpret_cast<char*>(
          __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(dst), row));
      x[pass] = *reinterpret_cast<const uint4*>(stg + row * 64 + 16 * (j ^ ((row >> 1) & 3)));
    }
#pragma unroll
    for (int pass = 0; pass < 4; ++pass)
      if (d[pass]) reinterpret_cast<uint4*>(d[pass])[j] = x[pass];
  }
  __syncwarp();  // the staging area is rewritten by the next chunk
}

// Schedule, identical in every thread.  Tiles t = nn * mt + m (m fastest, so
// CTAs in flight share weight tiles in L2) go whole to CTA t mod G in waves.
// The (non-casting) gated residual, whose pieces add up, may instead cut
// its k range: into S equal parts when tiles x S fit one wave (one piece per
// CTA), or, when the last wave would leave more than half the CTAs idle, by
// laying the R remainder tiles end to end by k-block and cutting them into
// Gr equal ranges (stream-K, at least MIN_KB_PER_CTA k-blocks each).
//
// Pairs (two CTAs of a cluster sharing one M = 256 MMA): the same, with a
// "tile" of two row tiles (2p, 2p + 1) and G the number of pairs.
struct Sched {
  int BN, stages, mt, nt, tiles, kbt, G, whole, Gr, S;
  bool pair;
  // every CTA holds at most one work item: its epilogue starts only once
  // all of its MMAs have read the ring, so the ring may run on over the
  // epilogue staging buffers that follow it
  bool alias;
  long long Wr;
  // S > 0: split-S (requires tiles * S <= grid); S == 0: waves (+ stream-K)
  __host__ __device__ void plan(int M, int bn, int n, int k, int grid, bool additive, int s,
                                bool pr) {
    BN = bn;
    pair = pr;
    stages = stages_for(bn, pr);
    const int mt_rows = (M + BM - 1) / BM;
    mt = pair ? (mt_rows + 1) / 2 : mt_rows;
    nt = n / BN;
    tiles = mt * nt;
    kbt = k / BK;
    G = pair ? grid / 2 : grid;
    S = s;
    alias = false;
    if (S > 0) {
      whole = 0;
      Wr = 0;
      Gr = 0;
      alias = true;  // one piece per CTA
      stages = stages_for(bn, pr, true);
      return;
    }
    const int R = tiles % G;
    const bool split = additive && R > 0 && 2 * R <= G && kbt >= 2 * MIN_KB_PER_CTA;
    whole = split ? tiles - R : tiles;
    Wr = split ? (long long)R * kbt : 0;
    long long g = Wr / MIN_KB_PER_CTA;
    if (g < 1) g = 1;
    Gr = split ? int(g < G ? g : G) : 0;
    alias = whole <= G && Gr == 0;
    stages = stages_for(bn, pr, alias);
  }
  // bytes of one stage in one CTA: A (128 x 64) and B (BN x 64, half of it
  // in each CTA of a pair)
  __host__ __device__ static int stage_bytes(int bn, bool pr) {
    return STAGE_A + (pr ? bn * BK : bn * BK * 2);
  }
  __host__ __device__ static int stages_for(int bn, bool pr, bool alias = false) {
    const int s = (RING_BYTES + (alias ? STAGING_BYTES : 0)) / stage_bytes(bn, pr);
    return s < MAX_STAGES ? s : MAX_STAGES;
  }
  // Estimated duration (SM cycles): k-blocks on the busiest CTA x per-k-block
  // time (operands at ~60 B/clk per SM, but no less than the MMA issue time)
  // plus its exposed epilogues (~20 B/clk per SM with twelve epilogue warps;
  // all rates measured); a stream-K CTA holds two pieces.
  __host__ __device__ float cost(int out_bytes) const {
    // one thread issues a tcgen05.mma about every 140 cycles (4 per k-block),
    // two together twice as fast (one work item per CTA, tiles up to 192)
    const float cmma = (alias && !pair && BN <= 192) ? 280.f : 560.f;
    const float ckb = fmaxf(float(stage_bytes(BN, pair)) * (1.f / 60.f), cmma);
    const float cep = float(BM * BN * out_bytes) * (1.f / 20.f);
    if (S > 0) return float((kbt + S - 1) / S) * ckb + cep;
    const int waves = (whole + G - 1) / G;
    float c = float(waves) * float(kbt) * ckb + (waves > 0 ? cep : 0.f);
    if (Gr > 0) c += float((Wr + Gr - 1) / Gr) * ckb + 2.f * cep;
    return c;
  }
  // Picks BN (n % BN == 0) and, for the additive gated residual, a split,
  // with the lowest estimate; ties go to wider tiles and fewer pieces.
  // Returns BN / 64 + 8 S.
  __host__ __device__ static int pick(int M, int n, int k, int grid, int mode, bool pr) {
    Sched s;
    const bool additive = mode == EPI_GATE_RES;
    const int out_bytes = mode == EPI_GATE_RES_CAST ? 10
                          : (mode == EPI_F32 || mode == EPI_GATE_RES) ? 4 : 2;
    const int cand[4] = {256, 192, 128, 64};
    float best = 3.4e38f;
    int code = 1;
    for (int i = 0; i < 4; ++i) {
      if (n % cand[i]) continue;
      for (int sp = 0; sp <= (additive ? 4 : 0); ++sp) {
        if (sp == 1) continue;
        s.plan(M, cand[i], n, k, grid, additive, sp, pr);
        if (sp > 0 && (s.tiles * sp > s.G || s.kbt < sp * MIN_KB_PER_CTA)) continue;
        const float c = s.cost(out_bytes);
        if (c < best * 0.999f) {
          best = c;
          code = cand[i] / 64 + 8 * sp;
        }
      }
    }
    return code;
  }
  // table: the host's pick for 1 .. BN_TABLE row tiles (0 = not tabulated)
  __device__ void init(int M, int n, int k, int grid, int mode, const uint8_t* table, bool pr) {
    const int m_tiles = (M + BM - 1) / BM;
    int code = m_tiles >= 1 && m_tiles <= BN_TABLE ? int(table[m_tiles - 1]) : 0;
    if (code == 0) code = pick(M, n, k, grid, mode, pr);
    plan(M, 64 * (code & 7), n, k, grid, mode == EPI_GATE_RES, code >> 3, pr);
  }
  __device__ long long bound(int c) const { return Wr * c / Gr; }
};

// The segments (tile, k-blocks [kb0, kb1)) of one CTA, in order.
struct Segs {
  const Sched* sc;
  int t_next;
  long long cur, end;
  __device__ void init(const Sched& s, int c) {
    sc = &s;
    t_next = c;
    cur = c < s.Gr ? s.bound(c) : 0;
    end = c < s.Gr ? s.bound(c + 1) : 0;
    if (s.S > 0) {  // split-S: CTA c < tiles * S holds piece c / tiles of tile c % tiles
      cur = 0;
      end = c < s.tiles * s.S ? 1 : 0;
    }
  }
  __device__ bool next(int& t, int& kb0, int& kb1) {
    if (sc->S > 0) {
      if (cur >= end) return false;
      ++cur;
      const int p = t_next / sc->tiles;
      t = t_next - p * sc->tiles;
      kb0 = p * sc->kbt / sc->S;
      kb1 = (p + 1) * sc->kbt / sc->S;
      return true;
    }
    if (t_next < sc->whole) {
      t = t_next;
      t_next += sc->G;
      kb0 = 0;
      kb1 = sc->kbt;
      return true;
    }
    if (cur >= end) return false;
    const int tr = int(cur / sc->kbt);
    kb0 = int(cur - (long long)tr * sc->kbt);
    kb1 = int(min((long long)sc->kbt, kb0 + (end - cur)));
    cur += kb1 - kb0;
    t = sc->whole + tr;
    return true;
  }
};

// PAIR: launched in clusters of two CTAs that share every MMA (cta_group::2,
// M = 256): each CTA loads its own 128 rows of A and half of the W tile, and
// the even CTA's MMA thread multiplies the pair's operands into both CTAs'
// tensor memory.  Per k-block a CTA then holds (and pulls from L2)
// 16 KB + BN x 64 B instead of 16 KB + BN x 128 B, so the ring keeps more
// k-blocks in flight -- the main loop is bound by k-blocks in flight per SM
// over the load latency.
template <bool PAIR>
__global__ void __launch_bounds__(THREADS, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ BMaps tmB,
               int Mbound, const int* __restrict__ dcount, int n, int k,
               const __grid_constant__ GemmEpi ep, const __grid_constant__ BnTable bt) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned operand ring, epilogue staging, then barriers
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  // the staging buffers follow the ring; a CTA with one work item lets its
  // ring run on over them (see Sched::alias)
  uint8_t* sStg = smem + RING_BYTES;
  float* sVec = reinterpret_cast<float*>(sStg + STAGING_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStg + STAGING_BYTES + VEC_BYTES);
  // bars: full[MAX_STAGES], empty[MAX_STAGES], tfull[2], tempty[2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * MAX_STAGES + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = saddr(bars), empty0 = saddr(bars + MAX_STAGES);
  const uint32_t tfull0 = saddr(bars + 2 * MAX_STAGES), tempty0 = saddr(bars + 2 * MAX_STAGES + 2);

  // rank 0 of a pair issues the MMAs; its barriers count the pair's loads
  // (full), and both CTAs' epilogue warps (tempty: one arrival per warp)
  const uint32_t rank = PAIR ? cluster_ctarank() : 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < MAX_STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, PAIR ? 24 : 12);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if (PAIR)
      tmem_alloc_pair(saddr(tmem_slot), TMEM_COLS);
    else
      tmem_alloc(saddr(tmem_slot), TMEM_COLS);
  }
  if (warp == 0 && lane == 0)
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // the peer's barriers are initialised before any of its loads, commits or
  // arrivals can reach them
  if (PAIR) cluster_sync();

  // everything above is private set-up.  The live row count was written two
  // or more launches earlier (a step's dirty count before its first block;
  // every kernel of the library waits for its predecessor before letting its
  // successor start), so it and the schedule come before the programmatic-
  // dependency wait; the operands and the residual are read after it
  const int M = live_count(dcount, Mbound, ep.err);
  Sched sc;
  sc.init(M, n, k, int(gridDim.x), sched_mode(ep), bt.w64, PAIR);
  pdl_wait();
  pdl_trigger();
  const int BN = sc.BN, STAGES = sc.stages;
  const int STAGE = Sched::stage_bytes(BN, PAIR);
  // split2: when every CTA holds one work item (so the second accumulator is
  // free), two MMA threads take the item's even and odd k-blocks into the two
  // accumulators, which the epilogue adds.  One thread issues a tcgen05.mma
  // only about every 140 cycles when the ring stage is known at run time,
  // whatever N; two threads together issue about twice as fast (measured).
  // It shortens the main loop where few rows leave it bound by that issue
  // rate (a sparse step at 5 % dirty: 397 -> 428 steps/s).  A 256-wide MMA
  // keeps the tensor pipe busy about as long as one thread takes to issue
  // it, so 256-wide tiles keep one issuer (the second accumulator's read in
  // the epilogue would cost more than it saves: 298.7 -> 301.8 steps/s at
  // 20 % dirty without it there).
  const bool split2 = !PAIR && sc.alias && sc.kbt >= 2 && BN <= 192;
  // schedule position: the pair (its row tiles 2p + rank) or the CTA
  const int pos = PAIR ? int(blockIdx.x) >> 1 : int(blockIdx.x);

  if (warp == 0) {
    // ------------------------------------------------------- TMA producer
    if (lane == 0) {
      // W as one box of BN rows, or BN / 2 rows per CTA of a pair (maps for
      // the heights that divide n)
      const int brows = PAIR ? BN / 2 : BN;
      const CUtensorMap* tmW = &tmB.m[bmap_index(brows)];
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmW)) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      Segs sg;
      sg.init(sc, pos);
      int t, kb0, kb1;
      while (sg.next(t, kb0, kb1)) {
        const int mq = t % sc.mt, nn = t / sc.mt;
        const int m = PAIR ? 2 * mq + int(rank) : mq;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1, abort_flag)) goto timeout;
          uint8_t* st = smem + stage * STAGE;
          if (PAIR) {
            // both CTAs' bytes land on rank 0's barrier, which expects them
            const uint32_t fb = mapa_shared(full0 + 8 * stage, 0);
            if (rank == 0) mbar_expect_tx(full0 + 8 * stage, 2 * STAGE);
            tma_load_2d_pair(saddr(st), &tmA, fb, kb * BK, m * BM);
            tma_load_2d_pair(saddr(st + STAGE_A), tmW, fb, kb * BK, nn * BN + int(rank) * brows);
          } else {
            // W comes from the W warp on the same barrier (which may see
            // its bytes before this expectation: the phase still needs this
            // arrival)
            mbar_expect_tx(full0 + 8 * stage, STAGE);
            tma_load_2d(saddr(st), &tmA, full0 + 8 * stage, kb * BK, m * BM);
          }
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
    }
  } else if (warp == W_WARP) {
    // ------------------------------------------------------- TMA: W (unpaired)
    if (!PAIR && lane == 0) {
      const CUtensorMap* tmW = &tmB.m[bmap_index(BN)];
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmW)) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      Segs sg;
      sg.init(sc, pos);
      int t, kb0, kb1;
      while (sg.next(t, kb0, kb1)) {
        const int nn = t / sc.mt;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1, abort_flag)) goto timeout;
          tma_load_2d(saddr(smem + stage * STAGE + STAGE_A), tmW, full0 + 8 * stage, kb * BK,
                      nn * BN);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    if (lane == 0 && rank == 0 && split2) {
      Segs sg;
      sg.init(sc, pos);
      int t, kb0, kb1;
      if (sg.next(t, kb0, kb1) &&
          !mma_half(0, kb0, kb1, STAGES, STAGE, saddr(smem), tmem_base,
                    IDESC_BASE | (uint32_t(BN >> 3) << 17), full0, empty0, tfull0, tempty0,
                    abort_flag))
        goto timeout;
    } else if (lane == 0 && rank == 0) {
      const uint32_t idesc = (PAIR ? IDESC_PAIR : IDESC_BASE) | (uint32_t(BN >> 3) << 17);
      const uint64_t da = sw128_desc(saddr(smem)), db = sw128_desc(saddr(smem + STAGE_A));
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      Segs sg;
      sg.init(sc, pos);
      int t, kb0, kb1;
      while (sg.next(t, kb0, kb1)) {
        if (!mbar_wait(tempty0 + 8 * acc, acc_phase ^ 1, abort_flag)) goto timeout;
        tc_fence_after();
        const uint32_t dtm = tmem_base + uint32_t(acc * 256);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) goto timeout;
          tc_fence_after();
          // stage descriptors differ only in the start address field
          // (address >> 4; no carry out of its 14 bits below 256 KB)
          const uint64_t so = uint64_t((stage * STAGE) >> 4);
          if (PAIR) {
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              umma_bf16_pair(dtm, da + so + 2 * kk, db + so + 2 * kk, idesc,
                             (kb > kb0 || kk > 0) ? 1u : 0u);
            umma_commit_pair(empty0 + 8 * stage);  // frees the stage in both CTAs
          } else {
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              umma_bf16(dtm, da + so + 2 * kk, db + so + 2 * kk, idesc,
                        (kb > kb0 || kk > 0) ? 1u : 0u);
            umma_commit(empty0 + 8 * stage);
          }
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (PAIR)
          umma_commit_pair(tfull0 + 8 * acc);
        else
          umma_commit(tfull0 + 8 * acc);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
    }
  } else if (warp == MMA2_WARP) {
    // ------------------------------------------------------- second MMA issuer
    if (lane == 0 && split2) {
      Segs sg;
      sg.init(sc, pos);
      int t, kb0, kb1;
      if (sg.next(t, kb0, kb1) &&
          !mma_half(1, kb0, kb1, STAGES, STAGE, saddr(smem), tmem_base,
                    IDESC_BASE | (uint32_t(BN >> 3) << 17), full0, empty0, tfull0, tempty0,
                    abort_flag))
        goto timeout;
    }
  } else {
    // ------------------------------------------------------- epilogue (warps 2..13)
    const int sp = warp & 3;  // TMEM lane sub-partition this warp may access
    int acc = 0;
    uint32_t acc_phase = 0;
    Segs sg;
    sg.init(sc, pos);
    int t, kb0, kb1;
    // the accumulator is drained once every epilogue warp of the pair (or
    // CTA) has arrived on rank 0's barrier
    const uint32_t tempty_r0 = PAIR ? mapa_shared(tempty0, 0) : tempty0;
    // every epilogue warp passes the same number of epi_sync barriers, also
    // after a failed wait (it then skips the rest of the work), so that no
    // warp is ever left waiting at one
    bool ok = true;
    while (sg.next(t, kb0, kb1)) {
      const int mq = t % sc.mt, nn = t / sc.mt;
      const int m = PAIR ? 2 * mq + int(rank) : mq;
      // everything that does not depend on the accumulator first, while the
      // main loop runs: the row's token / item, the tile's column vectors
      const int row = sp * 32 + lane;
      const int r = m * BM + row;
      int tok = 0, item = 0;
      if (r < M) {
        if (ep.mode == EPI_QKV) tok = ep.tok ? __ldg(ep.tok + r) : r;
        if (ep.item) item = __ldg(ep.item + r);
      }
      epi_sync();  // the previous tile's readers of sVec are done
      stage_vectors(ep, nn * BN, BN, kb0 == 0, sVec, int(threadIdx.x) - 64);
      epi_sync();
      if (ok && !mbar_wait_warp(tfull0 + 8 * acc, acc_phase, abort_flag)) ok = false;
      if (ok && split2 && !mbar_wait_warp(tfull0 + 8, 0, abort_flag)) ok = false;
      if (ok) {
        tc_fence_after();
        const uint32_t tbase = tmem_base + uint32_t(acc * 256) + (uint32_t(sp * 32) << 16);
#pragma unroll 1
        for (int ch = (warp - 2) >> 2; ch < BN / 32; ch += 3) {
          float v[32];
          if (split2)
            tmem_ld32_sum2(tbase + uint32_t(ch * 32), v);
          else
            tmem_ld32(tbase + uint32_t(ch * 32), v);
          const int c0 = nn * BN + ch * 32;
          epilogue_values(ep, c0, ch * 32, item, v, sVec);
          bf16* xb_row = (ep.mode == EPI_GATE_RES_CAST && r < M)
                             ? ep.out_bf + size_t(r) * ep.ld_out + c0 : nullptr;
          store_chunk(ep.mode, sStg + (warp - 2) * STAGING_WARP, lane, v,
                      chunk_dst(ep, r, M, tok, item, c0), xb_row);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (PAIR)
            mbar_arrive_cluster(tempty_r0 + 8 * acc);
          else
            mbar_arrive(tempty0 + 8 * acc);
        }
      }
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
    if (!ok) goto timeout;
  }
  goto done;
timeout:
  *abort_flag = 1;
  atomicOr(ep.err, DEVERR_TIMEOUT);
done:
  tc_fence_before();
  __syncthreads();
  // no CTA leaves (or frees its tensor memory) while its peer may still
  // load, commit or arrive into it
  if (PAIR) cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
    else
      tmem_dealloc(tmem_base, TMEM_COLS);
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

struct MapKey {
  const void* p;
  uint64_t rows, cols, ld;
  int box_rows;
  bool operator==(const MapKey& o) const {
    return p == o.p && rows == o.rows && cols == o.cols && ld == o.ld && box_rows == o.box_rows;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& k) const {
    return std::hash<const void*>()(k.p) ^ (k.rows * 1000003ull) ^ (k.cols * 7919ull) ^
           (k.ld * 131ull) ^ size_t(k.box_rows);
  }
};

// 2-D bf16 row-major [rows][cols] (row stride ld elements), box BK x box_rows,
// 128-byte swizzle; out-of-range rows read as zero.
cudaError_t tensor_map(const bf16* p, int rows, int cols, int ld, int box_rows, CUtensorMap* out) {
  static std::mutex mu;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  MapKey key{p, uint64_t(rows), uint64_t(cols), uint64_t(ld), box_rows};
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
  cuuint64_t dims[2] = {cuuint64_t(cols), cuuint64_t(rows)};
  cuuint64_t strides[1] = {cuuint64_t(ld) * sizeof(bf16)};
  cuuint32_t box[2] = {cuuint32_t(BK), cuuint32_t(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<bf16*>(p), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, *out);
  return cudaSuccess;
}

// Tile-width table of a GEMM shape, cached (the cost model runs up to 4 x 5
// plans per row-tile count).
BnTable bn_table(int n, int k, int grid, int mode, int mt_bound, bool pair) {
  static std::mutex mu;
  static std::unordered_map<uint64_t, BnTable> cache;
  const int mtb = mt_bound < BN_TABLE ? mt_bound : BN_TABLE;
  // bits: mtb 0-6, mode 7-9, pair 10, grid 11-18, k 19-40, n 41-63
  // (mode < 8, grid < 256, n, k < 2^22: checked by the launcher)
  const uint64_t full_key = uint64_t(mtb) | (uint64_t(mode & 7) << 7) |
                            (uint64_t(pair ? 1 : 0) << 10) | (uint64_t(grid & 255) << 11) |
                            (uint64_t(k & 0x3FFFFF) << 19) | (uint64_t(n) << 41);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(full_key);
    if (it != cache.end()) return it->second;
  }
  BnTable bt{};
  for (int mt = 1; mt <= mtb; ++mt)
    bt.w64[mt - 1] = uint8_t(Sched::pick(mt * BM, n, k, grid, mode, pair));
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() > 4096) cache.clear();
  cache.emplace(full_key, bt);
  return bt;
}

// Launch shape of the current device: CTA pairs (clusters of two, one CTA
// per SM) when every SM can hold one, else one CTA per SM unpaired.
// grid 0: no device.
struct GemmShape {
  int grid;
  bool pair;
};
constexpr int PAIR_MIN_ROWS = 2048;
int device_sms() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (!sms[dev] && cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev) !=
                       cudaSuccess)
    return 0;
  return sms[dev];
}
GemmShape device_shape() {
  static GemmShape shp[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return GemmShape{0, false};
  if (!shp[dev].grid) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        v >= 256)
      return GemmShape{0, false};
    if (cudaFuncSetAttribute(gemm_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(SMEM_BYTES)) != cudaSuccess ||
        cudaFuncSetAttribute(gemm_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(SMEM_BYTES)) != cudaSuccess)
      return GemmShape{0, false};
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(v & ~1);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nc = 0;
    if (cudaOccupancyMaxActiveClusters(&nc, gemm_tc_kernel<true>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      nc = 0;
    }
    shp[dev] = nc > 0 && 2 * nc == (v & ~1) ? GemmShape{2 * nc, true} : GemmShape{v, false};
  }
  return shp[dev];
}

}  // namespace

cudaError_t launch_gemm(const bf16* A, int lda, const bf16* W, int Mbound, const int* dcount,
                        int n, int k, const GemmEpi& ep, cudaStream_t st) {
  if (Mbound <= 0) return cudaSuccess;
  if (n % 64 || k % BK || n >= (1 << 22) || k >= (1 << 22) || ep.mode < 0 || ep.mode > 7)
    return cudaErrorInvalidValue;
  const GemmShape shp = device_shape();
  if (!shp.grid) return cudaErrorInvalidDevice;
  cudaError_t e;
  CUtensorMap ta;
  BMaps tb;
  if ((e = tensor_map(A, Mbound, k, lda, BM, &ta)) != cudaSuccess) return e;
  // one W map per box height that divides n (the kernel picks the one its
  // tile width needs); the others repeat the 32-row map and are never used
  const int heights[N_BMAPS] = {32, 64, 96, 128, 192, 256};
  for (int i = 0; i < N_BMAPS; ++i) {
    const int h = n % heights[i] == 0 ? heights[i] : 32;
    if ((e = tensor_map(W, n, k, k, h, &tb.m[i])) != cudaSuccess) return e;
  }
  // pairs pay for their coupling and the cluster launch only with many row
  // tiles per CTA: measured faster at 4096 rows (QKV 37 -> 36, fc1 52 -> 48,
  // fc2 56 -> 47 us) and slower at 831 (cross-q 14.3 -> 16.4 us).  The row
  // count must be known here: a device-side count keeps CTAs unpaired.
  const bool pair = shp.pair && !dcount && Mbound >= PAIR_MIN_ROWS;
  const int grid = pair ? shp.grid : device_sms();
  const BnTable bt = bn_table(n, k, grid, sched_mode(ep), (Mbound + BM - 1) / BM, pair);
  if (pair)
    RC_TRY(launch_k_cluster(gemm_tc_kernel<true>, dim3(shp.grid), dim3(THREADS), SMEM_BYTES, 2,
                            st, ta, tb, Mbound, dcount, n, k, ep, bt));
  else
    RC_TRY(launch_k(gemm_tc_kernel<false>, dim3(grid), dim3(THREADS), SMEM_BYTES, st, ta, tb,
                    Mbound, dcount, n, k, ep, bt));
  count_launches(1);
  return cudaSuccess;
}

}  // namespace rc
