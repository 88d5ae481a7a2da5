// Dirty-query attention on the tensor cores (Section 3.3, Region-Level Sparse
// Attention): the queries of the active tokens attend over every token's keys
// and values.  In the self-attention K/V come from the (layer, timestep) cache
// whose dirty rows the QKV GEMM has just refreshed; in the text cross-
// attention they are the per-layer text keys / values.
//
// One work unit = 128 queries of one head over one split of the keys.  CTAs
// are persistent (one per SM) and warp-specialised:
//   warp 0     TMA: Q once per unit, then K/V blocks of 128 keys (3 stages).
//              Every operand is loaded as 16-wide head-dim blocks through a
//              3-D tensor map (head_dim, head, row) whose head_dim extent is
//              the true 72: the pad to 80 reads as zero, so the padded
//              columns add nothing to Q K^T.
//   warp 1     TMEM owner and MMA issuer: S = Q K^T (M=128, N=128, 5 K-steps
//              of 16) into one of two TMEM S buffers, one block ahead of
//              O += P V (M=128, N=80, K=128; V is an MN-major operand).
//   warps 2-5  softmax, one thread per query row: reads its S row from TMEM,
//              online softmax in base 2 with lazy rescaling (O in TMEM is
//              rescaled only when the running max grows by more than 2^8),
//              writes its P row (bf16) to a 128-byte-swizzled shared buffer,
//              and at the end normalises O and stores it.
// Key splits of the same (query tile, head) leave their unnormalised O and
// row max / sum in a workspace; for each row, the last split to finish (an
// atomic ticket per row, no waiting) merges them in split order.
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

constexpr int BQ = 128, BKV = 128, THREADS = 192;
constexpr int KV_STAGES = 3;
constexpr int BLK = BQ * 32;       // one [128 rows][16 bf16] block, 32-byte swizzled
constexpr int P_BYTES = BQ * BKV * 2;
constexpr int PART_STRIDE = 76;    // floats per row of a split's partial result
constexpr float LAZY_RESCALE = 8.f;

template <int DH>
struct ACfg {
  static constexpr int NB = (DH + 15) / 16;  // head-dim blocks (5 for 72)
  static constexpr int DHP = NB * 16;        // padded head dim (80)
  static constexpr int Q_BYTES = NB * BLK;
  static constexpr int KV_BYTES = 2 * NB * BLK;
  static constexpr size_t SMEM = size_t(Q_BYTES) + KV_STAGES * KV_BYTES + 2 * P_BYTES + 1024 + 256;
  // kind::f16, D f32, A/B bf16; S: both K-major; PV: B (V) MN-major (bit 16)
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) |
                                      (uint32_t(BKV >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_PV = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) |
                                       (uint32_t(DHP >> 3) << 17) | (uint32_t(BQ >> 4) << 24);
  static_assert(DHP <= 128 && DH + 2 <= PART_STRIDE, "head dim too large");
};

// Work list of one launch, identical in every thread.
struct AttnSched {
  int qtiles, pairs, nkb, split, per, units;
  __device__ void init(int D, int heads, int Nk, int grid, int ws_units) {
    qtiles = (D + BQ - 1) / BQ;
    pairs = qtiles * heads;
    nkb = (Nk + BKV - 1) / BKV;
    split = 1;
    while (split < 8 && pairs * split < 2 * grid && split * 2 <= nkb &&
           pairs * split * 2 <= ws_units)
      split *= 2;
    per = (nkb + split - 1) / split;
    split = (nkb + per - 1) / per;  // no empty split
    units = pairs * split;
  }
  // unit -> (query tile, head, split, key blocks [kb0, kb1)); splits of one
  // (tile, head) are adjacent, heads outermost
  __device__ void decode(int u, int& qt, int& h, int& sp, int& kb0, int& kb1) const {
    sp = u % split;
    const int pair = u / split;
    qt = pair % qtiles;
    h = pair / qtiles;
    kb0 = sp * per;
    kb1 = min(nkb, kb0 + per);
  }
};

template <int DH>
__global__ void __launch_bounds__(THREADS, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, int Nk, bf16* __restrict__ O, int ldo,
               int heads, int Dbound, const int* __restrict__ dcount, float scale_log2,
               unsigned* err, float* __restrict__ part, int* __restrict__ tickets, int ws_units) {
  using C = ACfg<DH>;
  constexpr int NB = C::NB;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + C::Q_BYTES;
  uint8_t* sP = sKV + KV_STAGES * C::KV_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + 2 * P_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // barrier addresses
  const uint32_t b0 = saddr(bars);
  const uint32_t q_full = b0, q_empty = b0 + 8;
  const uint32_t kv_full = b0 + 16, kv_empty = kv_full + 8 * KV_STAGES;
  const uint32_t s_full = kv_empty + 8 * KV_STAGES, s_free = s_full + 16;
  const uint32_t p_ready = s_free + 16, p_free = p_ready + 16;
  const uint32_t o_full = p_free + 16, o_free = o_full + 8;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int s = 0; s < KV_STAGES; ++s) {
      mbar_init(kv_full + 8 * s, 1);
      mbar_init(kv_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full + 8 * b, 1);
      mbar_init(s_free + 8 * b, 128);
      mbar_init(p_ready + 8 * b, 128);
      mbar_init(p_free + 8 * b, 1);
    }
    mbar_init(o_full, 1);
    mbar_init(o_free, 128);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(saddr(tmem_slot), 512);
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t tS0 = tmem_base, tO = tmem_base + 256;

  pdl_wait();
  pdl_trigger();
  const int D = live_count(dcount, Dbound, err);
  AttnSched sc;
  sc.init(D, heads, Nk, gridDim.x, ws_units);

  if (warp == 0) {
    // ------------------------------------------------------------ TMA
    if (lane == 0) {
      int g = 0, uc = 0;
      for (int u = blockIdx.x; u < sc.units; u += gridDim.x, ++uc) {
        int qt, h, sp, kb0, kb1;
        sc.decode(u, qt, h, sp, kb0, kb1);
        if (!mbar_wait(q_empty, (uc + 1) & 1, abort_flag)) goto timeout;
        mbar_expect_tx(q_full, C::Q_BYTES);
        for (int jj = 0; jj < NB; ++jj)
          tma_load_3d(saddr(sQ + jj * BLK), &tmQ, q_full, jj * 16, h, qt * BQ);
        for (int kb = kb0; kb < kb1; ++kb, ++g) {
          const int st = g % KV_STAGES;
          if (!mbar_wait(kv_empty + 8 * st, ((g / KV_STAGES) & 1) ^ 1, abort_flag)) goto timeout;
          mbar_expect_tx(kv_full + 8 * st, C::KV_BYTES);
          uint8_t* base = sKV + st * C::KV_BYTES;
          for (int jj = 0; jj < NB; ++jj)
            tma_load_3d(saddr(base + jj * BLK), &tmK, kv_full + 8 * st, jj * 16, h, kb * BKV);
          for (int jj = 0; jj < NB; ++jj)
            tma_load_3d(saddr(base + (NB + jj) * BLK), &tmV, kv_full + 8 * st, jj * 16, h,
                        kb * BKV);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA
    if (lane == 0) {
      int g = 0, uc = 0;
      const uint32_t qb = saddr(sQ);
      for (int u = blockIdx.x; u < sc.units; u += gridDim.x, ++uc) {
        int qt, h, sp, kb0, kb1;
        sc.decode(u, qt, h, sp, kb0, kb1);
        const int n = kb1 - kb0;
        if (!mbar_wait(q_full, uc & 1, abort_flag)) goto timeout;
        tc_fence_after();
        for (int j = -1; j < n; ++j) {
          // S for block j + 1, one block ahead of P V for block j
          if (j + 1 < n) {
            const int gg = g + j + 1;
            const int st = gg % KV_STAGES;
            if (!mbar_wait(kv_full + 8 * st, (gg / KV_STAGES) & 1, abort_flag)) goto timeout;
            if (!mbar_wait(s_free + 8 * (gg & 1), ((gg >> 1) + 1) & 1, abort_flag)) goto timeout;
            tc_fence_after();
            const uint32_t kbase = saddr(sKV + st * C::KV_BYTES);
            for (int jj = 0; jj < NB; ++jj)
              umma_bf16(tS0 + 128u * uint32_t(gg & 1), sw32_kmajor_desc(qb + jj * BLK),
                        sw32_kmajor_desc(kbase + jj * BLK), C::IDESC_S, jj > 0 ? 1u : 0u);
            umma_commit(s_full + 8 * (gg & 1));
            if (j + 2 == n) umma_commit(q_empty);  // last S of the unit issued
          }
          if (j < 0) continue;
          const int gj = g + j;
          if (j == 0) {
            if (!mbar_wait(o_free, (uc + 1) & 1, abort_flag)) goto timeout;
          }
          if (!mbar_wait(p_ready + 8 * (gj & 1), (gj >> 1) & 1, abort_flag)) goto timeout;
          tc_fence_after();
          const int st = gj % KV_STAGES;
          const uint32_t vb = saddr(sKV + st * C::KV_BYTES + NB * BLK);
          const uint32_t pb = saddr(sP + (gj & 1) * P_BYTES);
#pragma unroll
          for (int kk = 0; kk < BKV / 16; ++kk)
            umma_bf16(tO, sw128_desc(pb + (kk >> 2) * (BQ * 128) + (kk & 3) * 32),
                      sw32_mnmajor_desc(vb + kk * 16 * 32, BLK), C::IDESC_PV,
                      (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(p_free + 8 * (gj & 1));
          umma_commit(kv_empty + 8 * st);
        }
        g += n;
        umma_commit(o_full);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int sp4 = warp & 3;
    const int row = sp4 * 32 + lane;
    const uint32_t lane_off = uint32_t(sp4 * 32) << 16;
    int g = 0, uc = 0;
    for (int u = blockIdx.x; u < sc.units; u += gridDim.x, ++uc) {
      int qt, h, sp, kb0, kb1;
      sc.decode(u, qt, h, sp, kb0, kb1);
      const int n = kb1 - kb0;
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < n; ++j, ++g) {
        if (!mbar_wait_warp(s_full + 8 * (g & 1), (g >> 1) & 1, abort_flag)) goto timeout;
        tc_fence_after();
        uint32_t r[BKV];
#pragma unroll
        for (int i = 0; i < BKV / 16; ++i)
          tmem_ld16_nowait(tS0 + 128u * uint32_t(g & 1) + lane_off + 16u * i, r + 16 * i);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(s_free + 8 * (g & 1));
        const int valid = Nk - (kb0 + j) * BKV;
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < BKV; ++c) {
          const float v = c < valid ? __uint_as_float(r[c]) * scale_log2 : -INFINITY;
          r[c] = __float_as_uint(v);
          mx = fmaxf(mx, v);
        }
        if (j == 0) {
          m = mx;
        } else if (__any_sync(0xffffffffu, mx > m + LAZY_RESCALE)) {
          // (warp-uniform branch: the TMEM accesses below are warp-wide)
          mx = fmaxf(mx, m);
          // O holds P V of blocks < j: wait for the last of them, then rescale
          if (!mbar_wait_warp(p_free + 8 * ((g - 1) & 1), ((g - 1) >> 1) & 1, abort_flag))
            goto timeout;
          tc_fence_after();
          const float alpha = exp2f(m - mx);
#pragma unroll
          for (int i = 0; i < NB; ++i) {
            uint32_t o16[16];
            tmem_ld16_nowait(tO + lane_off + 16u * i, o16);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) o16[e] = __float_as_uint(__uint_as_float(o16[e]) * alpha);
            tmem_st16(tO + lane_off + 16u * i, o16);
          }
          tmem_wait_st();
          l *= alpha;
          m = mx;
        }
        float sum = 0.f;
#pragma unroll
        for (int c = 0; c < BKV; ++c) {
          const float p = exp2f(__uint_as_float(r[c]) - m);
          r[c] = __float_as_uint(p);
          sum += p;
        }
        l += sum;
        // P buffer (g & 1) is free once P V of block g - 2 is done
        if (!mbar_wait_warp(p_free + 8 * (g & 1), ((g >> 1) + 1) & 1, abort_flag)) goto timeout;
        uint8_t* prow = sP + (g & 1) * P_BYTES + row * 128;
#pragma unroll
        for (int c16 = 0; c16 < BKV / 8; ++c16) {
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(r[8 * c16 + 0]), __uint_as_float(r[8 * c16 + 1]));
          w.y = pack_bf16x2(__uint_as_float(r[8 * c16 + 2]), __uint_as_float(r[8 * c16 + 3]));
          w.z = pack_bf16x2(__uint_as_float(r[8 * c16 + 4]), __uint_as_float(r[8 * c16 + 5]));
          w.w = pack_bf16x2(__uint_as_float(r[8 * c16 + 6]), __uint_as_float(r[8 * c16 + 7]));
          const int atom = c16 >> 3, ch = c16 & 7;
          *reinterpret_cast<uint4*>(prow + atom * (BQ * 128) + ((ch ^ (row & 7)) << 4)) = w;
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(p_ready + 8 * (g & 1));
      }
      // ---- unit epilogue
      if (!mbar_wait_warp(o_full, uc & 1, abort_flag)) goto timeout;
      tc_fence_after();
      uint32_t o[C::DHP];
#pragma unroll
      for (int i = 0; i < NB; ++i) tmem_ld16_nowait(tO + lane_off + 16u * i, o + 16 * i);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(o_free);
      const int qrow = qt * BQ + row;
      if (sc.split == 1) {
        if (qrow < D) {
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
        const int pair = u / sc.split;
        float* mine = part + (size_t(pair) * sc.split + sp) * (BQ * PART_STRIDE) +
                      size_t(row) * PART_STRIDE;
#pragma unroll
        for (int c4 = 0; c4 < DH / 4; ++c4)
          __stcg(reinterpret_cast<float4*>(mine) + c4,
                 make_float4(__uint_as_float(o[4 * c4]), __uint_as_float(o[4 * c4 + 1]),
                             __uint_as_float(o[4 * c4 + 2]), __uint_as_float(o[4 * c4 + 3])));
        __stcg(reinterpret_cast<float2*>(mine + DH), make_float2(m, l));
        // per-row ticket: the last split to finish this row merges it (no
        // cross-warp barrier, no waiting)
        __threadfence();
        int* tk = tickets + size_t(pair) * BQ + row;
        const bool last = atomicAdd(tk, 1) == sc.split - 1;
        if (last) {
          *tk = 0;  // re-armed for the next launch
          if (qrow < D) {
            __threadfence();
            const float* base = part + size_t(pair) * sc.split * (BQ * PART_STRIDE) +
                                size_t(row) * PART_STRIDE;
            float M = -INFINITY;
            for (int q = 0; q < sc.split; ++q)
              M = fmaxf(M, __ldcg(base + size_t(q) * (BQ * PART_STRIDE) + DH));
            float L = 0.f;
            float acc[DH];
#pragma unroll
            for (int c = 0; c < DH; ++c) acc[c] = 0.f;
            for (int q = 0; q < sc.split; ++q) {
              const float* sl = base + size_t(q) * (BQ * PART_STRIDE);
              const float2 ml = __ldcg(reinterpret_cast<const float2*>(sl + DH));
              const float w = exp2f(ml.x - M);
              L += w * ml.y;
#pragma unroll
              for (int c4 = 0; c4 < DH / 4; ++c4) {
                const float4 v = __ldcg(reinterpret_cast<const float4*>(sl) + c4);
                acc[4 * c4] += w * v.x;
                acc[4 * c4 + 1] += w * v.y;
                acc[4 * c4 + 2] += w * v.z;
                acc[4 * c4 + 3] += w * v.w;
              }
            }
            const float inv = L > 0.f ? 1.f / L : 0.f;
            uint4* dst = reinterpret_cast<uint4*>(O + size_t(qrow) * ldo + h * DH);
#pragma unroll
            for (int c8 = 0; c8 < DH / 8; ++c8) {
              uint4 w;
              w.x = pack_bf16x2(acc[8 * c8 + 0] * inv, acc[8 * c8 + 1] * inv);
              w.y = pack_bf16x2(acc[8 * c8 + 2] * inv, acc[8 * c8 + 3] * inv);
              w.z = pack_bf16x2(acc[8 * c8 + 4] * inv, acc[8 * c8 + 5] * inv);
              w.w = pack_bf16x2(acc[8 * c8 + 6] * inv, acc[8 * c8 + 7] * inv);
              dst[c8] = w;
            }
          }
        }
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
    tmem_dealloc(tmem_base, 512);
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
// holds `heads` blocks of dh; boxes of 16 x 1 x 128, 32-byte swizzle; reads
// outside the view (head_dim >= dh, row >= rows) return zero.
cudaError_t head_map(const bf16* p, int rows, int ld, int heads, int dh, CUtensorMap* out) {
  static std::mutex mu;
  static std::unordered_map<HeadMapKey, CUtensorMap, HeadMapHash> cache;
  HeadMapKey key{p, rows, ld, heads, dh};
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
  cuuint32_t box[3] = {16, 1, cuuint32_t(BQ)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<bf16*>(p), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B,
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
                             int(ACfg<64>::SMEM)) != cudaSuccess)
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
  return size_t(4) * (sms > 0 ? sms : 160) * BQ * PART_STRIDE;
}

// (query tile, head) pairs; the context allocates 128 row tickets per pair
int attention_tickets(int Nmax, int heads) { return ((Nmax + BQ - 1) / BQ) * heads; }

cudaError_t launch_attention(const bf16* Q, int ldq, const bf16* K, const bf16* V, int ldkv,
                             int Nk, bf16* O, int ldo, int heads, int dh, int Dbound,
                             const int* dcount, unsigned* err, const AttnScratch& as,
                             cudaStream_t st) {
  if (Dbound <= 0) return cudaSuccess;
  if (dh != 72 && dh != 64) return cudaErrorInvalidValue;
  const int sms = device_sms_attn();
  if (!sms) return cudaErrorInvalidDevice;
  CUtensorMap tq, tk, tv;
  RC_TRY(head_map(Q, Dbound, ldq, heads, dh, &tq));
  RC_TRY(head_map(K, Nk, ldkv, heads, dh, &tk));
  RC_TRY(head_map(V, Nk, ldkv, heads, dh, &tv));
  const float scale_log2 = float(1.4426950408889634 / sqrt(double(dh)));
  const int ws_units = int(as.part_floats / (size_t(BQ) * PART_STRIDE));
  if (dh == 72)
    RC_TRY(launch_k(attn_tc_kernel<72>, dim3(sms), dim3(THREADS), ACfg<72>::SMEM, st, tq, tk, tv,
                    Nk, O, ldo, heads, Dbound, dcount, scale_log2, err, as.part, as.tickets,
                    ws_units));
  else
    RC_TRY(launch_k(attn_tc_kernel<64>, dim3(sms), dim3(THREADS), ACfg<64>::SMEM, st, tq, tk, tv,
                    Nk, O, ldo, heads, Dbound, dcount, scale_log2, err, as.part, as.tickets,
                    ws_units));
  count_launches(1);
  return cudaSuccess;
}

}  // namespace rc
