// Tensor-core GEMM of the region-sparse block on sm_103a: tcgen05.mma with
// TMEM accumulators, operands staged by TMA (128-byte swizzle), persistent
// warp-specialised CTAs, and the block's epilogues fused (bias, tanh-GELU,
// gated residual, QKV with K/V rows written straight into the cache rows of
// the dirty tokens -- Section 3.4, Kernel Fusing -- and the merged hidden
// state written into the cache's H rows).
//
// C[M][n] = A[M][k] W[n][k]^T, A and W K-major bf16, f32 accumulation.
// M (the dirty-token count) may live on the device: every CTA reads it and
// derives a stream-K schedule (equal shares of all tiles' k-blocks, so small
// and ragged tile counts still fill the GPU).  The gated residual
// (x += gate (C + b)) is written as vector reductions into x, so pieces of a
// tile simply add up; for the other epilogues the pieces of a split tile
// reduce into a zeroed f32 workspace tile and a small finish kernel, launched
// right after, applies the epilogue and zeroes the tile again.
//
// CTA = 6 warps: warp 0 issues TMA loads, warp 1 owns TMEM and issues the
// MMAs (one thread), warps 2..5 drain the accumulator (one TMEM lane = one
// output row per thread).  Two TMEM accumulators (tiles of 128 x 192, or
// 128 x 128 when 192 does not divide n) let the epilogue of one tile overlap
// the main loop of the next.
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
constexpr int THREADS = 192;
constexpr int STAGE_A = BM * BK * 2;   // bytes
constexpr int MIN_KB_PER_CTA = 4;
constexpr int MAX_BN = 192;

// Tile width BN (output features per tile): 192 when it divides n (every
// PixArt-alpha width: 1152, 2304, 3456, 4608), else 128.
template <int BN>
struct TileCfg {
  static constexpr int STAGE_B = BN * BK * 2;
  static constexpr int STAGES = (200 * 1024) / (STAGE_A + STAGE_B);  // 6 for 128, 5 for 192
  static constexpr int TMEM_COLS = (2 * BN <= 256) ? 256 : 512;     // two accumulators
  static constexpr size_t SMEM_BYTES = size_t(STAGES) * (STAGE_A + STAGE_B) + 1024 + 256;
  // Instruction descriptor, kind::f16: D f32, A and B bf16, both K-major,
  // N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                    (uint32_t(BN >> 3) << 17) | (uint32_t(BM >> 4) << 24);
};

// ---------------------------------------------------------------- epilogue
__device__ __forceinline__ void load32(const float* p, float* v) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    float4 a = __ldg(reinterpret_cast<const float4*>(p) + i);
    v[4 * i] = a.x; v[4 * i + 1] = a.y; v[4 * i + 2] = a.z; v[4 * i + 3] = a.w;
  }
}
__device__ __forceinline__ void store32_bf16(bf16* p, const float* v) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint4 u;
    u.x = pack_bf16x2(v[8 * i + 0], v[8 * i + 1]);
    u.y = pack_bf16x2(v[8 * i + 2], v[8 * i + 3]);
    u.z = pack_bf16x2(v[8 * i + 4], v[8 * i + 5]);
    u.w = pack_bf16x2(v[8 * i + 6], v[8 * i + 7]);
    reinterpret_cast<uint4*>(p)[i] = u;
  }
}

__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c),
               "f"(d)
               : "memory");
}

// Applies the epilogue to columns c0 .. c0+31 of output row r (r < M).  The
// bias is added when with_bias (the gated residual adds it from split 0 only:
// its update is a sum over splits).
__device__ __forceinline__ void epilogue32(const GemmEpi& ep, int r, int c0, float* v,
                                           bool with_bias) {
  if (ep.bias && with_bias) {
    float b[32];
    load32(ep.bias + c0, b);
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] += b[i];
  }
  switch (ep.mode) {
    case EPI_F32: {
      float4* o = reinterpret_cast<float4*>(ep.out_f + size_t(r) * ep.ld_out + c0);
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      break;
    }
    case EPI_BIAS_BF16:
      store32_bf16(ep.out_bf + size_t(r) * ep.ld_out + c0, v);
      break;
    case EPI_GELU_BF16:
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = gelu_tanh(v[i]);
      store32_bf16(ep.out_bf + size_t(r) * ep.ld_out + c0, v);
      break;
    case EPI_GATE_RES: {
      // x += gate (acc + b), as vector reductions: no read of x, and the
      // partial sums of a split K add up in place
      if (ep.gate_tab) {
        float g[32];
        load32(ep.gate_tab + c0, g);
        if (ep.gate_tb) {
          float g2[32];
          load32(ep.gate_tb + c0, g2);
#pragma unroll
          for (int i = 0; i < 32; ++i) g[i] += g2[i];
        }
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] *= g[i];
      }
      float* xp = ep.xf + size_t(r) * ep.ld_xf + c0;
#pragma unroll
      for (int i = 0; i < 8; ++i) red_add_v4(xp + 4 * i, v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      break;
    }
    case EPI_QKV: {
      const int part = c0 / ep.dsplit;
      const int cc = c0 - part * ep.dsplit;
      if (part == 0) {
        store32_bf16(ep.out_bf + size_t(r) * ep.ld_out + cc, v);
      } else {
        const int tok = ep.idx ? ep.idx[r] : r;
        if (tok >= 0 && tok < ep.n_tokens)
          store32_bf16((part == 1 ? ep.kc : ep.vc) + size_t(tok) * ep.ld_kv + cc, v);
        else
          atomicOr(ep.err, DEVERR_INDEX);
      }
      break;
    }
  }
}

// Stream-K schedule: the tiles' k-blocks are laid end to end (tile t =
// nn * mt + m, m fastest so neighbouring CTAs share weight tiles in L2) and
// CTA c takes the contiguous range [bound(c), bound(c+1)); a tile cut by a
// range boundary is "split".  At least MIN_KB_PER_CTA k-blocks per CTA.
template <int BN>
struct Sched {
  int mt, nt, tiles, kbt, G;
  long long work;
  __device__ void init(int M, int n, int k, int grid) {
    mt = (M + BM - 1) / BM;
    nt = n / BN;
    tiles = mt * nt;
    kbt = k / BK;
    work = (long long)tiles * kbt;
    long long g = work / MIN_KB_PER_CTA;
    if (g < 1) g = 1;
    G = int(g < grid ? g : grid);
  }
  __device__ long long bound(int c) const { return work * c / G; }
  // Workspace slot of tile t when a CTA range starts strictly inside it (the
  // first such CTA index, 1..G-1), else -1.
  __device__ int split_slot(int t) const {
    const long long lo = (long long)t * kbt, hi = lo + kbt;
    long long c = ((lo + 1) * G + work - 1) / work;
    while (c > 1 && bound(int(c - 1)) > lo) --c;
    while (c < G && bound(int(c)) <= lo) ++c;
    return (c < G && bound(int(c)) < hi) ? int(c) : -1;
  }
};

template <int BN>
__global__ void __launch_bounds__(THREADS, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               int Mbound, const int* __restrict__ dcount, int n, int k, GemmEpi ep,
               float* __restrict__ ws, int ws_units) {
  using TC = TileCfg<BN>;
  constexpr int STAGES = TC::STAGES, STAGE_B = TC::STAGE_B, TMEM_COLS = TC::TMEM_COLS;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned operand stages, then barriers
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * STAGE_A;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + STAGES * STAGE_B);
  // bars: full[STAGES], empty[STAGES], tfull[2], tempty[2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = saddr(bars), empty0 = saddr(bars + STAGES);
  const uint32_t tfull0 = saddr(bars + 2 * STAGES), tempty0 = saddr(bars + 2 * STAGES + 2);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 128);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     saddr(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (warp == 0 && lane == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // everything above is private set-up; inputs written by earlier kernels
  // are read only after the predecessor has completed
  pdl_wait();
  pdl_trigger();
  const int M = live_count(dcount, Mbound, ep.err);
  Sched<BN> sc;
  sc.init(M, n, k, min(int(gridDim.x), ws_units));
  const long long seg_beg = blockIdx.x < sc.G ? sc.bound(blockIdx.x) : 0;
  const long long seg_end = blockIdx.x < sc.G ? sc.bound(blockIdx.x + 1) : 0;

  if (warp == 0) {
    // ------------------------------------------------------- TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (long long cur = seg_beg; cur < seg_end;) {
        const int t = int(cur / sc.kbt);
        const int kb0 = int(cur - (long long)t * sc.kbt);
        const int kb1 = int(min((long long)sc.kbt, kb0 + (seg_end - cur)));
        cur += kb1 - kb0;
        const int m = t % sc.mt, nn = t / sc.mt;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1, abort_flag)) goto timeout;
          mbar_expect_tx(full0 + 8 * stage, STAGE_A + STAGE_B);
          tma_load_2d(saddr(sA + stage * STAGE_A), &tmA, full0 + 8 * stage, kb * BK, m * BM);
          tma_load_2d(saddr(sB + stage * STAGE_B), &tmB, full0 + 8 * stage, kb * BK, nn * BN);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (long long cur = seg_beg; cur < seg_end;) {
        const int t = int(cur / sc.kbt);
        const int kb0 = int(cur - (long long)t * sc.kbt);
        const int kb1 = int(min((long long)sc.kbt, kb0 + (seg_end - cur)));
        cur += kb1 - kb0;
        if (!mbar_wait(tempty0 + 8 * acc, acc_phase ^ 1, abort_flag)) goto timeout;
        tc_fence_after();
        const uint32_t dtm = tmem_base + uint32_t(acc * (TMEM_COLS / 2));
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) goto timeout;
          tc_fence_after();
          const uint32_t a0 = saddr(sA + stage * STAGE_A), b0 = saddr(sB + stage * STAGE_B);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_bf16(dtm, sw128_desc(a0 + 32 * kk), sw128_desc(b0 + 32 * kk), TC::IDESC,
                      (kb > kb0 || kk > 0) ? 1u : 0u);
          umma_commit(empty0 + 8 * stage);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        umma_commit(tfull0 + 8 * acc);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
    }
  } else {
    // ------------------------------------------------------- epilogue (warps 2..5)
    const int sp = warp & 3;  // TMEM lane sub-partition this warp may access
    int acc = 0;
    uint32_t acc_phase = 0;
    for (long long cur = seg_beg; cur < seg_end;) {
      const int t = int(cur / sc.kbt);
      const int kb0 = int(cur - (long long)t * sc.kbt);
      const int kb1 = int(min((long long)sc.kbt, kb0 + (seg_end - cur)));
      cur += kb1 - kb0;
      const int m = t % sc.mt, nn = t / sc.mt;
      if (!mbar_wait_warp(tfull0 + 8 * acc, acc_phase, abort_flag)) goto timeout;
      tc_fence_after();
      const int row = sp * 32 + lane;
      const int r = m * BM + row;
      const uint32_t tbase = tmem_base + uint32_t(acc * (TMEM_COLS / 2)) + (uint32_t(sp * 32) << 16);
      // a whole tile, or any piece of a gated residual (its update is a sum),
      // goes straight to the epilogue; a piece of another epilogue reduces
      // into the tile's workspace slot and the finish kernel completes it
      const bool direct = (kb0 == 0 && kb1 == sc.kbt) || ep.mode == EPI_GATE_RES;
      float* acc_row = direct ? nullptr : ws + size_t(sc.split_slot(t)) * (BM * BN) + size_t(row) * BN;
#pragma unroll 1
      for (int ch = 0; ch < BN / 32; ++ch) {
        float v[32];
        tmem_ld32(tbase + uint32_t(ch * 32), v);
        if (direct) {
          if (r < M) epilogue32(ep, r, nn * BN + ch * 32, v, kb0 == 0);
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            red_add_v4(acc_row + ch * 32 + 4 * i, v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(tempty0 + 8 * acc);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
  }
  goto done;
timeout:
  *abort_flag = 1;
  atomicOr(ep.err, DEVERR_TIMEOUT);
done:
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

// Completes the split tiles of a non-additive epilogue: reads the reduced
// f32 tile from its workspace slot, zeroes it, applies the epilogue.  One
// thread per (slot, row, 32-column chunk), grid-stride.
template <int BN>
__global__ void __launch_bounds__(256)
gemm_finish_kernel(float* __restrict__ ws, int Mbound, const int* __restrict__ dcount, int n,
                   int k, int grid, GemmEpi ep) {
  pdl_wait();
  pdl_trigger();
  const int M = live_count(dcount, Mbound, ep.err);
  Sched<BN> sc;
  sc.init(M, n, k, grid);
  constexpr int CH = BN / 32;
  // split tiles = tiles whose first inner CTA boundary is c (c = 1 .. G-1)
  const int items = (sc.G - 1) * BM * CH;
  for (int it = blockIdx.x * 256 + threadIdx.x; it < items; it += gridDim.x * 256) {
    const int c = 1 + it / (BM * CH);
    const int rem = it - (c - 1) * (BM * CH);
    const int row = rem / CH, ch = rem - (rem / CH) * CH;
    const int t = int(sc.bound(c) / sc.kbt);
    if (sc.split_slot(t) != c) continue;
    float4* p4 = reinterpret_cast<float4*>(ws + size_t(c) * (BM * BN) + size_t(row) * BN + ch * 32);
    float v[32];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 a = __ldcg(p4 + i);
      v[4 * i] = a.x; v[4 * i + 1] = a.y; v[4 * i + 2] = a.z; v[4 * i + 3] = a.w;
      __stcg(p4 + i, make_float4(0.f, 0.f, 0.f, 0.f));
    }
    const int m = t % sc.mt, nn = t / sc.mt;
    const int r = m * BM + row;
    if (r < M) epilogue32(ep, r, nn * BN + ch * 32, v, true);
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

int device_sms() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (!sms[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaFuncSetAttribute(gemm_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(TileCfg<128>::SMEM_BYTES)) != cudaSuccess ||
        cudaFuncSetAttribute(gemm_tc_kernel<192>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(TileCfg<192>::SMEM_BYTES)) != cudaSuccess)
      return 0;
    sms[dev] = v;
  }
  return sms[dev];
}

}  // namespace

cudaError_t gemm_scratch_shape(int* units, size_t* ws_floats) {
  const int sms = device_sms();
  if (!sms) return cudaErrorInvalidDevice;
  *units = sms;
  *ws_floats = size_t(sms) * BM * MAX_BN;
  return cudaSuccess;
}

cudaError_t launch_gemm(const bf16* A, int lda, const bf16* W, int Mbound, const int* dcount,
                        int n, int k, const GemmEpi& ep, const GemmScratch& gs, cudaStream_t st) {
  if (Mbound <= 0) return cudaSuccess;
  if (n % 128 || k % BK) return cudaErrorInvalidValue;
  const int sms = device_sms();
  if (!sms) return cudaErrorInvalidDevice;
  const int BN = (n % 192 == 0) ? 192 : 128;
  cudaError_t e;
  CUtensorMap ta, tb;
  if ((e = tensor_map(A, Mbound, k, lda, BM, &ta)) != cudaSuccess) return e;
  if ((e = tensor_map(W, n, k, k, BN, &tb)) != cudaSuccess) return e;
  // one workspace slot per CTA range boundary
  const int grid = min(sms, gs.units);
  if (BN == 192)
    RC_TRY(launch_k(gemm_tc_kernel<192>, dim3(grid), dim3(THREADS), TileCfg<192>::SMEM_BYTES, st,
                    ta, tb, Mbound, dcount, n, k, ep, gs.ws, grid));
  else
    RC_TRY(launch_k(gemm_tc_kernel<128>, dim3(grid), dim3(THREADS), TileCfg<128>::SMEM_BYTES, st,
                    ta, tb, Mbound, dcount, n, k, ep, gs.ws, grid));
  count_launches(1);
  if (ep.mode != EPI_GATE_RES) {
    if (BN == 192)
      RC_TRY(launch_k(gemm_finish_kernel<192>, dim3(2 * sms), dim3(256), 0, st, gs.ws, Mbound,
                      dcount, n, k, grid, ep));
    else
      RC_TRY(launch_k(gemm_finish_kernel<128>, dim3(2 * sms), dim3(256), 0, st, gs.ws, Mbound,
                      dcount, n, k, grid, ep));
    count_launches(1);
  }
  return cudaSuccess;
}

}  // namespace rc
