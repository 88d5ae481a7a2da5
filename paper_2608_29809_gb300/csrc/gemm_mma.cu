// Warp-level (mma.sync m16n8k16) bf16 GEMM with the block's fused epilogues.
// C[M][n] = A[M][k] W[n][k]^T; M (the dirty-row count) may live on the device.
// 128x128x32 CTA tile, 8 warps of 64x32, 4-stage cp.async pipeline, XOR-
// swizzled shared memory read by ldmatrix.
#include "common.cuh"
#include "kernels.h"

namespace rc {

namespace {

constexpr int BM = 128, BN = 128, BK = 32, STAGES = 4, THREADS = 256;
constexpr int A_STAGE = BM * BK;  // elements
constexpr int B_STAGE = BN * BK;
constexpr size_t SMEM_BYTES = size_t(STAGES) * (A_STAGE + B_STAGE) * sizeof(bf16);

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src),
               "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                            uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float* c, const uint32_t* a, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte chunk `ch` of row `row` in a [rows][BK] bf16 tile:
// rows are 64 bytes; chunks are XOR-swizzled by (row >> 1) & 3 so that the 8
// rows an ldmatrix phase reads fall in distinct bank groups.
__device__ __forceinline__ uint32_t tile_off(int row, int ch) {
  return uint32_t(row * (BK * 2) + ((ch ^ ((row >> 1) & 3)) << 4));
}

// Applies the epilogue to the column pair (c, c+1) of row r.
__device__ __forceinline__ void epi_pair(const GemmEpi& ep, int r, int c, float v0, float v1) {
  if (ep.bias) {
    float2 b = *reinterpret_cast<const float2*>(ep.bias + c);
    v0 += b.x;
    v1 += b.y;
  }
  switch (ep.mode) {
    case EPI_F32:
      *reinterpret_cast<float2*>(ep.out_f + size_t(r) * ep.ld_out + c) = make_float2(v0, v1);
      break;
    case EPI_BIAS_BF16:
      *reinterpret_cast<uint32_t*>(ep.out_bf + size_t(r) * ep.ld_out + c) = pack_bf16x2(v0, v1);
      break;
    case EPI_GELU_BF16:
      *reinterpret_cast<uint32_t*>(ep.out_bf + size_t(r) * ep.ld_out + c) =
          pack_bf16x2(gelu_tanh(v0), gelu_tanh(v1));
      break;
    case EPI_GATE_RES: {
      if (ep.gate_tab) {
        float2 g = *reinterpret_cast<const float2*>(ep.gate_tab + c);
        if (ep.gate_tb) {
          float2 g2 = *reinterpret_cast<const float2*>(ep.gate_tb + c);
          g.x += g2.x;
          g.y += g2.y;
        }
        v0 *= g.x;
        v1 *= g.y;
      }
      float2* xp = reinterpret_cast<float2*>(ep.xf + size_t(r) * ep.ld_xf + c);
      float2 x = *xp;
      x.x += v0;
      x.y += v1;
      *xp = x;
      const uint32_t packed = pack_bf16x2(x.x, x.y);
      if (ep.copy_bf)
        *reinterpret_cast<uint32_t*>(ep.copy_bf + size_t(r) * ep.ld_copy + c) = packed;
      if (ep.scat) {
        const int tok = ep.idx ? ep.idx[r] : r;
        if (tok >= 0 && tok < ep.n_tokens)
          *reinterpret_cast<uint32_t*>(ep.scat + size_t(tok) * ep.ld_kv + c) = packed;
        else
          atomicOr(ep.err, DEVERR_INDEX);
      }
      break;
    }
    case EPI_QKV: {
      const uint32_t packed = pack_bf16x2(v0, v1);
      const int part = c / ep.dsplit;
      const int cc = c - part * ep.dsplit;
      if (part == 0) {
        *reinterpret_cast<uint32_t*>(ep.out_bf + size_t(r) * ep.ld_out + cc) = packed;
      } else {
        const int tok = ep.idx ? ep.idx[r] : r;
        if (tok >= 0 && tok < ep.n_tokens) {
          bf16* dst = (part == 1) ? ep.kc : ep.vc;
          *reinterpret_cast<uint32_t*>(dst + size_t(tok) * ep.ld_kv + cc) = packed;
        } else {
          atomicOr(ep.err, DEVERR_INDEX);
        }
      }
      break;
    }
  }
}

__global__ void __launch_bounds__(THREADS)
gemm_mma_kernel(const bf16* __restrict__ A, int lda, const bf16* __restrict__ W, int Mbound,
                const int* __restrict__ dcount, int n, int k, GemmEpi ep) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int M = live_count(dcount, Mbound, ep.err);
  const int m0 = blockIdx.y * BM;
  const int n0 = blockIdx.x * BN;
  if (m0 >= M) return;

  bf16* sA = reinterpret_cast<bf16*>(smem);
  bf16* sB = sA + STAGES * A_STAGE;
  const uint32_t sA0 = smem_u32(sA), sB0 = smem_u32(sB);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wm = warp >> 2, wn = warp & 3;
  const int KT = k / BK;

  auto load_stage = [&](int stage, int kt) {
    const int k0 = kt * BK;
#pragma unroll
    for (int it = 0; it < (BM * BK / 8) / THREADS; ++it) {
      const int c = tid + it * THREADS;
      const int row = c >> 2, ch = c & 3;
      const int grow = m0 + row;
      const bool ok = grow < M;
      const bf16* src = A + size_t(ok ? grow : m0) * lda + k0 + ch * 8;
      cp_async16(sA0 + stage * A_STAGE * 2 + tile_off(row, ch), src, ok ? 16 : 0);
    }
#pragma unroll
    for (int it = 0; it < (BN * BK / 8) / THREADS; ++it) {
      const int c = tid + it * THREADS;
      const int row = c >> 2, ch = c & 3;
      const bf16* src = W + size_t(n0 + row) * k + k0 + ch * 8;
      cp_async16(sB0 + stage * B_STAGE * 2 + tile_off(row, ch), src, 16);
    }
  };

  float acc[4][4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

#pragma unroll
  for (int s = 0; s < STAGES - 1; ++s) {
    if (s < KT) load_stage(s, s);
    cp_async_commit();
  }

  for (int kt = 0; kt < KT; ++kt) {
    cp_async_wait<STAGES - 2>();
    __syncthreads();
    const int nk = kt + STAGES - 1;
    if (nk < KT) load_stage(nk % STAGES, nk);
    cp_async_commit();

    const int stage = kt % STAGES;
    const uint32_t aBase = sA0 + stage * A_STAGE * 2;
    const uint32_t bBase = sB0 + stage * B_STAGE * 2;
#pragma unroll
    for (int kk = 0; kk < BK / 16; ++kk) {
      uint32_t af[4][4];
#pragma unroll
      for (int mi = 0; mi < 4; ++mi) {
        const int row = wm * 64 + mi * 16 + (lane & 15);
        const int ch = kk * 2 + (lane >> 4);
        ldmatrix_x4(aBase + tile_off(row, ch), af[mi][0], af[mi][1], af[mi][2], af[mi][3]);
      }
      uint32_t bfr[4][2];
#pragma unroll
      for (int nj = 0; nj < 2; ++nj) {
        const int row = wn * 32 + nj * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int ch = kk * 2 + ((lane >> 3) & 1);
        ldmatrix_x4(bBase + tile_off(row, ch), bfr[2 * nj][0], bfr[2 * nj][1],
                    bfr[2 * nj + 1][0], bfr[2 * nj + 1][1]);
      }
#pragma unroll
      for (int mi = 0; mi < 4; ++mi)
#pragma unroll
        for (int ni = 0; ni < 4; ++ni) mma_bf16_16816(acc[mi][ni], af[mi], bfr[ni][0], bfr[ni][1]);
    }
  }
  cp_async_wait<0>();

  const int g = lane >> 2, t4 = lane & 3;
#pragma unroll
  for (int mi = 0; mi < 4; ++mi) {
#pragma unroll
    for (int ni = 0; ni < 4; ++ni) {
      const int r = m0 + wm * 64 + mi * 16 + g;
      const int c = n0 + wn * 32 + ni * 8 + 2 * t4;
      if (r < M) epi_pair(ep, r, c, acc[mi][ni][0], acc[mi][ni][1]);
      if (r + 8 < M) epi_pair(ep, r + 8, c, acc[mi][ni][2], acc[mi][ni][3]);
    }
  }
}

}  // namespace

cudaError_t launch_gemm_mma(const bf16* A, int lda, const bf16* W, int Mbound, const int* dcount,
                            int n, int k, const GemmEpi& ep, cudaStream_t st) {
  if (Mbound <= 0) return cudaSuccess;
  static int attr_dev = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (attr_dev != dev) {
    cudaFuncSetAttribute(gemm_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         int(SMEM_BYTES));
    attr_dev = dev;
  }
  dim3 grid(n / BN, (Mbound + BM - 1) / BM);
  gemm_mma_kernel<<<grid, THREADS, SMEM_BYTES, st>>>(A, lda, W, Mbound, dcount, n, k, ep);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace rc
