// Dirty-query flash attention (Section 3.3, Region-Level Sparse Attention):
// the queries of the active tokens attend over every token's keys / values.
// In the self-attention the K/V rows come from the (layer, timestep) cache
// whose dirty rows the QKV GEMM has just refreshed; in the text cross-
// attention they are the 120 per-layer text keys / values.
//
// One CTA = 64 queries of one head (4 warps x 16 rows) over one split of the
// keys; K/V tiles of 64 keys are double-buffered in shared memory with
// cp.async; S = Q K^T and O += P V run on mma.sync (m16n8k16, plus m16n8k8 for
// the 8-wide tail of head_dim 72); the softmax is online, in registers, in
// base 2.  With several key splits, each split stores its unnormalised output
// and row max / sum; the last split of a (query tile, head) to finish (an
// atomic ticket, no waiting) merges them in split order.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rc {

namespace {

constexpr int BQ = 64, BKV = 64, THREADS = 128;

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
__device__ __forceinline__ void ldsm_x4(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x2(uint32_t a, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];\n"
               : "=r"(r0), "=r"(r1)
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}
__device__ __forceinline__ void ldsm_x2_t(uint32_t a, uint32_t& r0, uint32_t& r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];\n"
               : "=r"(r0), "=r"(r1)
               : "r"(a));
}
__device__ __forceinline__ void mma16816(float* c, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma1688(float* c, uint32_t a0, uint32_t a1, uint32_t b0) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(b0));
}

// DH: head dim (multiple of 8).  Shared-memory rows are SROW elements: DH
// itself when DH*2 bytes is an odd multiple of 16 (144 B for 72: the 8 rows
// of an ldmatrix phase land in distinct bank groups), else DH + 8.
template <int DH>
struct Cfg {
  static constexpr int NCH = DH / 8;                       // 16-byte chunks per row
  static constexpr int SROW = ((DH / 8) % 2 == 1) ? DH : DH + 8;
  static constexpr int KS16 = DH / 16;
  static constexpr bool TAIL8 = (DH % 16) == 8;
  static constexpr int NT = DH / 8;                        // n8 tiles of O
};

template <int DH>
__global__ void __launch_bounds__(THREADS)
attn_kernel(const bf16* __restrict__ Q, int ldq, const bf16* __restrict__ Kp,
            const bf16* __restrict__ Vp, int ldkv, int Nk, bf16* __restrict__ O, int ldo,
            int Dbound, const int* __restrict__ dcount, float scale_log2, unsigned* err,
            float* __restrict__ part, int* __restrict__ tickets) {
  using C = Cfg<DH>;
  __shared__ __align__(128) bf16 sQ[BQ * C::SROW];
  __shared__ __align__(128) bf16 sK[2][BKV * C::SROW];
  __shared__ __align__(128) bf16 sV[2][BKV * C::SROW];
  __shared__ int s_last;

  pdl_wait();
  pdl_trigger();
  const int D = live_count(dcount, Dbound, err);
  const int q0 = blockIdx.x * BQ;
  const int h = blockIdx.y;
  const int nsplit = gridDim.z, split = blockIdx.z;
  if (q0 >= D) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int hoff = h * DH;

  // ---- Q tile (rows beyond D are zero)
  for (int c = tid; c < BQ * C::NCH; c += THREADS) {
    const int row = c / C::NCH, ch = c - row * C::NCH;
    const bool ok = q0 + row < D;
    const bf16* src = Q + size_t(ok ? q0 + row : q0) * ldq + hoff + ch * 8;
    cp_async16(smem_u32(sQ + row * C::SROW + ch * 8), src, ok ? 16 : 0);
  }
  auto load_kv = [&](int buf, int kb) {
    const int k0 = kb * BKV;
    for (int c = tid; c < BKV * C::NCH; c += THREADS) {
      const int row = c / C::NCH, ch = c - row * C::NCH;
      const bool ok = k0 + row < Nk;
      const size_t off = size_t(ok ? k0 + row : 0) * ldkv + hoff + ch * 8;
      cp_async16(smem_u32(sK[buf] + row * C::SROW + ch * 8), Kp + off, ok ? 16 : 0);
      cp_async16(smem_u32(sV[buf] + row * C::SROW + ch * 8), Vp + off, ok ? 16 : 0);
    }
  };
  const int nkb_all = (Nk + BKV - 1) / BKV;
  const int per = (nkb_all + nsplit - 1) / nsplit;
  const int kb_begin = split * per;
  const int kb_end = min(nkb_all, kb_begin + per);
  const int nkb = kb_end > kb_begin ? kb_end - kb_begin : 0;
  if (nkb > 0) load_kv(0, kb_begin);
  cp_async_commit();

  uint32_t qa[C::KS16][4];
  uint32_t qt[2];
  float o[C::NT][4];
#pragma unroll
  for (int i = 0; i < C::NT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY};
  float lrow[2] = {0.f, 0.f};

  for (int kb = 0; kb < nkb; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < nkb) load_kv(buf ^ 1, kb_begin + kb + 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (kb == 0) {
      const uint32_t qb = smem_u32(sQ);
#pragma unroll
      for (int kk = 0; kk < C::KS16; ++kk) {
        const int row = warp * 16 + (lane & 15);
        const int ch = kk * 2 + (lane >> 4);
        ldsm_x4(qb + (row * C::SROW + ch * 8) * 2, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
      }
      if (C::TAIL8) {
        const int row = warp * 16 + (lane & 15);
        ldsm_x2(qb + (row * C::SROW + (C::NCH - 1) * 8) * 2, qt[0], qt[1]);
      }
    }
    const uint32_t kbase = smem_u32(sK[buf]);
    const uint32_t vbase = smem_u32(sV[buf]);

    // ---- S = Q K^T  (16 x 64 per warp)
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int np = 0; np < 4; ++np) {
#pragma unroll
      for (int kk = 0; kk < C::KS16; ++kk) {
        const int row = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int ch = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + (row * C::SROW + ch * 8) * 2, b0, b1, b2, b3);
        mma16816(s[2 * np], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
        mma16816(s[2 * np + 1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b2, b3);
      }
    }
    if (C::TAIL8) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int row = half * 32 + lane;  // lane>>3 selects the n-tile, lane&7 the key
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + (row * C::SROW + (C::NCH - 1) * 8) * 2, b0, b1, b2, b3);
        mma1688(s[4 * half + 0], qt[0], qt[1], b0);
        mma1688(s[4 * half + 1], qt[0], qt[1], b1);
        mma1688(s[4 * half + 2], qt[0], qt[1], b2);
        mma1688(s[4 * half + 3], qt[0], qt[1], b3);
      }
    }

    // ---- mask the ragged key tail, online softmax (base 2)
    const int g = lane >> 2, t4 = lane & 3;
    const int kbase_idx = (kb_begin + kb) * BKV;
    float mx[2] = {mrow[0], mrow[1]};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kbase_idx + nt * 8 + 2 * t4 + (e & 1);
        float v = s[nt][e] * scale_log2;
        if (key >= Nk) v = -INFINITY;
        s[nt][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float alpha[2], sub[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      sub[r] = (mx[r] == -INFINITY) ? 0.f : mx[r];
      alpha[r] = exp2f(mrow[r] - sub[r]);
      mrow[r] = mx[r];
    }
    float ls[2] = {0.f, 0.f};
    uint32_t pa[8][2];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = exp2f(s[nt][0] - sub[0]);
      const float p1 = exp2f(s[nt][1] - sub[0]);
      const float p2 = exp2f(s[nt][2] - sub[1]);
      const float p3 = exp2f(s[nt][3] - sub[1]);
      ls[0] += p0 + p1;
      ls[1] += p2 + p3;
      pa[nt][0] = pack_bf16x2(p0, p1);
      pa[nt][1] = pack_bf16x2(p2, p3);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      ls[r] += __shfl_xor_sync(0xffffffffu, ls[r], 1);
      ls[r] += __shfl_xor_sync(0xffffffffu, ls[r], 2);
      lrow[r] = lrow[r] * alpha[r] + ls[r];
    }
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) {
      o[nt][0] *= alpha[0];
      o[nt][1] *= alpha[0];
      o[nt][2] *= alpha[1];
      o[nt][3] *= alpha[1];
    }

    // ---- O += P V
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      const uint32_t a0 = pa[2 * kc][0], a1 = pa[2 * kc][1];
      const uint32_t a2 = pa[2 * kc + 1][0], a3 = pa[2 * kc + 1][1];
      const int krow = kc * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
#pragma unroll
      for (int np = 0; np < C::NT / 2; ++np) {
        const int ch = np * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vbase + (krow * C::SROW + ch * 8) * 2, b0, b1, b2, b3);
        mma16816(o[2 * np], a0, a1, a2, a3, b0, b1);
        mma16816(o[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
      if (C::NT % 2) {
        uint32_t b0, b1;
        ldsm_x2_t(vbase + (krow * C::SROW + (C::NT - 1) * 8) * 2, b0, b1);
        mma16816(o[C::NT - 1], a0, a1, a2, a3, b0, b1);
      }
    }
    __syncthreads();  // buffer `buf` is refilled by the next iteration's prefetch
  }

  cp_async_wait<0>();
  const int g = lane >> 2, t4 = lane & 3;
  if (nsplit > 1) {
    // ---- partial result of this split, then the merge by the last split
    constexpr int SLOT = BQ * (DH + 2);
    const int tile = blockIdx.x * gridDim.y + h;
    float* mine = part + (size_t(tile) * nsplit + split) * SLOT;
    const int rr = warp * 16 + g;
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) {
      const int c = nt * 8 + 2 * t4;
      __stcg(reinterpret_cast<float2*>(mine + rr * DH + c), make_float2(o[nt][0], o[nt][1]));
      __stcg(reinterpret_cast<float2*>(mine + (rr + 8) * DH + c), make_float2(o[nt][2], o[nt][3]));
    }
    if (t4 == 0) {
      __stcg(mine + BQ * DH + rr, mrow[0]);
      __stcg(mine + BQ * DH + rr + 8, mrow[1]);
      __stcg(mine + BQ * DH + BQ + rr, lrow[0]);
      __stcg(mine + BQ * DH + BQ + rr + 8, lrow[1]);
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const int prev = atomicAdd(tickets + tile, 1);
      s_last = (prev == nsplit - 1);
      if (s_last) tickets[tile] = 0;  // re-armed for the next launch
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const float* base = part + size_t(tile) * nsplit * SLOT;
    const int r = tid >> 1, c0 = (tid & 1) * (DH / 2);
    if (q0 + r >= D) return;
    float M = -INFINITY;
    for (int q = 0; q < nsplit; ++q) M = fmaxf(M, __ldcg(base + q * SLOT + BQ * DH + r));
    const float Msub = (M == -INFINITY) ? 0.f : M;
    float L = 0.f;
    float acc[DH / 2];
#pragma unroll
    for (int c = 0; c < DH / 2; ++c) acc[c] = 0.f;
    for (int q = 0; q < nsplit; ++q) {
      const float* sl = base + q * SLOT;
      const float w = exp2f(__ldcg(sl + BQ * DH + r) - Msub);
      L += w * __ldcg(sl + BQ * DH + BQ + r);
#pragma unroll
      for (int c = 0; c < DH / 2; c += 2) {
        const float2 v = __ldcg(reinterpret_cast<const float2*>(sl + r * DH + c0 + c));
        acc[c] += w * v.x;
        acc[c + 1] += w * v.y;
      }
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    bf16* orow = O + size_t(q0 + r) * ldo + hoff + c0;
#pragma unroll
    for (int c = 0; c < DH / 2; c += 2)
      *reinterpret_cast<uint32_t*>(orow + c) = pack_bf16x2(acc[c] * inv, acc[c + 1] * inv);
    return;
  }

  // ---- normalise and store
  const float inv0 = lrow[0] > 0.f ? 1.f / lrow[0] : 0.f;
  const float inv1 = lrow[1] > 0.f ? 1.f / lrow[1] : 0.f;
  const int r0 = q0 + warp * 16 + g;
#pragma unroll
  for (int nt = 0; nt < C::NT; ++nt) {
    const int c = hoff + nt * 8 + 2 * t4;
    if (r0 < D)
      *reinterpret_cast<uint32_t*>(O + size_t(r0) * ldo + c) =
          pack_bf16x2(o[nt][0] * inv0, o[nt][1] * inv0);
    if (r0 + 8 < D)
      *reinterpret_cast<uint32_t*>(O + size_t(r0 + 8) * ldo + c) =
          pack_bf16x2(o[nt][2] * inv1, o[nt][3] * inv1);
  }
}

}  // namespace

size_t attention_split_floats(int Nmax, int heads, int dh) {
  return size_t((Nmax + BQ - 1) / BQ) * heads * ATTN_MAX_SPLIT * BQ * (dh + 2);
}

int attention_tickets(int Nmax, int heads) { return ((Nmax + BQ - 1) / BQ) * heads; }

cudaError_t launch_attention(const bf16* Q, int ldq, const bf16* K, const bf16* V, int ldkv,
                             int Nk, bf16* O, int ldo, int heads, int dh, int Dbound,
                             const int* dcount, unsigned* err, const AttnScratch& as,
                             cudaStream_t st) {
  if (Dbound <= 0) return cudaSuccess;
  const float scale_log2 = float(1.4426950408889634 / sqrt(double(dh)));
  // keys per split >= 1024: 4 splits at 4096 keys, none for the 120 text keys
  int nsplit = Nk / 1024;
  if (nsplit > ATTN_MAX_SPLIT) nsplit = ATTN_MAX_SPLIT;
  if (nsplit < 1 || !as.part || (Dbound + BQ - 1) / BQ > as.max_qtiles) nsplit = 1;
  dim3 grid((Dbound + BQ - 1) / BQ, heads, nsplit);
  if (dh == 72) {
    RC_TRY(launch_k(attn_kernel<72>, grid, dim3(THREADS), 0, st, Q, ldq, K, V, ldkv, Nk, O, ldo,
                    Dbound, dcount, scale_log2, err, as.part, as.tickets));
  } else if (dh == 64) {
    RC_TRY(launch_k(attn_kernel<64>, grid, dim3(THREADS), 0, st, Q, ldq, K, V, ldkv, Nk, O, ldo,
                    Dbound, dcount, scale_log2, err, as.part, as.tickets));
  } else {
    return cudaErrorInvalidValue;
  }
  count_launches(1);
  return cudaSuccess;
}

}  // namespace rc
