// Row-wise and reduction kernels of the region-sparse DiT step: the
// localisation mask (Section 3.2, R_edit), adaLN modulation, patch embedding,
// timestep embedding, final layer + DDIM update, row gather/scatter.
// All of them are HBM- or latency-bound; rows are read with 128-bit loads.
#include <float.h>
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace rc {

static inline int cdiv(int a, int b) { return (a + b - 1) / b; }

int device_sm_count() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 128;
  if (!sms[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
      v = 128;
    sms[dev] = v;
  }
  return sms[dev];
}

// Grid of a row kernel: enough CTAs for the row bound, at most `per_sm` per
// SM; the kernels loop over rows, so a device-side row count below the bound
// costs no empty CTAs.
static inline int row_grid(int rows_bound, int rows_per_cta, int per_sm) {
  const int want = cdiv(rows_bound, rows_per_cta);
  const int cap = per_sm * device_sm_count();
  return want < cap ? want : cap;
}

// ============================================================ localisation
// Workspace: abar f32 [n_delta][N] | part f32x2 [nblk][n_delta] | union u8 [N]
// | cnt int [nblk].  One thread per token, MASK_ROWS tokens per CTA.
constexpr int MASK_ROWS = 256;

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t localize_workspace_bytes(int N, int n_delta) {
  int nblk = cdiv(N, MASK_ROWS);
  return align256(sizeof(float) * size_t(n_delta) * N) +
         align256(sizeof(float2) * size_t(nblk) * n_delta) + align256(size_t(N)) +
         align256(sizeof(int) * size_t(nblk));
}

struct MaskWs {
  float* abar;
  float2* part;
  uint8_t* uni;
  int* cnt;
};

static MaskWs carve(void* ws, int N, int n_delta) {
  int nblk = cdiv(N, MASK_ROWS);
  char* p = static_cast<char*>(ws);
  MaskWs w;
  w.abar = reinterpret_cast<float*>(p);
  p += align256(sizeof(float) * size_t(n_delta) * N);
  w.part = reinterpret_cast<float2*>(p);
  p += align256(sizeof(float2) * size_t(nblk) * n_delta);
  w.uni = reinterpret_cast<uint8_t*>(p);
  p += align256(size_t(N));
  w.cnt = reinterpret_cast<int*>(p);
  return w;
}

// Pass 1: a_j(i) = (sum_s A[s][i][j]) / S for each delta token j (summed in
// ascending s, f32 round-to-nearest), and per-CTA min / max of each column.
// A non-finite a_j(i) (NaN, +-Inf) enters the min / max as the pair
// (-Inf, +Inf): finite values never reach those bounds, so pass 2 reads them
// as "this column holds a non-finite value" and drops the column.
__global__ void __launch_bounds__(MASK_ROWS)
mask_colstats_kernel(const float* __restrict__ A, int S, int N, int M, DeltaIds ids,
                     float* __restrict__ abar, float2* __restrict__ part) {
  pdl_wait();
  pdl_trigger();
  __shared__ float smin[MASK_ROWS / 32], smax[MASK_ROWS / 32];
  const int i = blockIdx.x * MASK_ROWS + threadIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const size_t plane = size_t(N) * M;
  for (int j = 0; j < ids.n; ++j) {
    const int col = ids.id[j];
    float lo = FLT_MAX, hi = -FLT_MAX;
    if (i < N) {
      float a = __ldg(A + size_t(i) * M + col);
      for (int s = 1; s < S; ++s) a = __fadd_rn(a, __ldg(A + s * plane + size_t(i) * M + col));
      a = __fdiv_rn(a, float(S));
      abar[size_t(j) * N + i] = a;
      if (isfinite(a)) {
        lo = hi = a;
      } else {
        lo = -INFINITY;
        hi = INFINITY;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) { smin[warp] = lo; smax[warp] = hi; }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w = 1; w < MASK_ROWS / 32; ++w) { lo = fminf(lo, smin[w]); hi = fmaxf(hi, smax[w]); }
      part[size_t(blockIdx.x) * ids.n + j] = make_float2(lo, hi);
    }
    __syncthreads();
  }
}

// Pass 2: column min / max over all CTAs (exact, order-free), then the
// thresholded union over the delta tokens: ((a - mn) / (mx - mn)) >= tau.
// A constant column, or one holding a non-finite value, gives no token.
__global__ void __launch_bounds__(MASK_ROWS)
mask_threshold_kernel(const float* __restrict__ abar, const float2* __restrict__ part, int nblk,
                      int N, DeltaIds ids, float tau, uint8_t* __restrict__ uni) {
  pdl_wait();
  pdl_trigger();
  __shared__ float s_mn[64], s_rng[64];
  __shared__ int s_ok[64];
  if (threadIdx.x < ids.n) {
    const int j = threadIdx.x;
    float lo = FLT_MAX, hi = -FLT_MAX;
    for (int b = 0; b < nblk; ++b) {
      float2 v = part[size_t(b) * ids.n + j];
      lo = fminf(lo, v.x);
      hi = fmaxf(hi, v.y);
    }
    float rng = __fsub_rn(hi, lo);
    s_mn[j] = lo;
    s_rng[j] = rng;
    s_ok[j] = rng > 0.0f && lo != -INFINITY && hi != INFINITY;
  }
  __syncthreads();
  const int i = blockIdx.x * MASK_ROWS + threadIdx.x;
  if (i >= N) return;
  uint8_t u = 0;
  for (int j = 0; j < ids.n; ++j) {
    if (!s_ok[j]) continue;
    float nv = __fdiv_rn(__fsub_rn(abar[size_t(j) * N + i], s_mn[j]), s_rng[j]);
    u |= (nv >= tau) ? 1 : 0;
  }
  uni[i] = u;
}

// Pass 3: (2r+1)^2 dilation on the grid, and the per-CTA dirty count.
__global__ void __launch_bounds__(MASK_ROWS)
mask_dilate_kernel(const uint8_t* __restrict__ uni, int gh, int gw, int r,
                   uint8_t* __restrict__ mask, int* __restrict__ cnt) {
  pdl_wait();
  pdl_trigger();
  const int N = gh * gw;
  const int i = blockIdx.x * MASK_ROWS + threadIdx.x;
  int m = 0;
  if (i < N) {
    const int y = i / gw, x = i - (i / gw) * gw;
    const int y0 = max(0, y - r), y1 = min(gh - 1, y + r);
    const int x0 = max(0, x - r), x1 = min(gw - 1, x + r);
    for (int yy = y0; yy <= y1 && !m; ++yy)
      for (int xx = x0; xx <= x1; ++xx)
        if (uni[yy * gw + xx]) { m = 1; break; }
    mask[i] = uint8_t(m);
  }
  int c = __syncthreads_count(m);
  if (threadIdx.x == 0) cnt[blockIdx.x] = c;
}

// Pass 4: compaction.  Each CTA sums the counts of the CTAs before it, then a
// warp ballot + prefix over warps gives each dirty token its slot; the
// indices come out in ascending token order.
__global__ void __launch_bounds__(MASK_ROWS)
mask_compact_kernel(const uint8_t* __restrict__ mask, const int* __restrict__ cnt, int N,
                    int32_t* __restrict__ idx, int32_t* __restrict__ count) {
  pdl_wait();
  pdl_trigger();
  __shared__ int s_warp[MASK_ROWS / 32];
  __shared__ int s_base;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x < 32) {
    int acc = 0;
    for (int b = lane; b < int(blockIdx.x); b += 32) acc += cnt[b];
    acc = __reduce_add_sync(0xffffffffu, acc);
    if (lane == 0) s_base = acc;
  }
  const int i = blockIdx.x * MASK_ROWS + threadIdx.x;
  const int m = (i < N) ? mask[i] : 0;
  const unsigned bal = __ballot_sync(0xffffffffu, m);
  if (lane == 0) s_warp[warp] = __popc(bal);
  __syncthreads();
  int before = s_base;
  for (int w = 0; w < warp; ++w) before += s_warp[w];
  if (m) idx[before + __popc(bal & ((1u << lane) - 1u))] = i;
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
    int total = s_base;
    for (int w = 0; w < MASK_ROWS / 32; ++w) total += s_warp[w];
    *count = total;
  }
}

cudaError_t launch_localize(const float* A, int S, int N, int M, int gh, int gw,
                            const DeltaIds& ids, float tau, int dilation, uint8_t* mask,
                            int32_t* idx, int32_t* count, void* ws, cudaStream_t st) {
  const int nblk = cdiv(N, MASK_ROWS);
  MaskWs w = carve(ws, N, ids.n);
  RC_TRY(launch_k(mask_colstats_kernel, dim3(nblk), dim3(MASK_ROWS), 0, st, A, S, N, M, ids,
                  w.abar, w.part));
  RC_TRY(launch_k(mask_threshold_kernel, dim3(nblk), dim3(MASK_ROWS), 0, st, w.abar, w.part, nblk,
                  N, ids, tau, w.uni));
  RC_TRY(launch_k(mask_dilate_kernel, dim3(nblk), dim3(MASK_ROWS), 0, st, w.uni, gh, gw, dilation,
                  mask, w.cnt));
  RC_TRY(launch_k(mask_compact_kernel, dim3(nblk), dim3(MASK_ROWS), 0, st, mask, w.cnt, N, idx,
                  count));
  count_launches(4);
  return cudaSuccess;
}

// ================================================================= LN + mod
// One warp per row; the row stays in registers (hidden <= 1536, % 128 == 0).
constexpr int LN_WARPS = 8;
constexpr int LN_MAXV = 12;  // float4 per lane
constexpr int LN_SV = (LN_MAXV * 32 + LN_WARPS * 32 - 1) / (LN_WARPS * 32);  // float4 per thread
                                                                            // and staged vector

// False (and DEVERR_INDEX) when a row's token or item is out of range.
__device__ __forceinline__ bool row_valid(const RowMap& rm, int n_items, int tok, int item,
                                          unsigned* err, int lane) {
  if (tok < 0 || tok >= rm.n_tokens || item < 0 || item >= n_items) {
    if (lane == 0) atomicOr(err, DEVERR_INDEX);
    return false;
  }
  return true;
}

// Token and item of compact row r; false (and DEVERR_INDEX) when either is
// out of range.
__device__ __forceinline__ bool row_target(const RowMap& rm, int n_items, int r, int& tok,
                                           int& item, unsigned* err, int lane) {
  tok = rm.tok ? __ldg(rm.tok + r) : r;
  item = rm.item ? __ldg(rm.item + r) : 0;
  return row_valid(rm, n_items, tok, item, err, lane);
}

__global__ void __launch_bounds__(LN_WARPS * 32)
ln_mod_kernel(const float* __restrict__ x, const float* __restrict__ tab, int k_sh, int k_sc,
              const __grid_constant__ Items it, bf16* __restrict__ out, RowMap rm,
              long long hprev_off, int d, unsigned* err) {
  // shift and scale staged once per CTA: tab (+ the item's tb when the
  // launch has one item; otherwise each row adds its item's tb).  Loads that
  // do not depend on one another are all issued before any is used (the
  // vectors and the live row count, then the row with its token and item),
  // so a CTA waits for about two L2 round trips before its arithmetic.
  // The vectors and the row count are requested before the programmatic-
  // dependency wait: this kernel is never the first of a step or a block
  // call, and every kernel here waits for its predecessor before letting its
  // successor start, so whatever was written two or more launches earlier
  // (the modulation table and timestep vector, the dirty count) is complete
  // when this kernel starts; only the rows x come from the predecessor.
  extern __shared__ __align__(16) float s_mod[];  // [2][d]
  const int lane = threadIdx.x & 31;
  const int nv = d / 128, nq = d / 4;
  const float* tb0 = it.n == 1 ? it.tb[0] : nullptr;
  float4 m[4][LN_SV];  // tab shift, tab scale, tb shift, tb scale
#pragma unroll
  for (int j = 0; j < LN_SV; ++j) {
    const int q = threadIdx.x + j * LN_WARPS * 32;
#pragma unroll
    for (int u = 0; u < 4; ++u) m[u][j] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (q < nq && tab) {
      m[0][j] = __ldg(reinterpret_cast<const float4*>(tab + size_t(k_sh) * d) + q);
      m[1][j] = __ldg(reinterpret_cast<const float4*>(tab + size_t(k_sc) * d) + q);
    }
    if (q < nq && tb0) {
      m[2][j] = __ldg(reinterpret_cast<const float4*>(tb0 + size_t(k_sh) * d) + q);
      m[3][j] = __ldg(reinterpret_cast<const float4*>(tb0 + size_t(k_sc) * d) + q);
    }
  }
  const int D = live_count(rm.count, rm.bound, err);
  pdl_wait();
  pdl_trigger();
  int r = blockIdx.x * LN_WARPS + (threadIdx.x >> 5);
  float4 v[LN_MAXV];
  int tok = 0, item = 0;
  auto load_row = [&](int rr) {
    tok = rm.tok ? __ldg(rm.tok + rr) : rr;
    item = rm.item ? __ldg(rm.item + rr) : 0;
    const float4* xr = reinterpret_cast<const float4*>(x + size_t(rr) * d);
#pragma unroll
    for (int k = 0; k < LN_MAXV; ++k)
      if (k < nv) v[k] = xr[lane + 32 * k];
  };
  if (r < D) load_row(r);
#pragma unroll
  for (int j = 0; j < LN_SV; ++j) {
    const int q = threadIdx.x + j * LN_WARPS * 32;
    if (q < nq) {
      float4 a = m[0][j], b = m[1][j];
      if (tb0) {
        a.x += m[2][j].x; a.y += m[2][j].y; a.z += m[2][j].z; a.w += m[2][j].w;
        b.x += m[3][j].x; b.y += m[3][j].y; b.z += m[3][j].z; b.w += m[3][j].w;
      }
      reinterpret_cast<float4*>(s_mod)[q] = a;
      reinterpret_cast<float4*>(s_mod + d)[q] = b;
    }
  }
  __syncthreads();
  while (r < D) {
    if (row_valid(rm, it.n, tok, item, err, lane)) {
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < LN_MAXV; ++k)
        if (k < nv) s += (v[k].x + v[k].y) + (v[k].z + v[k].w);
      if (hprev_off >= 0) {
        uint2* hrow = reinterpret_cast<uint2*>(it.slice[item] + hprev_off + size_t(tok) * d);
#pragma unroll
        for (int k = 0; k < LN_MAXV; ++k)
          if (k < nv)
            hrow[lane + 32 * k] =
                make_uint2(pack_bf16x2(v[k].x, v[k].y), pack_bf16x2(v[k].z, v[k].w));
      }
      const float mean = warp_sum(s) / float(d);
      float q = 0.f;
#pragma unroll
      for (int k = 0; k < LN_MAXV; ++k)
        if (k < nv) {
          float a = v[k].x - mean, b = v[k].y - mean, c = v[k].z - mean, e = v[k].w - mean;
          q += (a * a + b * b) + (c * c + e * e);
        }
      const float rstd = 1.0f / sqrtf(warp_sum(q) / float(d) + 1e-6f);
      const float* tb = tb0 ? nullptr : it.tb[item];
      uint2* orow = reinterpret_cast<uint2*>(out + size_t(r) * d);
#pragma unroll
      for (int k = 0; k < LN_MAXV; ++k)
        if (k < nv) {
          const int c = 4 * (lane + 32 * k);
          float4 sh = *reinterpret_cast<const float4*>(s_mod + c);
          float4 sc = *reinterpret_cast<const float4*>(s_mod + d + c);
          if (tb) {
            const float4 a = *reinterpret_cast<const float4*>(tb + size_t(k_sh) * d + c);
            const float4 b = *reinterpret_cast<const float4*>(tb + size_t(k_sc) * d + c);
            sh.x += a.x; sh.y += a.y; sh.z += a.z; sh.w += a.w;
            sc.x += b.x; sc.y += b.y; sc.z += b.z; sc.w += b.w;
          }
          float y0 = (v[k].x - mean) * rstd * (1.f + sc.x) + sh.x;
          float y1 = (v[k].y - mean) * rstd * (1.f + sc.y) + sh.y;
          float y2 = (v[k].z - mean) * rstd * (1.f + sc.z) + sh.z;
          float y3 = (v[k].w - mean) * rstd * (1.f + sc.w) + sh.w;
          orow[lane + 32 * k] = make_uint2(pack_bf16x2(y0, y1), pack_bf16x2(y2, y3));
        }
    }
    r += gridDim.x * LN_WARPS;
    if (r < D) load_row(r);
  }
}

cudaError_t launch_ln_mod(const float* x, const float* tab, int k_sh, int k_sc, const Items& it,
                          bf16* out, const RowMap& rm, long long hprev_off, int d, unsigned* err,
                          cudaStream_t st) {
  if (rm.bound <= 0) return cudaSuccess;
  if (d % 128 || d > 128 * LN_MAXV) return cudaErrorInvalidValue;
  RC_TRY(launch_k(ln_mod_kernel, dim3(row_grid(rm.bound, LN_WARPS, 1)), dim3(LN_WARPS * 32),
                  size_t(2) * d * sizeof(float), st, x, tab, k_sh, k_sc, it, out, rm, hprev_off,
                  d, err));
  count_launches(1);
  return cudaSuccess;
}


// ============================================================ patch embed
// x_r = W_e patch(idx[r]) + b_e + pos[idx[r]], the patch vector ordered
// (channel, py, px).  W_e (<= 16 inputs per output) and b_e sit in shared
// memory; one warp per dirty token, grid-stride over the tokens.  A lane
// owns outputs lane + 32 m; a token's pos row (read from DRAM once per step)
// and its latent pixels are requested together before any is used, so a
// token costs one memory round trip instead of one per output group.
constexpr int PE_WARPS = 8;
constexpr int PE_MAXD = 1536;
constexpr int PE_MAXM = PE_MAXD / 32;  // outputs per lane

__global__ void __launch_bounds__(PE_WARPS * 32)
patch_embed_kernel(int gh, int gw, int p, int C, const bf16* __restrict__ We,
                   const float* __restrict__ be, const float* __restrict__ pos,
                   const __grid_constant__ Items it, RowMap rm, float* __restrict__ xf, int d,
                   unsigned* err) {
  // W_e and b_e are staged before the programmatic-dependency wait (weights
  // never change during a step); the latent, the row map and xf after it
  extern __shared__ __align__(16) uint8_t pe_smem[];
  bf16* s_w = reinterpret_cast<bf16*>(pe_smem);                    // [d][16], zero beyond P
  float* s_b = reinterpret_cast<float*>(pe_smem + size_t(d) * 32);  // [d]
  const int P = C * p * p;                                          // <= 16
  if (P == 16 && (reinterpret_cast<uintptr_t>(We) & 15u) == 0) {
    // rows of 16 weights are 32 bytes: a straight 16-byte copy, every load of
    // a thread in flight before its first store
    constexpr int NV = (PE_MAXD * 2 + PE_WARPS * 32 - 1) / (PE_WARPS * 32);
    uint4 t[NV];
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int v = threadIdx.x + j * PE_WARPS * 32;
      if (v < d * 2) t[j] = __ldg(reinterpret_cast<const uint4*>(We) + v);
    }
#pragma unroll
    for (int j = 0; j < NV; ++j) {
      const int v = threadIdx.x + j * PE_WARPS * 32;
      if (v < d * 2) reinterpret_cast<uint4*>(s_w)[v] = t[j];
    }
  } else {
    for (int e = threadIdx.x; e < d * 16; e += blockDim.x) {
      const int o = e >> 4, k = e & 15;
      s_w[e] = k < P ? We[size_t(o) * P + k] : f2bf(0.f);
    }
  }
  {
    constexpr int NB = (PE_MAXD + PE_WARPS * 32 - 1) / (PE_WARPS * 32);
    float t[NB];
#pragma unroll
    for (int j = 0; j < NB; ++j) {
      const int o = threadIdx.x + j * PE_WARPS * 32;
      if (o < d) t[j] = __ldg(be + o);
    }
#pragma unroll
    for (int j = 0; j < NB; ++j) {
      const int o = threadIdx.x + j * PE_WARPS * 32;
      if (o < d) s_b[o] = t[j];
    }
  }
  pdl_wait();
  pdl_trigger();
  __syncthreads();
  const int D = live_count(rm.count, rm.bound, err);
  const int lane = threadIdx.x & 31;
  const int W = gw * p, H = gh * p;
  const int nm = d / 32;
  for (int r = blockIdx.x * PE_WARPS + (threadIdx.x >> 5); r < D; r += gridDim.x * PE_WARPS) {
    int i, item;
    if (!row_target(rm, it.n, r, i, item, err, lane)) continue;
    const float* latent = it.latent[item];
    const int gy = i / gw, gx = i - gy * gw;
    float pv = 0.f;
    if (lane < P) {
      const int c = lane / (p * p), rem = lane - c * p * p;
      const int py = rem / p, px = rem - py * p;
      pv = latent[(size_t(c) * H + gy * p + py) * W + gx * p + px];
    }
    const float* prow = pos + size_t(i) * d;
    float pp[PE_MAXM];
#pragma unroll
    for (int m = 0; m < PE_MAXM; ++m)
      if (m < nm) pp[m] = __ldg(prow + lane + 32 * m);
    float patch[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) patch[k] = __shfl_sync(0xffffffffu, pv, k);
    float* xrow = xf + size_t(r) * d;
#pragma unroll
    for (int m = 0; m < PE_MAXM; ++m) {
      if (m >= nm) break;
      const int o = lane + 32 * m;
      const uint4* w4 = reinterpret_cast<const uint4*>(s_w + o * 16);
      float acc = 0.f;
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint4 w = w4[q];
        const float2 a = unpack_bf16x2(w.x), b = unpack_bf16x2(w.y);
        const float2 c2 = unpack_bf16x2(w.z), e2 = unpack_bf16x2(w.w);
        acc = fmaf(a.x, patch[8 * q], acc);
        acc = fmaf(a.y, patch[8 * q + 1], acc);
        acc = fmaf(b.x, patch[8 * q + 2], acc);
        acc = fmaf(b.y, patch[8 * q + 3], acc);
        acc = fmaf(c2.x, patch[8 * q + 4], acc);
        acc = fmaf(c2.y, patch[8 * q + 5], acc);
        acc = fmaf(e2.x, patch[8 * q + 6], acc);
        acc = fmaf(e2.y, patch[8 * q + 7], acc);
      }
      xrow[o] = acc + s_b[o] + pp[m];
    }
  }
}

cudaError_t launch_patch_embed(int gh, int gw, int p, int C, const bf16* We, const float* be,
                               const float* pos, const Items& it, const RowMap& rm, float* xf,
                               int d, unsigned* err, cudaStream_t st) {
  if (rm.bound <= 0) return cudaSuccess;
  if (d > PE_MAXD || d % 32 || C * p * p > 16) return cudaErrorInvalidValue;
  static bool attr_set = false;  // (55 KB at the largest hidden size)
  if (!attr_set) {
    RC_TRY(cudaFuncSetAttribute(patch_embed_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                int(size_t(PE_MAXD) * (16 * sizeof(bf16) + sizeof(float)))));
    attr_set = true;
  }
  RC_TRY(launch_k(patch_embed_kernel, dim3(row_grid(rm.bound, PE_WARPS, 1)), dim3(PE_WARPS * 32),
                  size_t(d) * (16 * sizeof(bf16) + sizeof(float)), st, gh, gw, p, C, We, be, pos,
                  it, rm, xf, d, err));
  count_launches(1);
  return cudaSuccess;
}

// ======================================================== timestep embed
// f[k] = cos(t w_k), f[half + k] = sin(t w_k), w_k = 10000^(-k/half); double
// precision for the argument so large timesteps keep their phase.
__global__ void sinusoid_kernel(float t, int dim, float* f) {
  pdl_wait();
  pdl_trigger();
  const int half = dim / 2;
  for (int k = threadIdx.x; k < half; k += blockDim.x) {
    double w = exp(-log(10000.0) * double(k) / double(half));
    double a = double(t) * w;
    f[k] = float(cos(a));
    f[half + k] = float(sin(a));
  }
}

// out[o] = sum_k W[o][k] act(in[k]) + b[o], act = SiLU when silu_in.  One warp
// per output; 16-byte weight loads.
__global__ void __launch_bounds__(256)
matvec_kernel(const bf16* __restrict__ W, const float* __restrict__ b,
              const float* __restrict__ in, float* __restrict__ out, int in_dim, int out_dim,
              int silu_in) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float s_in[];
  for (int k = threadIdx.x; k < in_dim; k += blockDim.x) {
    float v = in[k];
    s_in[k] = silu_in ? silu(v) : v;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int o = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (o >= out_dim) return;
  const bf16* w = W + size_t(o) * in_dim;
  float acc = 0.f;
  for (int k = lane * 8; k < in_dim; k += 256) {
    uint4 u = *reinterpret_cast<const uint4*>(w + k);
    float2 a0 = unpack_bf16x2(u.x), a1 = unpack_bf16x2(u.y);
    float2 a2 = unpack_bf16x2(u.z), a3 = unpack_bf16x2(u.w);
    acc = fmaf(a0.x, s_in[k + 0], acc);
    acc = fmaf(a0.y, s_in[k + 1], acc);
    acc = fmaf(a1.x, s_in[k + 2], acc);
    acc = fmaf(a1.y, s_in[k + 3], acc);
    acc = fmaf(a2.x, s_in[k + 4], acc);
    acc = fmaf(a2.y, s_in[k + 5], acc);
    acc = fmaf(a3.x, s_in[k + 6], acc);
    acc = fmaf(a3.y, s_in[k + 7], acc);
  }
  acc = warp_sum(acc);
  if (lane == 0) out[o] = acc + b[o];
}

cudaError_t launch_t_embed(float t_value, int freq_dim, int d, const bf16* Wt1, const float* bt1,
                           const bf16* Wt2, const float* bt2, const bf16* Wtb, const float* btb,
                           float* fbuf, float* h1, float* temb, float* tb, cudaStream_t st) {
  RC_TRY(launch_k(sinusoid_kernel, dim3(1), dim3(128), 0, st, t_value, freq_dim, fbuf));
  RC_TRY(launch_k(matvec_kernel, dim3(cdiv(d, 8)), dim3(256), freq_dim * sizeof(float), st, Wt1,
                  bt1, fbuf, h1, freq_dim, d, 0));
  RC_TRY(launch_k(matvec_kernel, dim3(cdiv(d, 8)), dim3(256), d * sizeof(float), st, Wt2, bt2, h1,
                  temb, d, d, 1));
  RC_TRY(launch_k(matvec_kernel, dim3(cdiv(6 * d, 8)), dim3(256), d * sizeof(float), st, Wtb, btb,
                  temb, tb, d, 6 * d, 1));
  count_launches(4);
  return cudaSuccess;
}

// ===================================================== final layer + DDIM
// One warp per token.  The eps outputs (py, px, c < c_in) of the final linear
// are computed for all tokens from the last block's hidden state; each updates
// one latent element: x0 = (x - sqrt(1-ab_t) eps) / sqrt(ab_t),
// x' = sqrt(ab_next) x0 + sqrt(1-ab_next) eps.
constexpr int FIN_WARPS = 8;
constexpr int FIN_MAXV = 12;  // 4-element groups per lane (hidden <= 1536)
constexpr int FIN_MAXO = 16;  // eps outputs per token (p*p*c_in)

__global__ void __launch_bounds__(FIN_WARPS * 32)
final_ddim_kernel(const bf16* __restrict__ H, const float* __restrict__ temb,
                  const float* __restrict__ table_f, const bf16* __restrict__ Wf,
                  const float* __restrict__ bfin, float* __restrict__ latent, int gh, int gw,
                  int p, int c_in, int c_out, int d, float ab_t, float ab_next) {
  // the modulation vectors and the eps rows of W_f are staged before the
  // programmatic-dependency wait: the weights never change during a step and
  // temb was written at its start, two or more launches earlier (every
  // kernel of the library waits for its predecessor before letting its
  // successor start); H and the latent are read after the wait
  extern __shared__ uint8_t smem_raw[];
  float* s_shift = reinterpret_cast<float*>(smem_raw);
  float* s_scale = s_shift + d;
  bf16* s_w = reinterpret_cast<bf16*>(s_scale + d);  // [n_eps][d]
  const int n_eps = p * p * c_in;
  // every load of a thread is issued before its first store (a loop of
  // dependent load / store pairs would wait one memory round trip each)
  {
    constexpr int NC = (FIN_MAXV * 128 + FIN_WARPS * 32 - 1) / (FIN_WARPS * 32);
    float a[NC], b[NC], e[NC];
#pragma unroll
    for (int j = 0; j < NC; ++j) {
      const int c = threadIdx.x + j * FIN_WARPS * 32;
      if (c < d) {
        a[j] = table_f[c];
        b[j] = table_f[d + c];
        e[j] = temb[c];
      }
    }
#pragma unroll
    for (int j = 0; j < NC; ++j) {
      const int c = threadIdx.x + j * FIN_WARPS * 32;
      if (c < d) {
        s_shift[c] = a[j] + e[j];
        s_scale[c] = b[j] + e[j];
      }
    }
  }
  // the eps rows of W_f, 16 bytes per thread and step (d % 8 == 0)
  const int d8 = d / 8;
  {
    constexpr int NW = (FIN_MAXO * FIN_MAXV * 16 + FIN_WARPS * 32 - 1) / (FIN_WARPS * 32);
    uint4 t[NW];
#pragma unroll
    for (int j = 0; j < NW; ++j) {
      const int v = threadIdx.x + j * FIN_WARPS * 32;
      if (v < n_eps * d8) {
        const int e = v / d8, c8 = v - e * d8;
        const int sub = e / c_in, ch = e - sub * c_in;
        t[j] = __ldg(reinterpret_cast<const uint4*>(Wf + size_t(sub * c_out + ch) * d) + c8);
      }
    }
#pragma unroll
    for (int j = 0; j < NW; ++j) {
      const int v = threadIdx.x + j * FIN_WARPS * 32;
      if (v < n_eps * d8) {
        const int e = v / d8, c8 = v - e * d8;
        reinterpret_cast<uint4*>(s_w + size_t(e) * d)[c8] = t[j];
      }
    }
  }
  pdl_wait();
  pdl_trigger();
  __syncthreads();
  const int N = gh * gw;
  const int lane = threadIdx.x & 31;
  const int nv = d / 128;
  const float sa = sqrtf(ab_t), sn = sqrtf(1.f - ab_t);
  const float ta = sqrtf(ab_next), tn = sqrtf(1.f - ab_next);
  const int W = gw * p, Hh = gh * p;
  for (int i = blockIdx.x * FIN_WARPS + (threadIdx.x >> 5); i < N; i += gridDim.x * FIN_WARPS) {
    const uint2* hr = reinterpret_cast<const uint2*>(H + size_t(i) * d);
    float y[FIN_MAXV][4];
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < FIN_MAXV; ++k)
      if (k < nv) {
        uint2 u = hr[lane + 32 * k];
        float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
        y[k][0] = a.x; y[k][1] = a.y; y[k][2] = b.x; y[k][3] = b.y;
        s += (a.x + a.y) + (b.x + b.y);
      }
    const float mean = warp_sum(s) / float(d);
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < FIN_MAXV; ++k)
      if (k < nv)
#pragma unroll
        for (int j = 0; j < 4; ++j) { float a = y[k][j] - mean; q += a * a; }
    const float rstd = 1.0f / sqrtf(warp_sum(q) / float(d) + 1e-6f);
#pragma unroll
    for (int k = 0; k < FIN_MAXV; ++k)
      if (k < nv)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int c = 4 * (lane + 32 * k) + j;
          y[k][j] = (y[k][j] - mean) * rstd * (1.f + s_scale[c]) + s_shift[c];
        }
    const int gy = i / gw, gx = i - gy * gw;
    // all eps dot products first (independent reductions), then one batched
    // latent update: lane e < n_eps owns output e
    float acc[FIN_MAXO];
#pragma unroll
    for (int e = 0; e < FIN_MAXO; ++e) {
      acc[e] = 0.f;
      if (e < n_eps) {
        const bf16* w = s_w + size_t(e) * d;
#pragma unroll
        for (int k = 0; k < FIN_MAXV; ++k)
          if (k < nv) {
            const int c = 4 * (lane + 32 * k);
            uint2 u = *reinterpret_cast<const uint2*>(w + c);
            float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
            acc[e] = fmaf(y[k][0], a.x, acc[e]);
            acc[e] = fmaf(y[k][1], a.y, acc[e]);
            acc[e] = fmaf(y[k][2], b.x, acc[e]);
            acc[e] = fmaf(y[k][3], b.y, acc[e]);
          }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int e = 0; e < FIN_MAXO; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    float mine = 0.f;
#pragma unroll
    for (int e = 0; e < FIN_MAXO; ++e)
      if (lane == e) mine = acc[e];
    if (lane < n_eps) {
      const int sub = lane / c_in, ch = lane - (lane / c_in) * c_in;
      const int py = sub / p, px = sub - py * p;
      const float eps = mine + bfin[sub * c_out + ch];
      float* xp = latent + (size_t(ch) * Hh + gy * p + py) * W + gx * p + px;
      const float x0 = (*xp - sn * eps) / sa;
      *xp = ta * x0 + tn * eps;
    }
  }
}

cudaError_t launch_final_ddim(const bf16* H, const float* temb, const float* table_f,
                              const bf16* Wf, const float* bf, float* latent, int gh, int gw,
                              int p, int c_in, int c_out, int d, float ab_t, float ab_next,
                              cudaStream_t st) {
  const int n_eps = p * p * c_in;
  const size_t smem = size_t(2) * d * sizeof(float) + size_t(n_eps) * d * sizeof(bf16);
  static bool attr_set = false;
  if (!attr_set) {
    cudaFuncSetAttribute(final_ddim_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         64 * 1024);
    attr_set = true;
  }
  const int N = gh * gw;
  // a warp per token (grid-stride): the per-token reductions are
  // latency-bound chains.  One wave of CTAs (two fit an SM by their
  // registers), so that each SM stages W_f and the modulation once per CTA
  // it holds rather than once per token group
  int grid = cdiv(N, FIN_WARPS);
  const int cap = 2 * device_sm_count();
  if (grid > cap) grid = cap;
  RC_TRY(launch_k(final_ddim_kernel, dim3(grid), dim3(FIN_WARPS * 32), smem, st, H, temb, table_f,
                  Wf, bf, latent, gh, gw, p, c_in, c_out, d, ab_t, ab_next));
  count_launches(1);
  return cudaSuccess;
}

// ======================================================= gather / scatter
// One warp per row, grid-stride over the rows.
constexpr int RW_WARPS = 8;

__global__ void __launch_bounds__(RW_WARPS * 32)
rows_f32_kernel(const float* __restrict__ src, float* __restrict__ dst,
                const int* __restrict__ idx, int Dbound, const int* __restrict__ dcount, int d,
                int N, int scatter, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int D = live_count(dcount, Dbound, err);
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * RW_WARPS + (threadIdx.x >> 5); r < D; r += gridDim.x * RW_WARPS) {
    const int i = idx[r];
    if (i < 0 || i >= N) {
      if (lane == 0) atomicOr(err, DEVERR_INDEX);
      continue;
    }
    const float4* s4 = reinterpret_cast<const float4*>(src + size_t(scatter ? r : i) * d);
    float4* t4 = reinterpret_cast<float4*>(dst + size_t(scatter ? i : r) * d);
    for (int c = lane; c < d / 4; c += 32) t4[c] = s4[c];
  }
}

__global__ void __launch_bounds__(RW_WARPS * 32)
scatter_bf16_kernel(const float* __restrict__ src, const __grid_constant__ Items it,
                    long long off, RowMap rm, int d, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int D = live_count(rm.count, rm.bound, err);
  const int lane = threadIdx.x & 31;
  for (int r = blockIdx.x * RW_WARPS + (threadIdx.x >> 5); r < D; r += gridDim.x * RW_WARPS) {
    int i, item;
    if (!row_target(rm, it.n, r, i, item, err, lane)) continue;
    const float4* s4 = reinterpret_cast<const float4*>(src + size_t(r) * d);
    uint2* t2 = reinterpret_cast<uint2*>(it.slice[item] + off + size_t(i) * d);
    for (int c = lane; c < d / 4; c += 32) {
      const float4 v = s4[c];
      t2[c] = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
    }
  }
}

// Host-tier write-back of one layer: the dirty rows tok[r] of the HBM window
// [H,K,V][N][d] go to the same rows of the host slice (device-mapped
// addresses); one warp per row, 16-byte accesses.  It runs beside the next
// layer's kernels, which fill the SMs' registers, so its CTAs are single
// warps that still fit next to them.
__global__ void __launch_bounds__(32)
writeback_kernel(const bf16* __restrict__ win, bf16* host, RowMap rm, int d, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int D = live_count(rm.count, rm.bound, err);
  const int lane = threadIdx.x & 31;
  const size_t Nd = size_t(rm.n_tokens) * d;
  for (int r = blockIdx.x; r < D; r += gridDim.x) {
    const int i = rm.tok ? __ldg(rm.tok + r) : r;
    if (i < 0 || i >= rm.n_tokens) {
      if (lane == 0) atomicOr(err, DEVERR_INDEX);
      continue;
    }
    for (int part = 0; part < 3; ++part) {
      const uint4* src = reinterpret_cast<const uint4*>(win + part * Nd + size_t(i) * d);
      uint4* dst = reinterpret_cast<uint4*>(host + part * Nd + size_t(i) * d);
      for (int c = lane; c < d / 8; c += 32) dst[c] = src[c];
    }
  }
}

cudaError_t launch_writeback(const bf16* win, bf16* host, const RowMap& rm, int d, unsigned* err,
                             cudaStream_t st) {
  if (rm.bound <= 0) return cudaSuccess;
  const int grid = rm.bound < 4 * device_sm_count() ? rm.bound : 4 * device_sm_count();
  RC_TRY(launch_k(writeback_kernel, dim3(grid), dim3(32), 0, st, win, host, rm, d, err));
  count_launches(1);
  return cudaSuccess;
}

// Concatenated rows of a multi-item step: block (x, i) fills rows of item i.
__global__ void __launch_bounds__(256)
batch_rows_kernel(const __grid_constant__ BatchIn in, int* __restrict__ tok,
                  int* __restrict__ item, int* __restrict__ meta, int n_tokens, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int i = blockIdx.y;
  int off = 0, tiles = 0, cnt = 0;
  for (int j = 0; j <= i; ++j) {
    int c = in.bound[j];
    if (in.count[j]) {
      c = *in.count[j];
      if (c < 0 || c > in.bound[j]) {
        if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(err, DEVERR_COUNT);
        c = 0;
      }
    }
    if (j < i) {
      off += c;
      tiles += (c + 127) / 128;
    } else {
      cnt = c;
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    meta[META_OFF + i] = off;
    meta[META_CNT + i] = cnt;
    meta[META_TILE + i] = tiles;
    if (i == in.n - 1) {
      meta[META_TOTAL] = off + cnt;
      meta[META_TILE + in.n] = tiles + (cnt + 127) / 128;
    }
  }
  const int* idx = in.idx[i];
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < cnt; r += gridDim.x * blockDim.x) {
    const int t = idx ? idx[r] : r;
    if (t < 0 || t >= n_tokens) atomicOr(err, DEVERR_INDEX);
    tok[off + r] = t;
    item[off + r] = i;
  }
}

cudaError_t launch_batch_rows(const BatchIn& in, int* tok, int* item, int* meta, int n_tokens,
                              unsigned* err, cudaStream_t st) {
  if (in.n <= 0 || in.n > MAX_ITEMS) return cudaErrorInvalidValue;
  int maxb = 1;
  for (int j = 0; j < in.n; ++j) maxb = maxb > in.bound[j] ? maxb : in.bound[j];
  const int gx = cdiv(maxb, 256) < 16 ? cdiv(maxb, 256) : 16;
  RC_TRY(launch_k(batch_rows_kernel, dim3(gx, in.n), dim3(256), 0, st, in, tok, item, meta,
                  n_tokens, err));
  count_launches(1);
  return cudaSuccess;
}

cudaError_t launch_rows_f32(const float* src, float* dst, const int* idx, int Dbound,
                            const int* dcount, int d, int N, bool scatter, unsigned* err,
                            cudaStream_t st) {
  if (Dbound <= 0) return cudaSuccess;
  RC_TRY(launch_k(rows_f32_kernel, dim3(row_grid(Dbound, RW_WARPS, 4)), dim3(RW_WARPS * 32), 0, st,
                  src, dst, idx, Dbound, dcount, d, N, scatter ? 1 : 0, err));
  count_launches(1);
  return cudaSuccess;
}

cudaError_t launch_scatter_bf16(const float* src, const Items& it, long long off,
                                const RowMap& rm, int d, unsigned* err, cudaStream_t st) {
  if (rm.bound <= 0) return cudaSuccess;
  RC_TRY(launch_k(scatter_bf16_kernel, dim3(row_grid(rm.bound, RW_WARPS, 1)), dim3(RW_WARPS * 32),
                  0, st, src, it, off, rm, d, err));
  count_launches(1);
  return cudaSuccess;
}

}  // namespace rc
