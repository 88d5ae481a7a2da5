// Internal launchers of the region-sparse DiT library.  Every launcher queues
// one or more kernels on `st` and returns the cudaError_t of the launch.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace rc {

typedef __nv_bfloat16 bf16;

// Kernels launched by this library in this process (reported by rc_launch_count).
void count_launches(int n);
// Sets the calling thread's rc_last_error() text.
void set_last_error(const char* msg);

// ------------------------------------------------------------- localisation
struct DeltaIds {
  int n;
  int id[64];
};
size_t localize_workspace_bytes(int N, int n_delta);
cudaError_t launch_localize(const float* A, int S, int N, int M, int gh, int gw,
                            const DeltaIds& ids, float tau, int dilation, uint8_t* mask,
                            int32_t* idx, int32_t* count, void* ws, cudaStream_t st);

// --------------------------------------------------------------- row kernels
// out[r] = bf16(LN(x[r]) * (1 + scale) + shift) for r < D; scale = tab_sc (+ tb_sc),
// shift = tab_sh (+ tb_sh) (the tb_* terms may be null).  With hprev non-null
// the row itself is also stored as bf16 to hprev[idx[r]] (the previous
// block's merged hidden state, Section 3.3).
cudaError_t launch_ln_mod(const float* x, int ldx, const float* tab_sh, const float* tb_sh,
                          const float* tab_sc, const float* tb_sc, bf16* out, int ldo,
                          int Dbound, const int* dcount, int d, bf16* hprev, const int* idx,
                          int n_tokens, unsigned* err, cudaStream_t st);
// out[r] = bf16(x[r]) for r < D.
cudaError_t launch_cast_rows(const float* x, int ldx, bf16* out, int ldo, int Dbound,
                             const int* dcount, int d, unsigned* err, cudaStream_t st);

// xf[r] = W_e patch(idx[r]) + b_e + pos[idx[r]]  (idx null: identity)
cudaError_t launch_patch_embed(const float* latent, int gh, int gw, int p, int C,
                               const bf16* We, const float* be, const float* pos,
                               const int* idx, int Dbound, const int* dcount, float* xf, int d,
                               unsigned* err, cudaStream_t st);

// Timestep embedding chain: f = sinusoid(t_value); h1 = W_t1 f + b; temb = W_t2 silu(h1) + b;
// tb = W_tb silu(temb) + b.  scratch h1/f are caller buffers.
cudaError_t launch_t_embed(float t_value, int freq_dim, int d, const bf16* Wt1, const float* bt1,
                           const bf16* Wt2, const float* bt2, const bf16* Wtb, const float* btb,
                           float* fbuf, float* h1, float* temb, float* tb, cudaStream_t st);

// Final layer over all N tokens of H (bf16 [N][d]) + DDIM update of latent.
cudaError_t launch_final_ddim(const bf16* H, const float* temb, const float* table_f,
                              const bf16* Wf, const float* bf, float* latent, int gh, int gw,
                              int p, int c_in, int c_out, int d, float ab_t, float ab_next,
                              cudaStream_t st);

// dst[r] = src[idx[r]] (gather) or dst[idx[r]] = src[r] (scatter), f32 rows of d.
cudaError_t launch_rows_f32(const float* src, float* dst, const int* idx, int Dbound,
                            const int* dcount, int d, int N, bool scatter, unsigned* err,
                            cudaStream_t st);
// dst[idx[r]] = bf16(src[r]), f32 rows -> bf16 rows.
cudaError_t launch_scatter_bf16(const float* src, bf16* dst, const int* idx, int Dbound,
                                const int* dcount, int d, int N, unsigned* err, cudaStream_t st);

// ---------------------------------------------------------------------- GEMM
enum EpiMode { EPI_F32 = 0, EPI_BIAS_BF16 = 1, EPI_GELU_BF16 = 2, EPI_GATE_RES = 3, EPI_QKV = 4 };

struct GemmEpi {
  int mode;
  const float* bias;       // [n] or null
  bf16* out_bf;            // BIAS_BF16 / GELU_BF16 / QKV (q part)
  int ld_out;
  float* out_f;            // F32
  float* xf;               // GATE_RES residual, f32
  int ld_xf;
  const float* gate_tab;   // gate = gate_tab[c] (+ gate_tb[c]); null tab = no gate
  const float* gate_tb;
  bf16* kc;                // QKV: K rows idx[r] (cache)
  bf16* vc;                // QKV: V rows idx[r] (cache)
  int ld_kv;
  int dsplit;              // QKV: hidden size (q | k | v boundaries)
  const int* idx;          // row -> token index (null: identity)
  int n_tokens;            // bound of idx values
  unsigned* err;
};

// C[M][n] = A[M][k] W[n][k]^T, epilogue `ep`.  M = *dcount if non-null (bounded
// by Mbound) else Mbound.  n % 128 == 0, k % 64 == 0.
cudaError_t launch_gemm(const bf16* A, int lda, const bf16* W, int Mbound, const int* dcount,
                        int n, int k, const GemmEpi& ep, cudaStream_t st);


// ----------------------------------------------------------------- attention
// Key-split scratch of one context: partial outputs of the key splits.
struct AttnScratch {
  float* part;
  size_t part_floats;
};
size_t attention_split_floats(int Nmax, int heads, int dh);

// O[r][h*dh..] = softmax(Q_r K^T / sqrt(dh)) V per head, over Nk keys.
// Q/O compact rows (r < D), K/V rows 0..Nk-1 with row stride ldkv.
cudaError_t launch_attention(const bf16* Q, int ldq, const bf16* K, const bf16* V, int ldkv,
                             int Nk, bf16* O, int ldo, int heads, int dh, int Dbound,
                             const int* dcount, unsigned* err, const AttnScratch& as,
                             cudaStream_t st);

}  // namespace rc
