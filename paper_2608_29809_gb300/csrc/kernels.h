// Internal launchers of the region-sparse DiT library.  Every launcher queues
// one or more kernels on `st` and returns the cudaError_t of the launch.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

struct rc_ctx;
struct rc_cache;

namespace rc {

typedef __nv_bfloat16 bf16;

// Kernels launched by this library in this process (reported by rc_launch_count).
void count_launches(int n);

// Sets the calling thread's rc_last_error() text.
void set_last_error(const char* msg);

// Facts about a context / cache for host code outside regioncache.cu.
int ctx_max_batch(const ::rc_ctx* c);
int ctx_timesteps(const ::rc_ctx* c);
const ::rc_ctx* cache_context(const ::rc_cache* k);
int cache_sessions(const ::rc_cache* k);
bool cache_host_tier(const ::rc_cache* k);

// ------------------------------------------------------------- localisation
struct DeltaIds {
  int n;
  int id[64];
};
size_t localize_workspace_bytes(int N, int n_delta);
cudaError_t launch_localize(const float* A, int S, int N, int M, int gh, int gw,
                            const DeltaIds& ids, float tau, int dilation, uint8_t* mask,
                            int32_t* idx, int32_t* count, void* ws, cudaStream_t st);

// ------------------------------------------------------------- step rows
// A step processes one or more items (an item = one session's denoising
// step).  Their dirty rows are concatenated into one compact row space: item
// i owns rows [off_i, off_i + cnt_i) and row r is token tok[r] of item item[r].
constexpr int MAX_ITEMS = 16;
enum {
  META_TOTAL = 0,                     // rows of all items
  META_OFF = 1,                       // off[i]
  META_CNT = 1 + MAX_ITEMS,           // cnt[i]
  META_TILE = 1 + 2 * MAX_ITEMS,      // first 128-row query tile of item i; [n] = all tiles
  META_INTS = 2 + 3 * MAX_ITEMS
};
struct RowMap {
  const int* tok;    // [rows] token of row r (null: row r is token r)
  const int* item;   // [rows] item of row r (null: every row is item 0)
  const int* meta;   // device META_* table (null: a single item holding every row)
  int bound;         // host bound of the row count
  const int* count;  // device row count (null: bound)
  int n_tokens;      // N; token indices outside [0, N) raise DEVERR_INDEX
};
// Per-item addressing (passed by value).
struct Items {
  int n;
  bf16* slice[MAX_ITEMS];      // the item's (session, t) cache slice [L][H,K,V][N][d]
  const float* tb[MAX_ITEMS];  // modulation [6][d] of the item's timestep (null: none)
  float* latent[MAX_ITEMS];    // the item's latent (patch embedding input)
};
// Host-tier write-back of a layer: rows tok[r] of the HBM window [H,K,V][N][d]
// go to the same rows of the host slice (device-mapped).
cudaError_t launch_writeback(const bf16* win, bf16* host, const RowMap& rm, int d, unsigned* err,
                             cudaStream_t st);

// Builds tok / item / meta of a multi-item step.  Item i contributes cnt_i =
// min(*count_i, bound_i) rows (count_i null: bound_i) taken from idx_i (null:
// tokens 0 .. cnt_i - 1).
struct BatchIn {
  int n;
  const int* idx[MAX_ITEMS];
  const int* count[MAX_ITEMS];
  int bound[MAX_ITEMS];
};
cudaError_t launch_batch_rows(const BatchIn& in, int* tok, int* item, int* meta, int n_tokens,
                              unsigned* err, cudaStream_t st);

// --------------------------------------------------------------- row kernels
// out[r] = bf16(LN(x[r]) (1 + scale) + shift) for live rows r, with
// shift = tab[k_sh] (+ tb_item[k_sh]), scale = tab[k_sc] (+ tb_item[k_sc])
// ([6][d] vectors; tab may be null).  With hprev_off >= 0 the row itself is
// also stored as bf16 to the item's cache slice at element offset
// hprev_off + tok[r] * d (the previous block's merged hidden state, Section 3.3).
cudaError_t launch_ln_mod(const float* x, const float* tab, int k_sh, int k_sc, const Items& it,
                          bf16* out, const RowMap& rm, long long hprev_off, int d, unsigned* err,
                          cudaStream_t st);

// xf[r] = W_e patch(tok[r]) + b_e + pos[tok[r]], the patch from the row's item latent.
cudaError_t launch_patch_embed(int gh, int gw, int p, int C, const bf16* We, const float* be,
                               const float* pos, const Items& it, const RowMap& rm, float* xf,
                               int d, unsigned* err, cudaStream_t st);

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
// item slice + off + tok[r] * d  <-  bf16(src[r]), f32 rows -> bf16 cache rows.
cudaError_t launch_scatter_bf16(const float* src, const Items& it, long long off,
                                const RowMap& rm, int d, unsigned* err, cudaStream_t st);

// ---------------------------------------------------------------------- GEMM
// EPI_GATE_RES: xf += gate (acc + b) as reductions (tiles may be split);
// EPI_GATE_RES_CAST: the same on whole tiles, then out_bf = bf16(xf).
enum EpiMode {
  EPI_F32 = 0,
  EPI_BIAS_BF16 = 1,
  EPI_GELU_BF16 = 2,
  EPI_GATE_RES = 3,
  EPI_QKV = 4,
  EPI_GATE_RES_CAST = 5
};

struct GemmEpi {
  int mode;
  const float* bias;       // [n] or null
  bf16* out_bf;            // BIAS_BF16 / GELU_BF16 / QKV (q part)
  int ld_out;
  float* out_f;            // F32
  float* xf;               // GATE_RES residual, f32
  int ld_xf;
  const float* gate_tab;   // gate = gate_tab[c] (+ tb_item[gate_off + c]); null tab = no gate
  long long gate_off;      // element offset of the gate in the item tb vectors (-1: none)
  long long k_off, v_off;  // QKV: K / V rows at item slice + k_off / v_off + tok * dsplit
  int dsplit;              // QKV: hidden size (q | k | v boundaries)
  const int* tok;          // row -> token (null: identity)
  const int* item;         // row -> item (null: item 0)
  int n_tokens;            // bound of token indices
  unsigned* err;
  Items its;               // per-item cache slices and modulation vectors
  int whole_tiles;         // GATE_RES: no k split (one reduction per element, reproducible)
};

// C[M][n] = A[M][k] W[n][k]^T, epilogue `ep`.  M = *dcount if non-null (bounded
// by Mbound) else Mbound.  n % 64 == 0, k % 64 == 0.
cudaError_t launch_gemm(const bf16* A, int lda, const bf16* W, int Mbound, const int* dcount,
                        int n, int k, const GemmEpi& ep, cudaStream_t st);


// ----------------------------------------------------------------- attention
// Key-split scratch of one context: partial outputs of the key splits.
struct AttnScratch {
  float* part;
  size_t part_floats;
};
size_t attention_split_floats(int Nmax, int heads, int dh);

// Per-item key / value placement of one attention launch: item i's keys are
// rows krow[i] .. krow[i] + Nk - 1 of K (values likewise from vrow[i] of V).
struct AttnItems {
  int n;
  int krow[MAX_ITEMS];
  int vrow[MAX_ITEMS];
};

// Capture of attention probabilities (the localisation scores of Section
// 3.2): for each listed key column id[q], out[tok(r)][id[q]] += w * P[r][id[q]]
// over every head of the launch (P the softmax probability of that key for
// query row r).  Needs all keys in one unit per (query tile, head), i.e. the
// short text cross-attention.
struct AttnCapture {
  int n;         // listed columns, 0 .. 8 (0: no capture)
  int id[8];
  float* out;    // [tokens][ldo]
  int ldo;
  float w;
};

// O[r][h*dh..] = softmax(Q_r K_i^T / sqrt(dh)) V_i per head over the Nk keys of
// row r's item i.  Q and O are compact rows (rm); K / V are row-major with row
// stride ldkv and kv_rows rows in all.  Keys beyond Nk are masked, but their
// values must be finite (they are multiplied by zero).
cudaError_t launch_attention(const bf16* Q, int ldq, const bf16* K, const bf16* V, int ldkv,
                             int kv_rows, const AttnItems& ai, int Nk, bf16* O, int ldo, int heads,
                             int dh, const RowMap& rm, unsigned* err, const AttnScratch& as,
                             cudaStream_t st, const AttnCapture* cap = nullptr);

// Text cross-attention with the query projection folded into the keys:
// S_h = xb W_xq,h^T K_h^T + b_h K_h^T = xb G_h^T + kb_h with G_h = K_h W_xq,h
// ([XK][d] per (session, layer, head), rows >= text_len zero) and
// kb_h = K_h b_xq,h.  launch_xq_fold computes G and kb of one (session,
// layer) for all heads from the text keys (row stride ldk) and W_xq, b_xq.
constexpr int XQ_KEYS = 128;
cudaError_t launch_xq_fold(const bf16* Kt, int ldk, const bf16* Wq, const float* bq, int M,
                           int heads, int dh, int d, bf16* G, float* kb, cudaStream_t st);
// O[r][h*dh..] = softmax((xb_r G_h^T + kb_h) / sqrt(dh)) V_h over the Nk <= 128
// text keys of row r's item.  G / kb rows of item i start at grow[i] (+ h *
// XQ_KEYS); its values at row vrow[i] of V (row stride ldv).  cap as in
// launch_attention.
struct XqItems {
  int n;
  int grow[MAX_ITEMS];
  int vrow[MAX_ITEMS];
};
cudaError_t launch_xattn_fused(const bf16* xb, int ldx, const bf16* G, const float* kb, int g_rows,
                               const bf16* V, int ldv, int v_rows, const XqItems& xi, int Nk,
                               bf16* O, int ldo, int heads, int dh, const RowMap& rm,
                               unsigned* err, cudaStream_t st, const AttnCapture* cap);

}  // namespace rc
