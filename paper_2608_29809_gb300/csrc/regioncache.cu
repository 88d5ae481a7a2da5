// C ABI of the region-sparse DiT step (see include/regioncache.h): context and
// cache management, host-side validation, and the launch sequence of a block
// and a denoising step.  Every compute step runs in this library's kernels.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>
#include <sys/mman.h>

#include <atomic>
#include <cmath>
#include <new>
#include <string>
#include <vector>

#include "../../include/regioncache.h"
#include "common.cuh"
#include "kernels.h"

using rc::bf16;

namespace {

thread_local std::string g_last_error;
std::atomic<uint64_t> g_launches{0};

rc_status fail(rc_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

rc_status cuda_fail(cudaError_t e, const char* what) {
  return fail(e == cudaErrorMemoryAllocation ? RC_ERR_OOM : RC_ERR_CUDA, "%s: %s", what,
              cudaGetErrorString(e));
}

#define RC_CUDA(call, what)                        \
  do {                                             \
    cudaError_t e_ = (call);                       \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace rc {
void count_launches(int n) { g_launches.fetch_add(uint64_t(n), std::memory_order_relaxed); }
void set_last_error(const char* msg) { g_last_error = msg; }
}  // namespace rc

struct rc_ctx {
  rc_dims dims;
  int N, d, F, dh, L, T, M;
  int max_batch;  // items per batched step; row scratch = max_batch * N rows
  int device;
  std::vector<rc_layer_weights> lw;
  std::vector<char> lw_set;
  // bumped by every rc_set_layer_weights: a session's text keys (and the
  // folded cross-query keys derived from them) are valid only for the
  // generation they were computed with
  uint64_t wgen = 0;
  rc_global_weights gw;
  bool gw_set = false;
  std::vector<float> t_values, alpha_bar;
  bool sched_set = false;
  // gated residual GEMMs on whole tiles only (rc_set_deterministic)
  bool deterministic = false;
  // device scratch (R = max_batch * N compact rows)
  float* xf = nullptr;   // [R][d] residual rows of the dirty tokens (compact)
  bf16* xb = nullptr;    // [R][d] GEMM input: modulated rows / residual copy
  bf16* ob = nullptr;    // [R][d] attention output
  bf16* q = nullptr;     // [R][d] queries (self, then cross)
  bf16* u = nullptr;     // [R][F] MLP hidden
  float* fbuf = nullptr; // [freq_dim]
  float* h1 = nullptr;   // [d]
  float* temb = nullptr; // [RC_MAX_BATCH][d] timestep embedding per item
  float* tb = nullptr;   // [RC_MAX_BATCH][6d] t_block modulation per item
  // the same for every scheduled timestep, [T][d] and [T][6d]: they depend
  // only on the global weights and the schedule, so they are computed once
  // (t_ready) and reused by every step
  float* temb_tab = nullptr;
  float* tb_tab = nullptr;
  bool t_ready = false;
  int* iota = nullptr;   // [N] identity row map (dense path)
  int* b_tok = nullptr;  // [R] token of each compact row (batched steps)
  int* b_item = nullptr; // [R] item of each compact row (batched steps)
  int* b_meta = nullptr; // [META_INTS] row offsets / counts / query tiles per item
  unsigned* err = nullptr;
  unsigned* wait_flag = nullptr;  // the self-test's flag (rc_selftest_wait)
  rc::AttnScratch as{};  // key-split partial outputs
  // timing probe
  int probe_which = RC_PROBE_OFF;
  int probe_n = 0;
  std::vector<cudaEvent_t> probe_ev;  // 2 * capacity
};

struct rc_cache {
  rc_ctx* ctx;
  int sessions;
  bf16* base = nullptr;  // [sessions][T][L][3 (H,K,V)][N][d] (device-addressable)
  bf16* text = nullptr;  // [sessions][L][M][2d], always in HBM
  // the text keys with the cross-query projection folded in (HBM):
  // xg [sessions][L][heads][XQ_KEYS][d] = K_h W_xq,h, xgb [..][XQ_KEYS] = K_h b_xq,h
  bf16* xg = nullptr;
  float* xgb = nullptr;
  std::vector<char> text_set;
  std::vector<uint64_t> text_gen;  // the context's weight generation at rc_set_text / import
  // host tier (Section 3.4, Pipelined Execution): the slots live in pinned,
  // mapped host memory (base is its device address).  A step runs layer l on
  // HBM window l % 3: the copy stream loads layer l + 2's cached K, V into
  // its window while layer l computes, and the write-back stream sends layer
  // l - 1's dirty H, K, V rows back to host memory
  static constexpr int WINDOWS = 3;
  bool host_tier = false;
  void* host_mem = nullptr;    // the pool: an anonymous mapping, page-locked
  void* host_map = nullptr;    // the mapping as made (host_mem is aligned inside)
  size_t host_map_bytes = 0;
  bf16* window = nullptr;  // [WINDOWS][3][N][d]
  cudaStream_t copy_st = nullptr, copy_st2 = nullptr, wb_st = nullptr;
  cudaEvent_t begin = nullptr;                // step start on the compute stream
  cudaEvent_t h_ready = nullptr;              // a layer's H rows are in its window
  cudaEvent_t wb_done = nullptr;              // the last write-back of a step
  cudaEvent_t loaded[WINDOWS] = {};           // window filled (H, K part)
  cudaEvent_t loaded2[WINDOWS] = {};          // window filled (V part)
  cudaEvent_t consumed[WINDOWS] = {};         // window no longer read

  size_t slot_elems() const { return size_t(ctx->N) * ctx->d; }
  // index of the [N][d] slot (s, l, t, which) in units of slots
  size_t slot_index(int s, int l, int t, int which) const {
    return ((size_t(s) * ctx->T + t) * ctx->L + l) * 3 + which;
  }
  bf16* slot(int s, int l, int t, int which) const {
    return base + slot_index(s, l, t, which) * slot_elems();
  }
  size_t total_rows() const { return size_t(sessions) * ctx->T * ctx->L * 3 * ctx->N; }
  bf16* text_kv(int s, int l) const {
    return text + (size_t(s) * ctx->L + l) * size_t(ctx->M) * 2 * ctx->d;
  }
  // first xg / xgb row of (session, layer)
  size_t xg_row(int s, int l) const {
    return (size_t(s) * ctx->L + l) * size_t(ctx->dims.heads) * rc::XQ_KEYS;
  }
  size_t xg_rows() const { return xg_row(sessions, 0); }
};

namespace rc {
int ctx_max_batch(const ::rc_ctx* c) { return c->max_batch; }
int ctx_timesteps(const ::rc_ctx* c) { return c->T; }
const ::rc_ctx* cache_context(const ::rc_cache* k) { return k->ctx; }
int cache_sessions(const ::rc_cache* k) { return k->sessions; }
bool cache_host_tier(const ::rc_cache* k) { return k->host_tier; }
}  // namespace rc

namespace {

// The bounded device wait every waiting kernel of this library uses, on its
// own: one thread polls `flag` until it is non-zero or `ns` nanoseconds of
// the global timer have passed; then it records DEVERR_TIMEOUT in the error
// word and returns.  With set_first the flag is raised first (the wait ends
// at once).
__global__ void selftest_wait_kernel(unsigned* flag, unsigned long long ns, int set_first,
                                     unsigned* err) {
  if (threadIdx.x != 0) return;
  volatile unsigned* f = flag;
  if (set_first) *f = 1u;
  unsigned long long t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  while (*f == 0u) {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    if (t - t0 > ns) {
      atomicOr(err, rc::DEVERR_TIMEOUT);
      return;
    }
    __nanosleep(1000);
  }
  *f = 0u;  // lowered again for the next call
}

__global__ void iota_kernel(int* p, int n) {
  int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) p[i] = i;
}

template <class T>
rc_status dalloc(T** p, size_t count, const char* what) {
  void* v = nullptr;
  cudaError_t e = cudaMalloc(&v, count * sizeof(T));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(RC_ERR_OOM, "cudaMalloc(%s, %zu bytes): %s", what, count * sizeof(T),
                cudaGetErrorString(e));
  }
  *p = static_cast<T*>(v);
  return RC_OK;
}

void probe_free(rc_ctx* c) {
  for (cudaEvent_t e : c->probe_ev) cudaEventDestroy(e);
  c->probe_ev.clear();
  c->probe_n = 0;
  c->probe_which = RC_PROBE_OFF;
}

// Brackets one launch of kernel class `which` with probe events.
struct Probe {
  rc_ctx* c;
  cudaStream_t st;
  bool on;
  Probe(rc_ctx* c_, int which, cudaStream_t st_)
      : c(c_), st(st_),
        on(c_->probe_which == which && 2 * (c_->probe_n + 1) <= int(c_->probe_ev.size())) {
    if (on) cudaEventRecord(c->probe_ev[2 * c->probe_n], st);
  }
  ~Probe() {
    if (on) {
      cudaEventRecord(c->probe_ev[2 * c->probe_n + 1], st);
      ++c->probe_n;
    }
  }
};

void free_ctx(rc_ctx* c) {
  if (!c) return;
  probe_free(c);
  void* ps[] = {c->xf,   c->xb,   c->ob,   c->q,    c->u,      c->fbuf,
                c->h1,   c->temb, c->tb,   c->iota, c->b_tok,  c->b_item,
                c->b_meta, c->err, c->wait_flag, c->as.part, c->temb_tab, c->tb_tab};
  for (void* p : ps)
    if (p) cudaFree(p);
  delete c;
}

rc_status check_session(const rc_cache* cache, int session) {
  if (session < 0 || session >= cache->sessions)
    return fail(RC_ERR_INVALID_ARG, "session %d outside [0, %d)", session, cache->sessions);
  return RC_OK;
}

rc_status check_ready(const rc_ctx* c, const rc_cache* cache, int session, bool need_sched) {
  for (int l = 0; l < c->L; ++l)
    if (!c->lw_set[l]) return fail(RC_ERR_STATE, "weights of layer %d not set", l);
  if (!c->gw_set) return fail(RC_ERR_STATE, "global weights not set");
  if (need_sched && !c->sched_set) return fail(RC_ERR_STATE, "schedule not set");
  if (!cache->text_set[session])
    return fail(RC_ERR_STATE, "text of session %d not set (rc_set_text)", session);
  if (cache->text_gen[session] != c->wgen)
    return fail(RC_ERR_STATE,
                "layer weights changed after the text of session %d was set: its text keys "
                "and folded cross-query keys are stale; call rc_set_text again", session);
  return RC_OK;
}

// The items of one step (one for rc_step / rc_block_forward_region): cache
// slices and modulation vectors for the kernels, key / value rows of every
// item for the attention launches.
struct StepItems {
  rc::Items its{};
  int session[rc::MAX_ITEMS] = {};
  int t[rc::MAX_ITEMS] = {};
  const bf16* win = nullptr;  // host tier: the layer's HBM window [H,K,V][N][d] (one item)
};

rc::AttnItems self_kv(const rc_cache* k, const StepItems& si, int l) {
  rc::AttnItems ai{};
  ai.n = si.its.n;
  if (si.win) {
    ai.krow[0] = k->ctx->N;
    ai.vrow[0] = 2 * k->ctx->N;
    return ai;
  }
  for (int i = 0; i < ai.n; ++i) {
    ai.krow[i] = int(k->slot_index(si.session[i], l, si.t[i], 1) * k->ctx->N);
    ai.vrow[i] = int(k->slot_index(si.session[i], l, si.t[i], 2) * k->ctx->N);
  }
  return ai;
}

rc::AttnItems text_kv_rows(const rc_cache* k, const StepItems& si, int l) {
  rc::AttnItems ai{};
  ai.n = si.its.n;
  for (int i = 0; i < ai.n; ++i)
    ai.krow[i] = ai.vrow[i] = (si.session[i] * k->ctx->L + l) * k->ctx->M;
  return ai;
}

// One region-sparse block on the compact residual rows c->xf (Section 3.3,
// Region-Level Sparse Attention; Section 3.4, Kernel Fusing).  The modulation
// vector of a row is tab (+ the row item's tb), each [6][d].  hprev_off >= 0:
// the block input (the previous block's merged output H^l) is also written to
// the cache slice at that element offset, and h_stored (if any) is recorded
// on st once it is there.
rc_status run_block(rc_ctx* c, rc_cache* k, int l, const rc::RowMap& rm, const StepItems& si,
                    const float* tab, long long hprev_off, cudaStream_t st,
                    const rc::AttnCapture* cap = nullptr, cudaEvent_t h_stored = nullptr) {
  const int d = c->d, F = c->F, N = c->N;
  const rc_layer_weights& w = c->lw[l];
  const size_t Nd = size_t(N) * d;

  // x_hat = LN(x)(1 + scale_msa) + shift_msa; x itself is the previous
  // block's output H^l of the dirty rows, written to their cache rows here
  {
    Probe pr(c, RC_PROBE_LN, st);
    RC_CUDA(rc::launch_ln_mod(c->xf, tab, 0, 1, si.its, c->xb, rm, hprev_off, d, c->err, st),
            "ln_mod(msa)");
  }
  if (h_stored) RC_CUDA(cudaEventRecord(h_stored, st), "H stored");
  // [q | k | v] = x_hat W_qkv^T + b; k, v rows go straight to cache rows tok[r]
  rc::GemmEpi e{};
  e.mode = rc::EPI_QKV;
  e.bias = w.b_qkv;
  e.out_bf = c->q;
  e.ld_out = d;
  e.k_off = (long long)(size_t(l) * 3 + 1) * Nd;
  e.v_off = (long long)(size_t(l) * 3 + 2) * Nd;
  e.dsplit = d;
  e.tok = rm.tok;
  e.item = rm.item;
  e.n_tokens = N;
  e.err = c->err;
  e.its = si.its;
  e.gate_off = -1;
  {
    Probe pr(c, RC_PROBE_GEMM, st);
    RC_CUDA(rc::launch_gemm(c->xb, d, static_cast<const bf16*>(w.W_qkv), rm.bound, rm.count,
                            3 * d, d, e, st), "gemm(qkv)");
  }
  // dirty queries over all N keys / values of each item's (session, l, t)
  {
    Probe pr(c, RC_PROBE_ATTENTION, st);
    const bf16* kv = si.win ? si.win : k->base;
    const int kv_rows = si.win ? 3 * N : int(k->total_rows());
    RC_CUDA(rc::launch_attention(c->q, d, kv, kv, d, kv_rows, self_kv(k, si, l), N, c->ob, d,
                                 c->dims.heads, c->dh, rm, c->err, c->as, st),
            "attention(self)");
  }
  // x += gate_msa (o W_o^T + b_o)
  auto gated = [&](const float* bias, int gate_k) {
    rc::GemmEpi g{};
    g.mode = rc::EPI_GATE_RES;
    g.bias = bias;
    g.xf = c->xf;
    g.ld_xf = d;
    g.gate_tab = gate_k >= 0 && tab ? tab + size_t(gate_k) * d : nullptr;
    g.gate_off = gate_k >= 0 ? (long long)gate_k * d : -1;
    g.item = rm.item;
    g.n_tokens = N;
    g.err = c->err;
    g.its = si.its;
    g.whole_tiles = c->deterministic ? 1 : 0;
    return g;
  };
  // (whole tiles, read-modify-write, also leaving xb = bf16(x) for the
  // cross-attention query projection)
  e = gated(w.b_o, 2);
  e.mode = rc::EPI_GATE_RES_CAST;
  e.out_bf = c->xb;
  e.ld_out = d;
  {
    Probe pr(c, RC_PROBE_GEMM, st);
    RC_CUDA(rc::launch_gemm(c->ob, d, static_cast<const bf16*>(w.W_o), rm.bound, rm.count, d, d,
                            e, st), "gemm(out)");
  }
  // the folded form multiplies x by 128 padded key rows per head where the
  // projection multiplies it by dh = 72 (1.8 x the FLOPs, x read once per
  // head); it wins while the rows are few (one launch less per block), the
  // separate GEMM (CTA pairs) once they are many and known on the host
  const bool fold = k->xg && (rm.count || rm.bound < 2048);
  if (fold) {
    // softmax((x W_xq^T + b) K^T / sqrt(dh)) V per head, with the query
    // projection folded into the text keys (x G_h^T + kb_h, G_h = K_h W_xq,h):
    // one kernel on the bf16 copy of x, no cross-query GEMM
    rc::XqItems xi{};
    xi.n = si.its.n;
    for (int i = 0; i < xi.n; ++i) {
      xi.grow[i] = int(k->xg_row(si.session[i], l));
      xi.vrow[i] = (si.session[i] * c->L + l) * c->M;
    }
    Probe pr(c, RC_PROBE_ATTENTION, st);
    RC_CUDA(rc::launch_xattn_fused(c->xb, d, k->xg, k->xgb, int(k->xg_rows()), k->text + d, 2 * d,
                                   k->sessions * c->L * c->M, xi, c->M, c->ob, d, c->dims.heads,
                                   c->dh, rm, c->err, st, cap),
            "attention(cross)");
  } else {
    // q' = x W_xq^T + b (on the bf16 copy of x)
    e = rc::GemmEpi{};
    e.mode = rc::EPI_BIAS_BF16;
    e.bias = w.b_xq;
    e.out_bf = c->q;
    e.ld_out = d;
    e.gate_off = -1;
    e.err = c->err;
    {
      Probe pr(c, RC_PROBE_GEMM, st);
      RC_CUDA(rc::launch_gemm(c->xb, d, static_cast<const bf16*>(w.W_xq), rm.bound, rm.count, d,
                              d, e, st), "gemm(xq)");
    }
    Probe pr(c, RC_PROBE_ATTENTION, st);
    RC_CUDA(rc::launch_attention(c->q, d, k->text, k->text + d, 2 * d,
                                 k->sessions * c->L * c->M, text_kv_rows(k, si, l), c->M, c->ob,
                                 d, c->dims.heads, c->dh, rm, c->err, c->as, st, cap),
            "attention(cross)");
  }
  // x += o' W_xo^T + b (no gate)
  e = gated(w.b_xo, -1);
  {
    Probe pr(c, RC_PROBE_GEMM, st);
    RC_CUDA(rc::launch_gemm(c->ob, d, static_cast<const bf16*>(w.W_xo), rm.bound, rm.count, d, d,
                            e, st), "gemm(xo)");
  }
  // MLP
  {
    Probe pr(c, RC_PROBE_LN, st);
    RC_CUDA(rc::launch_ln_mod(c->xf, tab, 3, 4, si.its, c->xb, rm, -1, d, c->err, st),
            "ln_mod(mlp)");
  }
  e = rc::GemmEpi{};
  e.mode = rc::EPI_GELU_BF16;
  e.bias = w.b_1;
  e.out_bf = c->u;
  e.ld_out = F;
  e.gate_off = -1;
  e.err = c->err;
  {
    Probe pr(c, RC_PROBE_GEMM, st);
    RC_CUDA(rc::launch_gemm(c->xb, d, static_cast<const bf16*>(w.W_1), rm.bound, rm.count, F, d,
                            e, st), "gemm(fc1)");
  }
  // x += gate_mlp (u W_2^T + b_2); the caller stores x as the merged H^{l+1}
  e = gated(w.b_2, 5);
  {
    Probe pr(c, RC_PROBE_GEMM, st);
    RC_CUDA(rc::launch_gemm(c->u, F, static_cast<const bf16*>(w.W_2), rm.bound, rm.count, d, F,
                            e, st), "gemm(fc2)");
  }
  return RC_OK;
}

}  // namespace

extern "C" {

const char* rc_status_string(rc_status s) {
  switch (s) {
    case RC_OK: return "ok";
    case RC_ERR_INVALID_ARG: return "invalid argument";
    case RC_ERR_SHAPE: return "shape mismatch";
    case RC_ERR_OOM: return "out of device memory";
    case RC_ERR_CUDA: return "CUDA error";
    case RC_ERR_TIMEOUT: return "device wait timed out";
    case RC_ERR_DEVICE_ASSERT: return "device-side index/count check failed";
    case RC_ERR_STATE: return "call order violated";
    default: return "unknown status";
  }
}

const char* rc_last_error(void) { return g_last_error.c_str(); }

uint64_t rc_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

rc_status rc_create(const rc_dims* dims, rc_ctx** out) {
  if (!dims || !out) return fail(RC_ERR_INVALID_ARG, "rc_create: null argument");
  *out = nullptr;
  const rc_dims& D = *dims;
  if (D.hidden <= 0 || D.heads <= 0 || D.mlp <= 0 || D.layers <= 0 || D.grid_h <= 0 ||
      D.grid_w <= 0 || D.patch <= 0 || D.in_ch <= 0 || D.out_ch <= 0 || D.text_len <= 0 ||
      D.timesteps <= 0 || D.freq_dim <= 0)
    return fail(RC_ERR_INVALID_ARG, "rc_create: every dimension must be positive");
  if (D.hidden % D.heads) return fail(RC_ERR_SHAPE, "hidden %% heads != 0");
  const int dh = D.hidden / D.heads;
  if (dh != 72 && dh != 64) return fail(RC_ERR_SHAPE, "head_dim %d not in {64, 72}", dh);
  if (D.hidden % 128 || D.hidden > 1536)
    return fail(RC_ERR_SHAPE, "hidden %d must be a multiple of 128 and <= 1536", D.hidden);
  if (D.mlp % 128) return fail(RC_ERR_SHAPE, "mlp %d must be a multiple of 128", D.mlp);
  if (D.freq_dim % 8 || D.freq_dim > 4096) return fail(RC_ERR_SHAPE, "freq_dim %d", D.freq_dim);
  const long long N = 1LL * D.grid_h * D.grid_w;
  if (N > 16384) return fail(RC_ERR_SHAPE, "N = %lld tokens > 16384", N);
  if (D.in_ch * D.patch * D.patch > 16 || D.out_ch < D.in_ch)
    return fail(RC_ERR_SHAPE, "in_ch * patch^2 must be <= 16 and out_ch >= in_ch");
  const int max_batch = D.max_batch <= 0 ? 1 : D.max_batch;
  if (max_batch > RC_MAX_BATCH)
    return fail(RC_ERR_INVALID_ARG, "max_batch %d above %d", D.max_batch, RC_MAX_BATCH);

  rc_ctx* c = new (std::nothrow) rc_ctx();
  if (!c) return fail(RC_ERR_OOM, "host allocation");
  c->dims = D;
  c->N = int(N);
  c->d = D.hidden;
  c->F = D.mlp;
  c->dh = dh;
  c->L = D.layers;
  c->T = D.timesteps;
  c->M = D.text_len;
  c->max_batch = max_batch;
  cudaGetDevice(&c->device);
  c->lw.resize(c->L);
  c->lw_set.assign(c->L, 0);
  rc_status s = RC_OK;
  const size_t R = size_t(max_batch) * N;  // compact rows of a step
  const size_t Rd = R * D.hidden;
  if ((s = dalloc(&c->xf, Rd, "xf")) || (s = dalloc(&c->xb, Rd, "xb")) ||
      (s = dalloc(&c->ob, Rd, "ob")) || (s = dalloc(&c->q, Rd, "q")) ||
      (s = dalloc(&c->u, R * D.mlp, "u")) || (s = dalloc(&c->fbuf, D.freq_dim, "f")) ||
      (s = dalloc(&c->h1, D.hidden, "h1")) ||
      (s = dalloc(&c->temb, size_t(RC_MAX_BATCH) * D.hidden, "temb")) ||
      (s = dalloc(&c->tb, size_t(RC_MAX_BATCH) * 6 * D.hidden, "tb")) ||
      (s = dalloc(&c->temb_tab, size_t(D.timesteps) * D.hidden, "temb table")) ||
      (s = dalloc(&c->tb_tab, size_t(D.timesteps) * 6 * D.hidden, "tb table")) ||
      (s = dalloc(&c->iota, N, "iota")) || (s = dalloc(&c->b_tok, R, "batch tok")) ||
      (s = dalloc(&c->b_item, R, "batch item")) ||
      (s = dalloc(&c->b_meta, size_t(rc::META_INTS), "batch meta")) ||
      (s = dalloc(&c->err, 1, "err")) || (s = dalloc(&c->wait_flag, 1, "wait flag"))) {
    free_ctx(c);
    return s;
  }
  c->as.part_floats = rc::attention_split_floats(int(N), D.heads, dh);
  if ((s = dalloc(&c->as.part, c->as.part_floats, "attn part"))) {
    free_ctx(c);
    return s;
  }
  iota_kernel<<<int((N + 255) / 256), 256>>>(c->iota, int(N));
  rc::count_launches(1);
  cudaError_t e = cudaMemset(c->err, 0, sizeof(unsigned));
  if (e == cudaSuccess) e = cudaMemset(c->wait_flag, 0, sizeof(unsigned));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    free_ctx(c);
    return cuda_fail(e, "rc_create");
  }
  *out = c;
  return RC_OK;
}

void rc_destroy(rc_ctx* ctx) { free_ctx(ctx); }

rc_status rc_set_layer_weights(rc_ctx* c, int layer, const rc_layer_weights* w) {
  if (!c || !w) return fail(RC_ERR_INVALID_ARG, "rc_set_layer_weights: null argument");
  if (layer < 0 || layer >= c->L)
    return fail(RC_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, c->L);
  const void* ps[] = {w->W_qkv, w->b_qkv, w->W_o, w->b_o, w->W_xq, w->b_xq, w->W_xkv, w->b_xkv,
                      w->W_xo,  w->b_xo,  w->W_1, w->b_1, w->W_2,  w->b_2,  w->table};
  for (const void* p : ps)
    if (!p || !aligned16(p))
      return fail(RC_ERR_INVALID_ARG, "layer %d: null or unaligned (16 B) weight", layer);
  c->lw[layer] = *w;
  c->lw_set[layer] = 1;
  ++c->wgen;
  return RC_OK;
}

rc_status rc_set_global_weights(rc_ctx* c, const rc_global_weights* w) {
  if (!c || !w) return fail(RC_ERR_INVALID_ARG, "rc_set_global_weights: null argument");
  const void* ps[] = {w->W_e, w->b_e,  w->pos,     w->W_t1, w->b_t1, w->W_t2,
                      w->b_t2, w->W_tb, w->b_tb, w->table_f, w->W_f, w->b_f};
  for (const void* p : ps)
    if (!p || !aligned16(p))
      return fail(RC_ERR_INVALID_ARG, "global weights: null or unaligned (16 B) pointer");
  c->gw = *w;
  c->gw_set = true;
  c->t_ready = false;
  return RC_OK;
}

rc_status rc_set_schedule(rc_ctx* c, const float* tv, const float* ab) {
  if (!c || !tv || !ab) return fail(RC_ERR_INVALID_ARG, "rc_set_schedule: null argument");
  for (int i = 0; i <= c->T; ++i)
    if (!(ab[i] > 0.f && ab[i] <= 1.f))
      return fail(RC_ERR_INVALID_ARG, "alpha_bar[%d] = %g outside (0, 1]", i, double(ab[i]));
  c->t_values.assign(tv, tv + c->T);
  c->alpha_bar.assign(ab, ab + c->T + 1);
  c->sched_set = true;
  c->t_ready = false;
  return RC_OK;
}

rc_status rc_set_deterministic(rc_ctx* c, int on) {
  if (!c) return fail(RC_ERR_INVALID_ARG, "rc_set_deterministic: null context");
  c->deterministic = on != 0;
  return RC_OK;
}

// The folded text keys of every (session, layer), zero-filled (rows past the
// text length stay zero).  Only when the text fits one cross-attention pass.
static rc_status alloc_xg(rc_cache* k) {
  const rc_ctx* c = k->ctx;
  if (c->M > rc::XQ_KEYS) return RC_OK;
  rc_status s = dalloc(&k->xg, k->xg_rows() * c->d, "folded text keys");
  if (s == RC_OK) s = dalloc(&k->xgb, k->xg_rows(), "folded text key biases");
  if (s == RC_OK && (cudaMemset(k->xg, 0, k->xg_rows() * c->d * sizeof(bf16)) != cudaSuccess ||
                     cudaMemset(k->xgb, 0, k->xg_rows() * sizeof(float)) != cudaSuccess))
    s = fail(RC_ERR_CUDA, "folded text keys zero fill failed");
  return s;
}

rc_status rc_cache_create(rc_ctx* c, int sessions, rc_cache** out) {
  if (!c || !out) return fail(RC_ERR_INVALID_ARG, "rc_cache_create: null argument");
  *out = nullptr;
  if (sessions <= 0) return fail(RC_ERR_INVALID_ARG, "sessions = %d", sessions);
  rc_cache* k = new (std::nothrow) rc_cache();
  if (!k) return fail(RC_ERR_OOM, "host allocation");
  k->ctx = c;
  k->sessions = sessions;
  k->text_set.assign(sessions, 0);
  k->text_gen.assign(sessions, 0);
  // attention addresses every cache row with a 32-bit tensor coordinate
  if (k->total_rows() >= (size_t(1) << 31) || size_t(sessions) * c->L * c->M >= (size_t(1) << 31)) {
    delete k;
    return fail(RC_ERR_SHAPE, "cache of %d sessions has 2^31 rows or more", sessions);
  }
  const size_t n = size_t(sessions) * c->T * c->L * 3 * k->slot_elems();
  rc_status s = dalloc(&k->base, n, "cache");
  const size_t n_text = size_t(sessions) * c->L * c->M * 2 * c->d;
  if (s == RC_OK) s = dalloc(&k->text, n_text, "text kv");
  if (s == RC_OK) s = alloc_xg(k);
  // zero-filled: the attention reads whole 64-key blocks, and keys past a
  // slot's end (weighted by zero) come from the next slot, which must be finite
  if (s == RC_OK && (cudaMemset(k->base, 0, n * sizeof(bf16)) != cudaSuccess ||
                     cudaMemset(k->text, 0, n_text * sizeof(bf16)) != cudaSuccess ||
                     cudaDeviceSynchronize() != cudaSuccess))
    s = fail(RC_ERR_CUDA, "cache zero fill failed");
  if (s != RC_OK) {
    if (k->base) cudaFree(k->base);
    if (k->text) cudaFree(k->text);
    if (k->xg) cudaFree(k->xg);
    if (k->xgb) cudaFree(k->xgb);
    delete k;
    return s;
  }
  *out = k;
  return RC_OK;
}

void rc_cache_destroy(rc_cache* k) {
  if (!k) return;
  if (k->host_tier) {
    for (cudaStream_t q : {k->copy_st, k->copy_st2, k->wb_st})
      if (q) cudaStreamSynchronize(q);
    if (k->host_mem) cudaHostUnregister(k->host_mem);
    if (k->host_map) munmap(k->host_map, k->host_map_bytes);
    if (k->window) cudaFree(k->window);
    for (cudaEvent_t e : {k->begin, k->h_ready, k->wb_done}) if (e) cudaEventDestroy(e);
    for (int i = 0; i < rc_cache::WINDOWS; ++i) {
      if (k->loaded[i]) cudaEventDestroy(k->loaded[i]);
      if (k->loaded2[i]) cudaEventDestroy(k->loaded2[i]);
      if (k->consumed[i]) cudaEventDestroy(k->consumed[i]);
    }
    for (cudaStream_t q : {k->copy_st, k->copy_st2, k->wb_st})
      if (q) cudaStreamDestroy(q);
  } else if (k->base) {
    cudaFree(k->base);
  }
  if (k->text) cudaFree(k->text);
  if (k->xg) cudaFree(k->xg);
  if (k->xgb) cudaFree(k->xgb);
  delete k;
}

rc_status rc_cache_create_host(rc_ctx* c, int sessions, rc_cache** out) {
  if (!c || !out) return fail(RC_ERR_INVALID_ARG, "rc_cache_create_host: null argument");
  *out = nullptr;
  if (sessions <= 0) return fail(RC_ERR_INVALID_ARG, "sessions = %d", sessions);
  rc_cache* k = new (std::nothrow) rc_cache();
  if (!k) return fail(RC_ERR_OOM, "host allocation");
  k->ctx = c;
  k->sessions = sessions;
  k->text_set.assign(sessions, 0);
  k->text_gen.assign(sessions, 0);
  k->host_tier = true;
  const size_t n = size_t(sessions) * c->T * c->L * 3 * k->slot_elems();
  const size_t n_text = size_t(sessions) * c->L * c->M * 2 * c->d;
  rc_status s = RC_OK;
  // an anonymous mapping aligned to 512 MB and advised for transparent huge
  // pages (fewer translations for the copy engines and the write-back),
  // zero-filled, then page-locked and mapped for the device
  const size_t bytes = n * sizeof(bf16), huge = size_t(512) << 20;
  k->host_map_bytes = bytes + huge;
  void* m = mmap(nullptr, k->host_map_bytes, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS,
                 -1, 0);
  if (m == MAP_FAILED) {
    k->host_map_bytes = 0;
    s = fail(RC_ERR_OOM, "host cache mapping of %zu bytes", bytes);
  } else {
    k->host_map = m;
    void* a = reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(m) + huge - 1) & ~(huge - 1));
    madvise(a, bytes, MADV_HUGEPAGE);  // advice only: small pages work too
    memset(a, 0, bytes);
    if (cudaHostRegister(a, bytes, cudaHostRegisterMapped | cudaHostRegisterPortable) !=
        cudaSuccess) {
      cudaGetLastError();
      s = fail(RC_ERR_OOM, "page-locking a host cache of %zu bytes", bytes);
    } else {
      k->host_mem = a;
    }
  }
  void* dev = nullptr;
  if (s == RC_OK && cudaHostGetDevicePointer(&dev, k->host_mem, 0) != cudaSuccess)
    s = fail(RC_ERR_CUDA, "no device address for the host cache");
  if (s == RC_OK) {
    k->base = static_cast<bf16*>(dev);
    s = dalloc(&k->window, rc_cache::WINDOWS * 3 * k->slot_elems(), "cache window");
  }
  if (s == RC_OK) s = dalloc(&k->text, n_text, "text kv");
  if (s == RC_OK) s = alloc_xg(k);
  if (s == RC_OK &&
      (cudaMemset(k->window, 0, rc_cache::WINDOWS * 3 * k->slot_elems() * sizeof(bf16)) !=
           cudaSuccess ||
       cudaMemset(k->text, 0, n_text * sizeof(bf16)) != cudaSuccess ||
       cudaStreamCreateWithFlags(&k->copy_st, cudaStreamNonBlocking) != cudaSuccess ||
       cudaStreamCreateWithFlags(&k->copy_st2, cudaStreamNonBlocking) != cudaSuccess ||
       cudaStreamCreateWithFlags(&k->wb_st, cudaStreamNonBlocking) != cudaSuccess))
    s = fail(RC_ERR_CUDA, "host cache set-up failed");
  cudaEvent_t* evs[] = {&k->begin,      &k->h_ready,    &k->wb_done,    &k->loaded[0],
                        &k->loaded[1],  &k->loaded[2],  &k->loaded2[0], &k->loaded2[1],
                        &k->loaded2[2], &k->consumed[0], &k->consumed[1], &k->consumed[2]};
  for (cudaEvent_t* e : evs)
    if (s == RC_OK && cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess)
      s = fail(RC_ERR_CUDA, "host cache events");
  if (s == RC_OK && cudaDeviceSynchronize() != cudaSuccess)
    s = fail(RC_ERR_CUDA, "host cache set-up failed");
  if (s != RC_OK) {
    rc_cache_destroy(k);
    return s;
  }
  *out = k;
  return RC_OK;
}

static rc_status cache_copy(rc_cache* k, int s, int l, int t, void* H, void* K, void* V,
                            bool fill, cudaStream_t st) {
  if (!k) return fail(RC_ERR_INVALID_ARG, "null cache");
  rc_status r = check_session(k, s);
  if (r) return r;
  if (l < 0 || l >= k->ctx->L || t < 0 || t >= k->ctx->T)
    return fail(RC_ERR_INVALID_ARG, "layer %d / t %d out of range", l, t);
  void* ps[3] = {H, K, V};
  const size_t bytes = k->slot_elems() * sizeof(bf16);
  for (int w = 0; w < 3; ++w) {
    if (!ps[w]) continue;
    bf16* slot = k->slot(s, l, t, w);
    RC_CUDA(cudaMemcpyAsync(fill ? static_cast<void*>(slot) : ps[w],
                            fill ? static_cast<const void*>(ps[w]) : slot, bytes,
                            cudaMemcpyDefault, st),
            "cache copy");
  }
  return RC_OK;
}

rc_status rc_cache_fill(rc_cache* k, int s, int l, int t, const void* H, const void* K,
                        const void* V, rc_stream st) {
  return cache_copy(k, s, l, t, const_cast<void*>(H), const_cast<void*>(K), const_cast<void*>(V),
                    true, static_cast<cudaStream_t>(st));
}

rc_status rc_cache_read(rc_cache* k, int s, int l, int t, void* H, void* K, void* V,
                        rc_stream st) {
  return cache_copy(k, s, l, t, H, K, V, false, static_cast<cudaStream_t>(st));
}

// The cross-query projection folded into the text keys of one session, all
// layers (Section 3.3's cross-attention, reassociated: see run_block).
static rc_status fold_text(rc_ctx* c, rc_cache* k, int s, cudaStream_t st) {
  if (!k->xg) return RC_OK;
  for (int l = 0; l < c->L; ++l)
    RC_CUDA(rc::launch_xq_fold(k->text_kv(s, l), 2 * c->d, static_cast<const bf16*>(c->lw[l].W_xq),
                               c->lw[l].b_xq, c->M, c->dims.heads, c->dh, c->d,
                               k->xg + k->xg_row(s, l) * c->d, k->xgb + k->xg_row(s, l), st),
            "fold text keys");
  return RC_OK;
}

// Session file: magic, then int32 version, N, hidden, layers, timesteps,
// text_len, text_set; then the session's slots in cache order
// ([t][layer][H,K,V][N][hidden]) and its text keys / values
// ([layer][text_len][2 hidden]), bf16.
static const char kCacheMagic[8] = {'R', 'C', 'C', 'A', 'C', 'H', 'E', '1'};

// Copies `elems` bf16 between device-addressable `dev` and the file through a
// pinned staging buffer.
static rc_status session_io(bf16* dev, size_t elems, FILE* f, bool write, void* stage,
                            size_t stage_bytes) {
  const size_t per = stage_bytes / sizeof(bf16);
  for (size_t off = 0; off < elems; off += per) {
    const size_t n = elems - off < per ? elems - off : per;
    if (write) {
      RC_CUDA(cudaMemcpy(stage, dev + off, n * sizeof(bf16), cudaMemcpyDefault), "export copy");
      if (fwrite(stage, sizeof(bf16), n, f) != n) return fail(RC_ERR_IO, "short write");
    } else {
      if (fread(stage, sizeof(bf16), n, f) != n) return fail(RC_ERR_IO, "short read");
      RC_CUDA(cudaMemcpy(dev + off, stage, n * sizeof(bf16), cudaMemcpyDefault), "import copy");
    }
  }
  return RC_OK;
}

static rc_status session_file(rc_cache* k, int s, const char* path, bool write) {
  if (!k || !path) return fail(RC_ERR_INVALID_ARG, "null cache or path");
  rc_status r = check_session(k, s);
  if (r) return r;
  const rc_ctx* c = k->ctx;
  RC_CUDA(cudaDeviceSynchronize(), "synchronise");
  FILE* f = fopen(path, write ? "wb" : "rb");
  if (!f) return fail(RC_ERR_IO, "cannot open %s", path);
  bool header_ok = write;  // an import overwrites the session only past a good header
  int32_t hdr[7] = {1, c->N, c->d, c->L, c->T, c->M, write ? int32_t(k->text_set[s]) : 0};
  if (write) {
    if (fwrite(kCacheMagic, 1, 8, f) != 8 || fwrite(hdr, sizeof(int32_t), 7, f) != 7)
      r = fail(RC_ERR_IO, "short write");
  } else {
    char magic[8];
    int32_t got[7];
    if (fread(magic, 1, 8, f) != 8 || memcmp(magic, kCacheMagic, 8) != 0)
      r = fail(RC_ERR_IO, "%s is not a cache file", path);
    else if (fread(got, sizeof(int32_t), 7, f) != 7)
      r = fail(RC_ERR_IO, "short read");
    else if (got[0] != 1 || memcmp(got + 1, hdr + 1, 5 * sizeof(int32_t)) != 0)
      r = fail(RC_ERR_SHAPE, "file dims N %d hidden %d layers %d T %d text %d differ", got[1],
               got[2], got[3], got[4], got[5]);
    else {
      hdr[6] = got[6];
      header_ok = true;
    }
  }
  void* stage = nullptr;
  const size_t stage_bytes = size_t(64) << 20;
  if (r == RC_OK && cudaMallocHost(&stage, stage_bytes) != cudaSuccess) {
    cudaGetLastError();
    stage = nullptr;
    r = fail(RC_ERR_OOM, "pinned staging buffer");
  }
  if (r == RC_OK)
    r = session_io(k->slot(s, 0, 0, 0), size_t(c->T) * c->L * 3 * k->slot_elems(), f, write,
                   stage, stage_bytes);
  if (r == RC_OK)
    r = session_io(k->text_kv(s, 0), size_t(c->L) * c->M * 2 * c->d, f, write, stage,
                   stage_bytes);
  if (stage) cudaFreeHost(stage);
  if (fclose(f) != 0 && r == RC_OK) r = fail(RC_ERR_IO, "closing %s", path);
  if (r == RC_OK && !write && hdr[6] != 0) {
    // the folded text keys are derived data: recomputed from the imported
    // keys and the context's cross-query weights
    for (int l = 0; l < c->L && r == RC_OK; ++l)
      if (!c->lw_set[l]) r = fail(RC_ERR_STATE, "weights of layer %d not set before import", l);
    if (r == RC_OK) r = fold_text(k->ctx, k, s, nullptr);
    if (r == RC_OK && cudaStreamSynchronize(nullptr) != cudaSuccess)
      r = fail(RC_ERR_CUDA, "folding the imported text keys");
  }
  if (!write && header_ok) {
    // after a good header the session's slots and text are being replaced:
    // a failure part-way leaves a mix of old and new data, so the session
    // needs rc_set_text (or another import) before its next step
    k->text_set[s] = char(r == RC_OK && hdr[6] != 0);
    k->text_gen[s] = k->ctx->wgen;
  }
  return r;
}

rc_status rc_cache_export(rc_cache* k, int s, const char* path) {
  return session_file(k, s, path, true);
}
rc_status rc_cache_import(rc_cache* k, int s, const char* path) {
  return session_file(k, s, path, false);
}

rc_status rc_set_text(rc_ctx* c, rc_cache* k, int s, const void* ctx_bf16, rc_stream stream) {
  if (!c || !k || !ctx_bf16) return fail(RC_ERR_INVALID_ARG, "rc_set_text: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  rc_status r = check_session(k, s);
  if (r) return r;
  if (!aligned16(ctx_bf16)) return fail(RC_ERR_INVALID_ARG, "text context not 16-B aligned");
  for (int l = 0; l < c->L; ++l)
    if (!c->lw_set[l]) return fail(RC_ERR_STATE, "weights of layer %d not set", l);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  for (int l = 0; l < c->L; ++l) {
    rc::GemmEpi e{};
    e.mode = rc::EPI_BIAS_BF16;
    e.bias = c->lw[l].b_xkv;
    e.out_bf = k->text_kv(s, l);
    e.ld_out = 2 * c->d;
    e.err = c->err;
    RC_CUDA(rc::launch_gemm(static_cast<const bf16*>(ctx_bf16), c->d,
                            static_cast<const bf16*>(c->lw[l].W_xkv), c->M, nullptr, 2 * c->d,
                            c->d, e, st), "gemm(text kv)");
  }
  if ((r = fold_text(c, k, s, st))) return r;
  k->text_set[s] = 1;
  k->text_gen[s] = c->wgen;
  return RC_OK;
}

size_t rc_localize_workspace_size(int N, int n_delta) {
  if (N <= 0 || n_delta <= 0) return 0;
  return rc::localize_workspace_bytes(N, n_delta);
}

rc_status rc_localize_mask(const float* xattn, int S, int N, int M, int grid_h, int grid_w,
                           const int32_t* delta_ids_host, int n_delta, float threshold,
                           int dilation, uint8_t* mask, int32_t* dirty_idx, int32_t* dirty_count,
                           void* workspace, size_t workspace_bytes, rc_stream stream) {
  if (!xattn || !delta_ids_host || !mask || !dirty_idx || !dirty_count || !workspace)
    return fail(RC_ERR_INVALID_ARG, "rc_localize_mask: null pointer");
  if (S < 1 || M < 1 || N < 1 || grid_h < 1 || grid_w < 1)
    return fail(RC_ERR_SHAPE, "rc_localize_mask: S, M, N and the grid must be positive");
  if (1LL * grid_h * grid_w != N) return fail(RC_ERR_SHAPE, "N != grid_h * grid_w");
  if (N > 16384) return fail(RC_ERR_SHAPE, "N = %d > 16384", N);
  if (n_delta < 1 || n_delta > 64) return fail(RC_ERR_INVALID_ARG, "n_delta %d not in 1..64", n_delta);
  if (dilation < 0 || dilation > 8) return fail(RC_ERR_INVALID_ARG, "dilation %d not in 0..8", dilation);
  if (!(threshold == threshold) || threshold > 3.4e38f || threshold < -3.4e38f)
    return fail(RC_ERR_INVALID_ARG, "threshold is not finite");
  if (workspace_bytes < rc::localize_workspace_bytes(N, n_delta))
    return fail(RC_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes,
                rc::localize_workspace_bytes(N, n_delta));
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return fail(RC_ERR_INVALID_ARG, "workspace not 256-B aligned");
  rc::DeltaIds ids{};
  ids.n = n_delta;
  for (int j = 0; j < n_delta; ++j) {
    if (delta_ids_host[j] < 0 || delta_ids_host[j] >= M)
      return fail(RC_ERR_INVALID_ARG, "delta id %d outside [0, %d)", delta_ids_host[j], M);
    ids.id[j] = delta_ids_host[j];
  }
  RC_CUDA(rc::launch_localize(xattn, S, N, M, grid_h, grid_w, ids, threshold, dilation, mask,
                              dirty_idx, dirty_count, workspace, static_cast<cudaStream_t>(stream)),
          "localize");
  return RC_OK;
}

// The dirty rows of one item: host bound and optional device count.
static rc_status dirty_rows(const rc_ctx* c, const int32_t* idx, int D, const int32_t* dcount,
                            int* bound) {
  if (D < -1 || D > c->N) return fail(RC_ERR_INVALID_ARG, "D = %d outside [-1, %d]", D, c->N);
  if (D == -1 && !dcount) return fail(RC_ERR_INVALID_ARG, "D = -1 needs a device dirty_count");
  *bound = D < 0 ? c->N : D;
  if (*bound > 0 && !idx) return fail(RC_ERR_INVALID_ARG, "dirty_idx is null");
  if (idx && (reinterpret_cast<uintptr_t>(idx) & 3u))
    return fail(RC_ERR_INVALID_ARG, "dirty_idx not 4-B aligned");
  return RC_OK;
}

rc_status rc_block_forward_region(rc_ctx* c, rc_cache* k, int s, int l, int t, float* hidden,
                                  const int32_t* dirty_idx, int D, const int32_t* dirty_count,
                                  const float* mod6, rc_stream stream) {
  if (!c || !k || !hidden || !mod6)
    return fail(RC_ERR_INVALID_ARG, "rc_block_forward_region: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (k->host_tier)
    return fail(RC_ERR_INVALID_ARG, "rc_block_forward_region needs a device-tier cache");
  rc_status r = check_session(k, s);
  if (r) return r;
  if (l < 0 || l >= c->L || t < 0 || t >= c->T)
    return fail(RC_ERR_INVALID_ARG, "layer %d / t %d out of range", l, t);
  if (!aligned16(hidden) || !aligned16(mod6))
    return fail(RC_ERR_INVALID_ARG, "hidden / mod6 not 16-B aligned");
  if ((r = check_ready(c, k, s, false))) return r;
  int bound = 0;
  if ((r = dirty_rows(c, dirty_idx, D, dirty_count, &bound))) return r;
  if (bound == 0) return RC_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  StepItems si;
  si.its.n = 1;
  si.its.slice[0] = k->slot(s, 0, t, 0);
  si.session[0] = s;
  si.t[0] = t;
  const rc::RowMap rm{dirty_idx, nullptr, nullptr, bound, dirty_count, c->N};
  RC_CUDA(rc::launch_rows_f32(hidden, c->xf, dirty_idx, bound, dirty_count, c->d, c->N, false,
                              c->err, st), "gather");
  if ((r = run_block(c, k, l, rm, si, mod6, -1, st))) return r;
  RC_CUDA(rc::launch_scatter_bf16(c->xf, si.its, (long long)(size_t(l) * 3) * c->N * c->d, rm,
                                  c->d, c->err, st), "H scatter");
  RC_CUDA(rc::launch_rows_f32(c->xf, hidden, dirty_idx, bound, dirty_count, c->d, c->N, true,
                              c->err, st), "scatter");
  return RC_OK;
}

// Host tier: window l % 3 receives layer l's cached K, V of item (s, t) (and
// H for the last layer, which the final layer reads over all tokens) on the
// copy stream, once the window's previous readers are done.
static rc_status host_load(rc_cache* k, int s, int t, int l) {
  const size_t Nd = k->slot_elems();
  const int first = l == k->ctx->L - 1 ? 0 : 1, w = l % rc_cache::WINDOWS;
  // V on a second copy stream (a second copy engine): H (last layer) and K
  // on the first
  RC_CUDA(cudaStreamWaitEvent(k->copy_st, k->consumed[w], 0), "window wait");
  RC_CUDA(cudaStreamWaitEvent(k->copy_st2, k->consumed[w], 0), "window wait");
  RC_CUDA(cudaMemcpyAsync(k->window + (size_t(w) * 3 + first) * Nd, k->slot(s, l, t, first),
                          (2 - first) * Nd * sizeof(bf16), cudaMemcpyDefault, k->copy_st),
          "window load");
  RC_CUDA(cudaMemcpyAsync(k->window + (size_t(w) * 3 + 2) * Nd, k->slot(s, l, t, 2),
                          Nd * sizeof(bf16), cudaMemcpyDefault, k->copy_st2),
          "window load");
  RC_CUDA(cudaEventRecord(k->loaded[w], k->copy_st), "window event");
  RC_CUDA(cudaEventRecord(k->loaded2[w], k->copy_st2), "window event");
  return RC_OK;
}

// Host tier: once layer l's H rows are in window l % 3 (h_ready, recorded on
// st by the next block after its first LN, or here for the last layer), the
// write-back stream sends its dirty H, K, V rows to the host slice.
static rc_status host_writeback(rc_ctx* c, rc_cache* k, int s, int t, int l,
                                const rc::RowMap& rm, cudaStream_t st, bool last) {
  const int w = l % rc_cache::WINDOWS;
  if (last) RC_CUDA(cudaEventRecord(k->h_ready, st), "write-back event");
  RC_CUDA(cudaStreamWaitEvent(k->wb_st, k->h_ready, 0), "write-back wait");
  RC_CUDA(rc::launch_writeback(k->window + size_t(w) * 3 * k->slot_elems(), k->slot(s, l, t, 0),
                               rm, c->d, c->err, k->wb_st),
          "write-back");
  RC_CUDA(cudaEventRecord(k->consumed[w], k->wb_st), "window event");
  if (last) RC_CUDA(cudaEventRecord(k->wb_done, k->wb_st), "write-back event");
  return RC_OK;
}

// The timestep embedding and t_block modulation of every scheduled timestep
// into temb_tab / tb_tab, queued on st, when the global weights or the
// schedule changed since they were last computed.
static rc_status fill_t_tables(rc_ctx* c, cudaStream_t st) {
  if (c->t_ready) return RC_OK;
  const rc_global_weights& g = c->gw;
  const int d = c->d;
  for (int t = 0; t < c->T; ++t)
    RC_CUDA(rc::launch_t_embed(c->t_values[t], c->dims.freq_dim, d,
                               static_cast<const bf16*>(g.W_t1), g.b_t1,
                               static_cast<const bf16*>(g.W_t2), g.b_t2,
                               static_cast<const bf16*>(g.W_tb), g.b_tb, c->fbuf, c->h1,
                               c->temb_tab + size_t(t) * d, c->tb_tab + size_t(t) * 6 * d, st),
            "t_embed");
  c->t_ready = true;
  return RC_OK;
}

// Denoising steps of n items (validated by the callers); cap (DENSE single
// item only) captures cross-attention probabilities of listed text tokens.
// On a host-tier cache (one item) the layers run on HBM windows while the
// copy stream loads the layers ahead (Section 3.4, Pipelined Execution).
static rc_status step_items(rc_ctx* c, rc_cache* k, const rc_batch_item* items, int n,
                            cudaStream_t st, const rc::AttnCapture* cap = nullptr) {
  const rc_global_weights& g = c->gw;
  const int d = c->d, N = c->N;
  const size_t Nd = size_t(N) * d;
  StepItems si;
  si.its.n = n;
  rc::BatchIn bin{};
  bin.n = n;
  long long rows = 0;
  // the per-timestep tables, unless this stream is being captured before
  // they exist (a capture by the caller: the step then computes its items'
  // embeddings itself, as part of the captured work)
  bool tables = c->t_ready;
  if (!tables) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    RC_CUDA(cudaStreamIsCapturing(st, &cs), "capture status");
    if (cs == cudaStreamCaptureStatusNone) {
      rc_status r = fill_t_tables(c, st);
      if (r) return r;
      tables = true;
    }
  }
  const float* temb_of[rc::MAX_ITEMS] = {};
  for (int i = 0; i < n; ++i) {
    const rc_batch_item& it = items[i];
    si.session[i] = it.session;
    si.t[i] = it.t;
    si.its.slice[i] = k->slot(it.session, 0, it.t, 0);
    si.its.tb[i] = tables ? c->tb_tab + size_t(it.t) * 6 * d : c->tb + size_t(i) * 6 * d;
    temb_of[i] = tables ? c->temb_tab + size_t(it.t) * d : c->temb + size_t(i) * d;
    si.its.latent[i] = it.latent;
    if (it.mode == RC_MODE_DENSE) {
      bin.idx[i] = c->iota;
      bin.bound[i] = N;
    } else if (it.mode == RC_MODE_SPARSE) {
      bin.idx[i] = it.dirty_idx;
      bin.count[i] = it.dirty_count;
      bin.bound[i] = it.D < 0 ? N : it.D;
    }
    rows += bin.bound[i];
    if (!tables)
      RC_CUDA(rc::launch_t_embed(c->t_values[it.t], c->dims.freq_dim, d,
                                 static_cast<const bf16*>(g.W_t1), g.b_t1,
                                 static_cast<const bf16*>(g.W_t2), g.b_t2,
                                 static_cast<const bf16*>(g.W_tb), g.b_tb, c->fbuf, c->h1,
                                 c->temb + size_t(i) * d, c->tb + size_t(i) * 6 * d, st),
              "t_embed");
  }
  const bool host = k->host_tier;
  const int s0 = items[0].session, t0 = items[0].t, L = c->L;
  const size_t wstride = 3 * Nd;  // elements per window
  bf16* const win_last =
      host ? k->window + size_t((L - 1) % rc_cache::WINDOWS) * wstride : nullptr;
  if (host) {
    if (n != 1) return fail(RC_ERR_INVALID_ARG, "a host-tier cache steps one item at a time");
    RC_CUDA(cudaEventRecord(k->begin, st), "step event");
    RC_CUDA(cudaStreamWaitEvent(k->copy_st, k->begin, 0), "step wait");
    RC_CUDA(cudaStreamWaitEvent(k->copy_st2, k->begin, 0), "step wait");
    rc_status r = host_load(k, s0, t0, rows > 0 ? 0 : L - 1);
    if (r == RC_OK && rows > 0 && L > 1) r = host_load(k, s0, t0, 1);
    if (r) return r;
  }
  if (rows > 0) {
    // compact rows: a single item uses its own index list; several items are
    // concatenated on the device (their counts may live there)
    rc::RowMap rm{bin.idx[0], nullptr, nullptr, int(rows), bin.count[0], N};
    if (n > 1) {
      RC_CUDA(rc::launch_batch_rows(bin, c->b_tok, c->b_item, c->b_meta, N, c->err, st),
              "batch rows");
      rm = rc::RowMap{c->b_tok, c->b_item, c->b_meta, int(rows), c->b_meta + rc::META_TOTAL, N};
    }
    RC_CUDA(rc::launch_patch_embed(c->dims.grid_h, c->dims.grid_w, c->dims.patch, c->dims.in_ch,
                                   static_cast<const bf16*>(g.W_e), g.b_e, g.pos, si.its, rm,
                                   c->xf, d, c->err, st),
            "patch_embed");
    for (int l = 0; l < L; ++l) {
      if (!host) {
        rc_status r = run_block(c, k, l, rm, si, c->lw[l].table,
                                l > 0 ? (long long)(size_t(l - 1) * 3) * Nd : -1, st, cap);
        if (r) return r;
        continue;
      }
      // the window stands in for the slice: its K, V rows take the QKV
      // epilogue's writes and feed the self-attention, and the block's first
      // LN stores its input (layer l - 1's output H) into window (l - 1) % 3,
      // after which the write-back stream sends layer l - 1's rows home
      const int w = l % rc_cache::WINDOWS, wp = (l + rc_cache::WINDOWS - 1) % rc_cache::WINDOWS;
      bf16* win = k->window + size_t(w) * wstride;
      si.win = win;
      si.its.slice[0] = reinterpret_cast<bf16*>(reinterpret_cast<uintptr_t>(win) -
                                                size_t(l) * wstride * sizeof(bf16));
      const long long hprev =
          l > 0 ? (long long)(size_t(wp) * wstride + size_t(l) * wstride) - (long long)(w * wstride)
                : -1;
      RC_CUDA(cudaStreamWaitEvent(st, k->loaded[w], 0), "window ready");
      RC_CUDA(cudaStreamWaitEvent(st, k->loaded2[w], 0), "window ready");
      rc_status r = run_block(c, k, l, rm, si, c->lw[l].table, hprev, st, cap,
                              l > 0 ? k->h_ready : nullptr);
      if (r) return r;
      if (l > 0 && (r = host_writeback(c, k, s0, t0, l - 1, rm, st, false))) return r;
      if (l + 2 < L && (r = host_load(k, s0, t0, l + 2))) return r;
    }
    RC_CUDA(rc::launch_scatter_bf16(c->xf, si.its, (long long)(size_t(L - 1) * 3) * Nd, rm, d,
                                    c->err, st), "H scatter");
    if (host) {
      rc_status r = host_writeback(c, k, s0, t0, L - 1, rm, st, true);
      if (r) return r;
    }
  } else if (host) {
    RC_CUDA(cudaStreamWaitEvent(st, k->loaded[(L - 1) % rc_cache::WINDOWS], 0), "window ready");
    RC_CUDA(cudaStreamWaitEvent(st, k->loaded2[(L - 1) % rc_cache::WINDOWS], 0), "window ready");
  }
  for (int i = 0; i < n; ++i) {
    const rc_batch_item& it = items[i];
    RC_CUDA(rc::launch_final_ddim(host ? win_last : k->slot(it.session, L - 1, it.t, 0),
                                  temb_of[i],
                                  g.table_f, static_cast<const bf16*>(g.W_f), g.b_f, it.latent,
                                  c->dims.grid_h, c->dims.grid_w, c->dims.patch, c->dims.in_ch,
                                  c->dims.out_ch, d, c->alpha_bar[it.t], c->alpha_bar[it.t + 1],
                                  st), "final_ddim");
  }
  if (host) {
    // the step ends when its write-backs have landed; the next step's loads
    // also wait for the final layer's reads
    if (rows > 0) RC_CUDA(cudaStreamWaitEvent(st, k->wb_done, 0), "write-back done");
    for (int i = 0; i < rc_cache::WINDOWS; ++i)
      RC_CUDA(cudaEventRecord(k->consumed[i], st), "window event");
  }
  return RC_OK;
}

static rc_status check_item(rc_ctx* c, rc_cache* k, const rc_batch_item& it) {
  rc_status r = check_session(k, it.session);
  if (r) return r;
  if (it.t < 0 || it.t >= c->T) return fail(RC_ERR_INVALID_ARG, "t %d outside [0, %d)", it.t, c->T);
  if (!it.latent || !aligned16(it.latent))
    return fail(RC_ERR_INVALID_ARG, "latent null or not 16-B aligned");
  if (it.mode != RC_MODE_DENSE && it.mode != RC_MODE_SPARSE && it.mode != RC_MODE_REUSE)
    return fail(RC_ERR_INVALID_ARG, "mode %d is not a mode", it.mode);
  if ((r = check_ready(c, k, it.session, true))) return r;
  int bound = 0;
  if (it.mode == RC_MODE_SPARSE && (r = dirty_rows(c, it.dirty_idx, it.D, it.dirty_count, &bound)))
    return r;
  return RC_OK;
}

rc_status rc_step(rc_ctx* c, rc_cache* k, int s, float* latent, int t,
                  const uint8_t* schedule_host, const int32_t* dirty_idx, int D,
                  const int32_t* dirty_count, rc_stream stream) {
  if (!c || !k || !latent || !schedule_host)
    return fail(RC_ERR_INVALID_ARG, "rc_step: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (t < 0 || t >= c->T) return fail(RC_ERR_INVALID_ARG, "t %d outside [0, %d)", t, c->T);
  rc_batch_item it{s, latent, t, int(schedule_host[t]), dirty_idx, D, dirty_count};
  rc_status r = check_item(c, k, it);
  if (r) return r;
  return step_items(c, k, &it, 1, static_cast<cudaStream_t>(stream));
}

struct rc_graph {
  rc_ctx* ctx = nullptr;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  uint64_t launches = 0;  // kernels per replay
};

void rc_graph_destroy(rc_graph* gr) {
  if (!gr) return;
  if (gr->exec) cudaGraphExecDestroy(gr->exec);
  if (gr->graph) cudaGraphDestroy(gr->graph);
  delete gr;
}

rc_status rc_step_graph_create(rc_ctx* c, rc_cache* k, int s, float* latent, int t,
                               const uint8_t* schedule_host, const int32_t* dirty_idx, int D,
                               const int32_t* dirty_count, rc_graph** out) {
  if (!c || !k || !latent || !schedule_host || !out)
    return fail(RC_ERR_INVALID_ARG, "rc_step_graph_create: null argument");
  *out = nullptr;
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (k->host_tier) return fail(RC_ERR_INVALID_ARG, "no graphs of host-tier cache steps");
  if (c->probe_which != RC_PROBE_OFF)
    return fail(RC_ERR_INVALID_ARG, "a timing probe is enabled");
  if (t < 0 || t >= c->T) return fail(RC_ERR_INVALID_ARG, "t %d outside [0, %d)", t, c->T);
  rc_batch_item it{s, latent, t, int(schedule_host[t]), dirty_idx, D, dirty_count};
  rc_status r = check_item(c, k, it);
  if (r) return r;
  rc_graph* gr = new (std::nothrow) rc_graph();
  if (!gr) return fail(RC_ERR_OOM, "host allocation");
  gr->ctx = c;
  cudaStream_t cs = nullptr;
  cudaError_t e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking);
  if (e != cudaSuccess) {
    delete gr;
    return cuda_fail(e, "capture stream");
  }
  // the per-timestep embedding tables first, outside the capture, so that
  // replays read them instead of recomputing them
  r = fill_t_tables(c, cs);
  if (r == RC_OK && (e = cudaStreamSynchronize(cs)) != cudaSuccess) r = cuda_fail(e, "t tables");
  if (r != RC_OK) {
    cudaStreamDestroy(cs);
    delete gr;
    return r;
  }
  const uint64_t n0 = rc_launch_count();
  e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed);
  if (e == cudaSuccess) {
    r = step_items(c, k, &it, 1, cs);
    e = cudaStreamEndCapture(cs, &gr->graph);  // ends the capture whatever happened
  }
  const uint64_t n = rc_launch_count() - n0;
  g_launches.fetch_sub(n, std::memory_order_relaxed);  // counted when replayed
  cudaStreamDestroy(cs);
  if (r == RC_OK && e != cudaSuccess) r = cuda_fail(e, "stream capture");
  if (r == RC_OK && (e = cudaGraphInstantiate(&gr->exec, gr->graph, 0)) != cudaSuccess)
    r = cuda_fail(e, "graph instantiation");
  if (r != RC_OK) {
    cudaGetLastError();
    rc_graph_destroy(gr);
    return r;
  }
  gr->launches = n;
  *out = gr;
  return RC_OK;
}

rc_status rc_graph_launch(rc_graph* gr, rc_stream stream) {
  if (!gr || !gr->exec) return fail(RC_ERR_INVALID_ARG, "rc_graph_launch: null graph");
  RC_CUDA(cudaGraphLaunch(gr->exec, static_cast<cudaStream_t>(stream)), "graph launch");
  rc::count_launches(int(gr->launches));
  return RC_OK;
}

rc_status rc_step_batched(rc_ctx* c, rc_cache* k, const rc_batch_item* items, int n,
                          rc_stream stream) {
  if (!c || !k || !items) return fail(RC_ERR_INVALID_ARG, "rc_step_batched: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (n < 1 || n > c->max_batch)
    return fail(RC_ERR_INVALID_ARG, "n_items %d outside [1, %d]", n, c->max_batch);
  if (k->host_tier && n != 1)
    return fail(RC_ERR_INVALID_ARG, "a host-tier cache steps one item at a time");
  for (int i = 0; i < n; ++i) {
    rc_status r = check_item(c, k, items[i]);
    if (r) return r;
    for (int j = 0; j < i; ++j)
      if (items[j].session == items[i].session && items[j].t == items[i].t)
        return fail(RC_ERR_INVALID_ARG, "items %d and %d share session %d, t %d", j, i,
                    items[i].session, items[i].t);
  }
  return step_items(c, k, items, n, static_cast<cudaStream_t>(stream));
}

rc_status rc_step_capture(rc_ctx* c, rc_cache* k, int s, float* latent, int t,
                          const int32_t* delta_ids_host, int n_delta, float* scores,
                          rc_stream stream) {
  if (!c || !k || !latent || !delta_ids_host || !scores)
    return fail(RC_ERR_INVALID_ARG, "rc_step_capture: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (t < 0 || t >= c->T) return fail(RC_ERR_INVALID_ARG, "t %d outside [0, %d)", t, c->T);
  if (n_delta < 1 || n_delta > 8)
    return fail(RC_ERR_INVALID_ARG, "n_delta %d not in 1..8", n_delta);
  if (!aligned16(scores)) return fail(RC_ERR_INVALID_ARG, "scores not 16-B aligned");
  rc::AttnCapture cap{};
  cap.n = n_delta;
  for (int q = 0; q < n_delta; ++q) {
    if (delta_ids_host[q] < 0 || delta_ids_host[q] >= c->M)
      return fail(RC_ERR_INVALID_ARG, "delta id %d outside [0, %d)", delta_ids_host[q], c->M);
    cap.id[q] = delta_ids_host[q];
  }
  cap.out = scores;
  cap.ldo = c->M;
  cap.w = 1.f / float(c->L * c->dims.heads);
  rc_batch_item it{s, latent, t, RC_MODE_DENSE, nullptr, 0, nullptr};
  rc_status r = check_item(c, k, it);
  if (r) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  RC_CUDA(cudaMemsetAsync(scores, 0, sizeof(float) * size_t(c->N) * c->M, st), "scores reset");
  return step_items(c, k, &it, 1, st, &cap);
}

rc_status rc_localize_scores(rc_ctx* c, rc_cache* k, int s, int t, const float* latent,
                             const int32_t* delta_ids_host, int n_delta, float* scores,
                             rc_stream stream) {
  if (!c || !k || !latent || !delta_ids_host || !scores)
    return fail(RC_ERR_INVALID_ARG, "rc_localize_scores: null argument");
  if (k->ctx != c) return fail(RC_ERR_INVALID_ARG, "cache belongs to another context");
  if (k->host_tier)
    return fail(RC_ERR_INVALID_ARG, "rc_localize_scores needs a device-tier cache");
  rc_status r = check_session(k, s);
  if (r) return r;
  if (t < 0 || t >= c->T) return fail(RC_ERR_INVALID_ARG, "t %d outside [0, %d)", t, c->T);
  if (n_delta < 1 || n_delta > 8)
    return fail(RC_ERR_INVALID_ARG, "n_delta %d not in 1..8", n_delta);
  if (!aligned16(scores) || !aligned16(latent))
    return fail(RC_ERR_INVALID_ARG, "scores / latent not 16-B aligned");
  rc::AttnCapture cap{};
  cap.n = n_delta;
  for (int q = 0; q < n_delta; ++q) {
    if (delta_ids_host[q] < 0 || delta_ids_host[q] >= c->M)
      return fail(RC_ERR_INVALID_ARG, "delta id %d outside [0, %d)", delta_ids_host[q], c->M);
    cap.id[q] = delta_ids_host[q];
  }
  if ((r = check_ready(c, k, s, false))) return r;
  cap.out = scores;
  cap.ldo = c->M;
  cap.w = 1.f / float(c->L * c->dims.heads);
  const int N = c->N, d = c->d;
  const rc_global_weights& g = c->gw;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  RC_CUDA(cudaMemsetAsync(scores, 0, sizeof(float) * size_t(N) * c->M, st), "scores reset");
  // every token is a query row, in token order
  const rc::RowMap rm{nullptr, nullptr, nullptr, N, nullptr, N};
  // the state entering block 0: the patch embedding of the latent (f32),
  // then its bf16 copy for the query side of the cross-attention
  rc::Items its{};
  its.n = 1;
  its.latent[0] = const_cast<float*>(latent);
  RC_CUDA(rc::launch_patch_embed(c->dims.grid_h, c->dims.grid_w, c->dims.patch, c->dims.in_ch,
                                 static_cast<const bf16*>(g.W_e), g.b_e, g.pos, its, rm, c->xf, d,
                                 c->err, st),
          "patch_embed");
  rc::Items cast{};
  cast.n = 1;
  cast.slice[0] = c->xb;
  RC_CUDA(rc::launch_scatter_bf16(c->xf, cast, 0, rm, d, c->err, st), "embedding cast");
  for (int l = 0; l < c->L; ++l) {
    // the input of block l as cached at step t: block l - 1's output slot
    const bf16* h_in = l == 0 ? c->xb : k->slot(s, l - 1, t, 0);
    if (k->xg) {
      // (x W_xq^T + b) K^T = x G_h^T + kb_h with the folded text keys; the
      // kernel's P V output goes to scratch, only the captured columns matter
      rc::XqItems xi{};
      xi.n = 1;
      xi.grow[0] = int(k->xg_row(s, l));
      xi.vrow[0] = (s * c->L + l) * c->M;
      RC_CUDA(rc::launch_xattn_fused(h_in, d, k->xg, k->xgb, int(k->xg_rows()), k->text + d,
                                     2 * d, k->sessions * c->L * c->M, xi, c->M, c->ob, d,
                                     c->dims.heads, c->dh, rm, c->err, st, &cap),
              "scores(cross)");
    } else {
      rc::GemmEpi e{};
      e.mode = rc::EPI_BIAS_BF16;
      e.bias = c->lw[l].b_xq;
      e.out_bf = c->q;
      e.ld_out = d;
      e.gate_off = -1;
      e.err = c->err;
      RC_CUDA(rc::launch_gemm(h_in, d, static_cast<const bf16*>(c->lw[l].W_xq), N, nullptr, d,
                              d, e, st), "gemm(xq)");
      StepItems si;
      si.its.n = 1;
      si.session[0] = s;
      si.t[0] = t;
      RC_CUDA(rc::launch_attention(c->q, d, k->text, k->text + d, 2 * d,
                                   k->sessions * c->L * c->M, text_kv_rows(k, si, l), c->M,
                                   c->ob, d, c->dims.heads, c->dh, rm, c->err, c->as, st, &cap),
              "scores(cross)");
    }
  }
  return RC_OK;
}

rc_status rc_prompt_similarity(const float* e_minus, const float* e_plus, int dim, float* s_out) {
  if (!e_minus || !e_plus || !s_out || dim <= 0)
    return fail(RC_ERR_INVALID_ARG, "rc_prompt_similarity: null argument or dim <= 0");
  double dot = 0.0, na = 0.0, nb = 0.0;
  for (int i = 0; i < dim; ++i) {
    dot += double(e_minus[i]) * e_plus[i];
    na += double(e_minus[i]) * e_minus[i];
    nb += double(e_plus[i]) * e_plus[i];
  }
  if (!(na > 0.0) || !(nb > 0.0))
    return fail(RC_ERR_INVALID_ARG, "rc_prompt_similarity: zero embedding");
  *s_out = float(dot / (std::sqrt(na) * std::sqrt(nb)));
  return RC_OK;
}

rc_status rc_reuse_schedule(float s, float tau_s, float rho, int T, uint8_t* modes_out) {
  if (!modes_out || T <= 0) return fail(RC_ERR_INVALID_ARG, "rc_reuse_schedule: T or output");
  if (!(rho >= 0.f && rho <= 1.f) || s != s || tau_s != tau_s)
    return fail(RC_ERR_INVALID_ARG, "rc_reuse_schedule: rho outside [0, 1] or NaN input");
  const int t_reuse = s >= tau_s ? T : int(std::floor(double(rho) * T));
  for (int t = 0; t < T; ++t) modes_out[t] = uint8_t(t < t_reuse ? RC_MODE_REUSE : RC_MODE_SPARSE);
  return RC_OK;
}

rc_status rc_step_dense(rc_ctx* c, rc_cache* k, int s, float* latent, int t, rc_stream stream) {
  if (!c) return fail(RC_ERR_INVALID_ARG, "rc_step_dense: null context");
  std::vector<uint8_t> sched(size_t(c->T), uint8_t(RC_MODE_DENSE));
  return rc_step(c, k, s, latent, t, sched.data(), nullptr, 0, nullptr, stream);
}

rc_status rc_linear(rc_ctx* c, const void* x, const void* W, const float* b, float* y, int rows,
                    int n, int kdim, rc_stream stream) {
  if (!c || !x || !W || !y) return fail(RC_ERR_INVALID_ARG, "rc_linear: null argument");
  if (rows < 0 || n <= 0 || kdim <= 0 || n % 128 || kdim % 64)
    return fail(RC_ERR_SHAPE, "rc_linear: rows %d n %d k %d (n %% 128, k %% 64 must be 0)", rows,
                n, kdim);
  if (!aligned16(x) || !aligned16(W) || !aligned16(y) || (b && !aligned16(b)))
    return fail(RC_ERR_INVALID_ARG, "rc_linear: pointers must be 16-B aligned");
  rc::GemmEpi e{};
  e.mode = rc::EPI_F32;
  e.bias = b;
  e.out_f = y;
  e.ld_out = n;
  e.err = c->err;
  RC_CUDA(rc::launch_gemm(static_cast<const bf16*>(x), kdim, static_cast<const bf16*>(W), rows,
                          nullptr, n, kdim, e, static_cast<cudaStream_t>(stream)),
          "gemm(linear)");
  return RC_OK;
}

rc_status rc_attention(rc_ctx* c, const void* Q, int ldq, const void* K, const void* V, int ldkv,
                       int Nq, int Nk, void* O, int ldo, rc_stream stream) {
  if (!c || !Q || !K || !V || !O) return fail(RC_ERR_INVALID_ARG, "rc_attention: null argument");
  const int hd = c->dims.heads * c->dh;
  if (Nq < 0 || Nk < 0 || ldq < hd || ldkv < hd || ldo < hd || ldq % 8 || ldkv % 8 || ldo % 8)
    return fail(RC_ERR_SHAPE, "rc_attention: Nq %d Nk %d ldq %d ldkv %d ldo %d", Nq, Nk, ldq,
                ldkv, ldo);
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O))
    return fail(RC_ERR_INVALID_ARG, "rc_attention: pointers must be 16-B aligned");
  if (Nq == 0) return RC_OK;
  if (Nk == 0) return fail(RC_ERR_SHAPE, "rc_attention: Nk = 0 with queries");
  rc::AttnItems ai{};
  ai.n = 1;
  const rc::RowMap rm{nullptr, nullptr, nullptr, Nq, nullptr, Nk};
  RC_CUDA(rc::launch_attention(static_cast<const bf16*>(Q), ldq, static_cast<const bf16*>(K),
                               static_cast<const bf16*>(V), ldkv, Nk, ai, Nk,
                               static_cast<bf16*>(O), ldo, c->dims.heads, c->dh, rm, c->err,
                               c->as, static_cast<cudaStream_t>(stream)),
          "attention");
  return RC_OK;
}

rc_status rc_probe_enable(rc_ctx* c, int which, int capacity) {
  if (!c) return fail(RC_ERR_INVALID_ARG, "rc_probe_enable: null context");
  if (which < RC_PROBE_OFF || which > RC_PROBE_LN || capacity < 0 || capacity > 1 << 20)
    return fail(RC_ERR_INVALID_ARG, "rc_probe_enable: which %d capacity %d", which, capacity);
  probe_free(c);
  if (which == RC_PROBE_OFF) return RC_OK;
  c->probe_ev.resize(size_t(2) * capacity);
  for (auto& e : c->probe_ev) RC_CUDA(cudaEventCreate(&e), "cudaEventCreate");
  c->probe_which = which;
  return RC_OK;
}

rc_status rc_probe_read_each(rc_ctx* c, float* ms_out, int capacity, int* launches) {
  if (!c || !launches || (capacity > 0 && !ms_out) || capacity < 0)
    return fail(RC_ERR_INVALID_ARG, "rc_probe_read_each: null or negative argument");
  const int n = c->probe_n;
  for (int i = 0; i < n; ++i) {
    RC_CUDA(cudaEventSynchronize(c->probe_ev[2 * i + 1]), "cudaEventSynchronize");
    float ms = 0.f;
    RC_CUDA(cudaEventElapsedTime(&ms, c->probe_ev[2 * i], c->probe_ev[2 * i + 1]),
            "cudaEventElapsedTime");
    if (i < capacity) ms_out[i] = ms;
  }
  *launches = n;
  c->probe_n = 0;
  return RC_OK;
}

rc_status rc_probe_read(rc_ctx* c, double* total_ms, int* launches) {
  if (!c || !total_ms || !launches) return fail(RC_ERR_INVALID_ARG, "rc_probe_read: null");
  std::vector<float> ms(size_t(c->probe_n));
  rc_status s = rc_probe_read_each(c, ms.data(), int(ms.size()), launches);
  if (s != RC_OK) return s;
  double tot = 0.0;
  for (float v : ms) tot += v;
  *total_ms = tot;
  return RC_OK;
}

rc_status rc_selftest_wait(rc_ctx* c, int timeout_us, int set_flag, rc_stream stream) {
  if (!c) return fail(RC_ERR_INVALID_ARG, "rc_selftest_wait: null context");
  if (timeout_us < 1 || timeout_us > 1000000)
    return fail(RC_ERR_INVALID_ARG, "rc_selftest_wait: timeout %d us not in 1 .. 10^6", timeout_us);
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      c->wait_flag, 1000ull * unsigned(timeout_us), set_flag ? 1 : 0, c->err);
  RC_CUDA(cudaGetLastError(), "selftest wait");
  rc::count_launches(1);
  return RC_OK;
}

rc_status rc_sync(rc_ctx* c, rc_stream stream) {
  if (!c) return fail(RC_ERR_INVALID_ARG, "rc_sync: null context");
  RC_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream sync");
  unsigned w = 0;
  RC_CUDA(cudaMemcpy(&w, c->err, sizeof(w), cudaMemcpyDeviceToHost), "read error word");
  if (w) {
    RC_CUDA(cudaMemset(c->err, 0, sizeof(unsigned)), "clear error word");
    if (w & rc::DEVERR_TIMEOUT) return fail(RC_ERR_TIMEOUT, "a bounded device wait gave up");
    return fail(RC_ERR_DEVICE_ASSERT, "device check failed (bits 0x%x: %s%s)", w,
                (w & rc::DEVERR_INDEX) ? "index out of range " : "",
                (w & rc::DEVERR_COUNT) ? "count out of range" : "");
  }
  return RC_OK;
}

}  // extern "C"
