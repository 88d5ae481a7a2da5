// Cross-session serving scheduler (see include/regioncache.h, rc_server_*):
// sessions join and leave between steps; every tick runs one batched
// denoising step over the sessions it picks.  Host code only: the compute is
// rc_step_batched's.
#include <stdio.h>

#include <algorithm>
#include <new>
#include <vector>

#include "../../include/regioncache.h"
#include "kernels.h"

namespace {

struct Turn {
  int session;
  float* latent;
  std::vector<uint8_t> schedule;  // [timesteps]
  const int32_t* dirty_idx;
  int D;
  const int32_t* dirty_count;
  int t_next;              // next step of the turn
  unsigned long long seq;  // admission order
  long long last_tick;     // tick that last stepped it (-1: none yet)
};

rc_status fail(rc_status s, const char* msg) {
  rc::set_last_error(msg);
  return s;
}

}  // namespace

struct rc_server {
  rc_ctx* ctx;
  rc_cache* cache;
  int max_items;
  int timesteps;
  int sessions;
  unsigned long long seq = 0;
  long long tick = 0;
  std::vector<Turn> active;
};

extern "C" {

rc_status rc_server_create(rc_ctx* ctx, rc_cache* cache, int max_items, rc_server** out) {
  if (!ctx || !cache || !out) return fail(RC_ERR_INVALID_ARG, "rc_server_create: null argument");
  *out = nullptr;
  if (rc::cache_context(cache) != ctx)
    return fail(RC_ERR_INVALID_ARG, "rc_server_create: cache belongs to another context");
  const int cap = rc::cache_host_tier(cache) ? 1 : rc::ctx_max_batch(ctx);
  if (max_items < 1 || max_items > cap) {
    char msg[160];
    snprintf(msg, sizeof(msg), "rc_server_create: max_items %d outside [1, %d]", max_items, cap);
    return fail(RC_ERR_INVALID_ARG, msg);
  }
  rc_server* s = new (std::nothrow) rc_server();
  if (!s) return fail(RC_ERR_OOM, "host allocation");
  s->ctx = ctx;
  s->cache = cache;
  s->max_items = max_items;
  s->timesteps = rc::ctx_timesteps(ctx);
  s->sessions = rc::cache_sessions(cache);
  *out = s;
  return RC_OK;
}

void rc_server_destroy(rc_server* s) { delete s; }

rc_status rc_server_admit(rc_server* s, int session, float* latent, const uint8_t* schedule_host,
                          const int32_t* dirty_idx, int D, const int32_t* dirty_count) {
  if (!s || !latent || !schedule_host)
    return fail(RC_ERR_INVALID_ARG, "rc_server_admit: null argument");
  if (session < 0 || session >= s->sessions)
    return fail(RC_ERR_INVALID_ARG, "rc_server_admit: session out of range");
  for (const Turn& u : s->active)
    if (u.session == session)
      return fail(RC_ERR_INVALID_ARG, "rc_server_admit: the session's turn is still running");
  Turn u;
  u.session = session;
  u.latent = latent;
  u.schedule.assign(schedule_host, schedule_host + s->timesteps);
  bool sparse = false;
  for (uint8_t m : u.schedule) {
    if (m != RC_MODE_DENSE && m != RC_MODE_SPARSE && m != RC_MODE_REUSE)
      return fail(RC_ERR_INVALID_ARG, "rc_server_admit: schedule holds a value that is no mode");
    sparse |= m == RC_MODE_SPARSE;
  }
  if (sparse && (D < -1 || (D == -1 && !dirty_count) || (D != 0 && !dirty_idx)))
    return fail(RC_ERR_INVALID_ARG, "rc_server_admit: SPARSE steps need a dirty list");
  u.dirty_idx = dirty_idx;
  u.D = D;
  u.dirty_count = dirty_count;
  u.t_next = 0;
  u.seq = s->seq++;
  u.last_tick = -1;
  s->active.push_back(u);
  return RC_OK;
}

rc_status rc_server_tick(rc_server* s, rc_stream stream, int* sessions_out, int* n_out) {
  if (!s || !n_out) return fail(RC_ERR_INVALID_ARG, "rc_server_tick: null argument");
  *n_out = 0;
  if (s->active.empty()) return RC_OK;
  // least recently stepped first, then admission order: with more running
  // turns than items per tick, every turn advances in round robin
  std::vector<int> order(s->active.size());
  for (size_t i = 0; i < order.size(); ++i) order[i] = int(i);
  std::sort(order.begin(), order.end(), [&](int a, int b) {
    const Turn &x = s->active[size_t(a)], &y = s->active[size_t(b)];
    if (x.last_tick != y.last_tick) return x.last_tick < y.last_tick;
    return x.seq < y.seq;
  });
  const int n = std::min(int(order.size()), s->max_items);
  rc_batch_item items[RC_MAX_BATCH];
  for (int i = 0; i < n; ++i) {
    const Turn& u = s->active[size_t(order[size_t(i)])];
    const int mode = u.schedule[size_t(u.t_next)];
    items[i] = rc_batch_item{u.session, u.latent, u.t_next, mode,
                             mode == RC_MODE_SPARSE ? u.dirty_idx : nullptr,
                             mode == RC_MODE_SPARSE ? u.D : 0,
                             mode == RC_MODE_SPARSE ? u.dirty_count : nullptr};
  }
  rc_status r = rc_step_batched(s->ctx, s->cache, items, n, stream);
  if (r != RC_OK) return r;  // nothing advanced; rc_last_error() says why
  for (int i = 0; i < n; ++i) {
    Turn& u = s->active[size_t(order[size_t(i)])];
    ++u.t_next;
    u.last_tick = s->tick;
    if (sessions_out) sessions_out[i] = u.session;
  }
  *n_out = n;
  ++s->tick;
  s->active.erase(std::remove_if(s->active.begin(), s->active.end(),
                                 [&](const Turn& u) { return u.t_next >= s->timesteps; }),
                  s->active.end());
  return RC_OK;
}

rc_status rc_server_state(const rc_server* s, int session, int* next_t) {
  if (!s || !next_t) return fail(RC_ERR_INVALID_ARG, "rc_server_state: null argument");
  *next_t = -1;
  for (const Turn& u : s->active)
    if (u.session == session) *next_t = u.t_next;
  return RC_OK;
}

int rc_server_running(const rc_server* s) { return s ? int(s->active.size()) : 0; }

}  // extern "C"
