// Trace loading: validation, event ordering and upload (host side of the
// C ABI).  A trace is the paper's workload model (Sec. III-A): sessions of
// turns with arrival a_{s,k}, completion c_{s,k} and KV sizes.  The event
// stream is the runtime's event FIFO of Sec. IV-A (request arrival = gap
// closure, completion = gap onset).
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "common.cuh"

using namespace unison;

extern "C" const char *unison_strerror(int code) {
  switch (code) {
    case UNISON_OK: return "ok";
    case UNISON_ERR_ARG: return "invalid argument";
    case UNISON_ERR_IO: return "file could not be read";
    case UNISON_ERR_FORMAT: return "trace breaks its ordering rules";
    case UNISON_ERR_RANGE: return "value beyond a documented limit";
    case UNISON_ERR_CUDA: return "CUDA runtime error";
    case UNISON_ERR_OOM: return "out of memory";
    case UNISON_ERR_LOG_FULL: return "decision log capacity exceeded";
    case UNISON_ERR_TIMEOUT: return "bounded device wait gave up";
    case UNISON_ERR_CAPACITY: return "resident-list bound exceeded";
    default: return "unknown status";
  }
}

extern "C" int unison_version(void) { return 10000; }

namespace {

struct HostEvent {
  uint64_t time;
  uint32_t session;
  uint32_t turn;  // index of the turn inside its session
  uint32_t arrival;  // 1 = arrival, 0 = completion
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int check_turns(const unison_turns *t) {
  if (!t || !t->turn_off) return UNISON_ERR_ARG;
  const uint64_t S = t->n_sessions, T = t->n_turns;
  if (S >= kIdMask) return UNISON_ERR_RANGE;  // ids must leave ~id != 0 in 24 bits
  if (T >= (1ull << 31)) return UNISON_ERR_RANGE;
  if (T > 0 && (!t->arrival_us || !t->completion_us || !t->in_tok || !t->out_tok)) return UNISON_ERR_ARG;
  if (t->turn_off[0] != 0 || t->turn_off[S] != T) return UNISON_ERR_FORMAT;
  const uint64_t lim = 1ull << 31;
  for (uint64_t s = 0; s < S; s++) {
    const uint64_t b = t->turn_off[s], e = t->turn_off[s + 1];
    if (e <= b) return UNISON_ERR_FORMAT;
    if (e - b >= 65536) return UNISON_ERR_RANGE;
    if (s && t->arrival_us[b] < t->arrival_us[t->turn_off[s - 1]]) return UNISON_ERR_FORMAT;
    for (uint64_t i = b; i < e; i++) {
      const uint64_t a = t->arrival_us[i], c = t->completion_us[i];
      if (c <= a) return UNISON_ERR_FORMAT;
      if (c - a >= lim) return UNISON_ERR_RANGE;
      if (t->in_tok[i] == 0 || t->out_tok[i] < t->in_tok[i]) return UNISON_ERR_FORMAT;
      if (i > b) {
        if (a <= t->completion_us[i - 1]) return UNISON_ERR_FORMAT;
        if (a - t->completion_us[i - 1] >= lim) return UNISON_ERR_RANGE;
        if (t->in_tok[i] < t->out_tok[i - 1]) return UNISON_ERR_FORMAT;
      }
    }
  }
  return UNISON_OK;
}

}  // namespace

extern "C" int unison_trace_create(const unison_turns *turns, unison_trace **out) {
  if (!out) return UNISON_ERR_ARG;
  *out = nullptr;
  int rc = check_turns(turns);
  if (rc != UNISON_OK) return rc;
  const uint64_t S = turns->n_sessions, T = turns->n_turns, E = 2 * T;

  // Event order: time, then completions before arrivals, then session id.
  std::vector<HostEvent> ev;
  try {
    ev.resize(E);
  } catch (const std::bad_alloc &) {
    return UNISON_ERR_OOM;
  }
  uint64_t m = 0;
  for (uint64_t s = 0; s < S; s++)
    for (uint64_t i = turns->turn_off[s]; i < turns->turn_off[s + 1]; i++) {
      const uint32_t k = (uint32_t)(i - turns->turn_off[s]);
      ev[m++] = {turns->arrival_us[i], (uint32_t)s, k, 1u};
      ev[m++] = {turns->completion_us[i], (uint32_t)s, k, 0u};
    }
  std::sort(ev.begin(), ev.end(), [](const HostEvent &x, const HostEvent &y) {
    if (x.time != y.time) return x.time < y.time;
    if (x.arrival != y.arrival) return x.arrival < y.arrival;
    return x.session < y.session;
  });
  for (uint64_t i = 1; i < E; i++)
    if (ev[i].time - ev[i - 1].time >= (1ull << 31)) return UNISON_ERR_RANGE;

  unison_trace *tr = new (std::nothrow) unison_trace();
  if (!tr) return UNISON_ERR_OOM;
  tr->n_sessions = (uint32_t)S;
  tr->n_turns = T;
  tr->n_events = E;
  size_t off = 0;
  tr->off_ev = off;        off = align_up(off + 16 * E, 256);
  tr->off_prev_out = off;  off = align_up(off + 4 * E, 256);
  tr->off_nref = off;      off = align_up(off + 4 * E, 256);
  tr->off_prev_ev = off;   off = align_up(off + 4 * E, 256);
  tr->off_turn_ev = off;   off = align_up(off + 8 * T, 256);
  tr->off_turn_t = off;    off = align_up(off + 8 * T, 256);
  tr->off_turn_off = off;  off = align_up(off + 4 * (S + 1), 256);
  tr->off_tps = off;       off = align_up(off + 4 * S + 4, 256);
  tr->block_bytes = off;
  // Page-locked staging makes the upload a true async DMA; without a CUDA
  // driver (host-only validation) ordinary memory serves as staging.
  if (cudaMallocHost(&tr->h_block, tr->block_bytes) != cudaSuccess) {
    cudaGetLastError();
    tr->h_block = std::malloc(tr->block_bytes);
    tr->h_pinned = false;
    if (!tr->h_block) {
      delete tr;
      return UNISON_ERR_OOM;
    }
  } else {
    tr->h_pinned = true;
  }
  std::memset(tr->h_block, 0, tr->block_bytes);

  uint4 *hev = tr->h<uint4>(tr->off_ev);
  uint32_t *prev_out = tr->h<uint32_t>(tr->off_prev_out);
  uint32_t *nref = tr->h<uint32_t>(tr->off_nref);
  uint32_t *prev_ev = tr->h<uint32_t>(tr->off_prev_ev);
  uint32_t *turn_ev = tr->h<uint32_t>(tr->off_turn_ev);
  uint32_t *turn_t = tr->h<uint32_t>(tr->off_turn_t);
  uint32_t *toff = tr->h<uint32_t>(tr->off_turn_off);
  uint32_t *tps = tr->h<uint32_t>(tr->off_tps);

  uint32_t min_out = 0xFFFFFFFFu;
  for (uint64_t s = 0; s <= S; s++) toff[s] = (uint32_t)turns->turn_off[s];
  for (uint64_t s = 0; s < S; s++) tps[s] = (uint32_t)(turns->turn_off[s + 1] - turns->turn_off[s]);
  for (uint64_t i = 0; i < T; i++) {
    turn_t[2 * i] = (uint32_t)turns->arrival_us[i];
    turn_t[2 * i + 1] = (uint32_t)turns->completion_us[i];
    min_out = std::min(min_out, turns->out_tok[i]);
  }
  tr->min_out_tok = T ? min_out : 1;
  for (uint64_t e = 0; e < E; e++) {
    const HostEvent &x = ev[e];
    const uint64_t ti = turns->turn_off[x.session] + x.turn;
    const uint32_t ts = tps[x.session];
    turn_ev[2 * ti + (x.arrival ? 0 : 1)] = (uint32_t)e;
    uint32_t w1 = x.session;
    if (x.arrival) {
      w1 |= kEvArrival;
      if (x.turn == 0) w1 |= kEvEdge;
      hev[e] = make_uint4((uint32_t)x.time, w1, turns->in_tok[ti], turns->out_tok[ti]);
      prev_out[e] = x.turn ? turns->out_tok[ti - 1] : 0u;
    } else {
      if (x.turn + 1 == ts) w1 |= kEvEdge;
      hev[e] = make_uint4((uint32_t)x.time, w1, 0u, 0u);
      prev_out[e] = 0u;
    }
  }
  for (uint64_t e = 0; e < E; e++) {
    const HostEvent &x = ev[e];
    nref[e] = kNoRef;
    prev_ev[e] = kNoRef;
    if (x.arrival) {
      const uint64_t ti = turns->turn_off[x.session] + x.turn;
      if (x.turn + 1 < tps[x.session]) nref[e] = turn_ev[2 * (ti + 1)];
      if (x.turn > 0) prev_ev[e] = turn_ev[2 * (ti - 1) + 1];
    }
  }
  *out = tr;
  return UNISON_OK;
}

extern "C" int unison_trace_load(const char *path, unison_trace **out) {
  if (!path || !out) return UNISON_ERR_ARG;
  *out = nullptr;
  FILE *f = std::fopen(path, "rb");
  if (!f) return UNISON_ERR_IO;
  unsigned char head[16];
  int rc = UNISON_OK;
  if (std::fread(head, 1, 16, f) != 16 || std::memcmp(head, "UTR1", 4) != 0) {
    std::fclose(f);
    return UNISON_ERR_FORMAT;
  }
  auto rd32 = [](const unsigned char *p) {
    return (uint32_t)p[0] | (uint32_t)p[1] << 8 | (uint32_t)p[2] << 16 | (uint32_t)p[3] << 24;
  };
  const uint64_t S = rd32(head + 4);
  const uint64_t T = (uint64_t)rd32(head + 8) | (uint64_t)rd32(head + 12) << 32;
  if (S >= kIdMask || T >= (1ull << 31)) {
    std::fclose(f);
    return UNISON_ERR_RANGE;
  }
  std::vector<uint64_t> toff, arr, cmp;
  std::vector<uint32_t> in, outv;
  try {
    toff.resize(S + 1);
    arr.resize(T);
    cmp.resize(T);
    in.resize(T);
    outv.resize(T);
  } catch (const std::bad_alloc &) {
    std::fclose(f);
    return UNISON_ERR_OOM;
  }
  // Little-endian payload; decode byte by byte so the host's order is irrelevant.
  auto read_u64 = [&](std::vector<uint64_t> &v) {
    std::vector<unsigned char> b(8 * v.size());
    if (std::fread(b.data(), 1, b.size(), f) != b.size()) return false;
    for (size_t i = 0; i < v.size(); i++) {
      uint64_t x = 0;
      for (int j = 7; j >= 0; j--) x = (x << 8) | b[8 * i + j];
      v[i] = x;
    }
    return true;
  };
  auto read_u32 = [&](std::vector<uint32_t> &v) {
    std::vector<unsigned char> b(4 * v.size());
    if (std::fread(b.data(), 1, b.size(), f) != b.size()) return false;
    for (size_t i = 0; i < v.size(); i++) v[i] = rd32(&b[4 * i]);
    return true;
  };
  if (!read_u64(toff) || !read_u64(arr) || !read_u64(cmp) || !read_u32(in) || !read_u32(outv))
    rc = UNISON_ERR_FORMAT;
  std::fclose(f);
  if (rc != UNISON_OK) return rc;
  unison_turns t;
  t.n_sessions = (uint32_t)S;
  t.reserved = 0;
  t.n_turns = T;
  t.turn_off = toff.data();
  t.arrival_us = arr.data();
  t.completion_us = cmp.data();
  t.in_tok = in.data();
  t.out_tok = outv.data();
  return unison_trace_create(&t, out);
}

extern "C" int unison_trace_upload(unison_trace *tr, void *cuda_stream) {
  if (!tr) return UNISON_ERR_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISON_ERR_CUDA;
  if (tr->d_block && tr->device != dev) return UNISON_ERR_ARG;
  if (!tr->d_block) {
    if (unison_fault_alloc() || cudaMalloc(&tr->d_block, tr->block_bytes) != cudaSuccess) {
      cudaGetLastError();
      tr->d_block = nullptr;
      return UNISON_ERR_OOM;
    }
    tr->device = dev;
  }
  if (cudaMemcpyAsync(tr->d_block, tr->h_block, tr->block_bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
    return UNISON_ERR_CUDA;
  tr->last_stream = st;
  return UNISON_OK;
}

extern "C" void unison_trace_free(unison_trace *tr) {
  if (!tr) return;
  if (tr->d_block) {
    cudaDeviceSynchronize();
    cudaFree(tr->d_block);
  }
  if (tr->h_block) {
    if (tr->h_pinned)
      cudaFreeHost(tr->h_block);
    else
      std::free(tr->h_block);
  }
  delete tr;
}

extern "C" int unison_trace_info(const unison_trace *tr, uint32_t *n_sessions, uint64_t *n_turns,
                                 uint64_t *n_events) {
  if (!tr) return UNISON_ERR_ARG;
  if (n_sessions) *n_sessions = tr->n_sessions;
  if (n_turns) *n_turns = tr->n_turns;
  if (n_events) *n_events = tr->n_events;
  return UNISON_OK;
}

extern "C" uint64_t unison_trace_device_bytes(const unison_trace *tr) {
  return tr ? (uint64_t)tr->block_bytes : 0;
}
