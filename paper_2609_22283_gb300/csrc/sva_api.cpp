// Host runtime of the C ABI declared in include/sva.h.
//
// Owns the (seq, chunk, level) -> slot table of the KV cache (Section 3.2),
// the integer rules of context selection (Eq. 2-3), pipeline rounds (Eq. 6)
// and availability (Eq. 7), the validation of every launch, the TMA
// descriptors, and the launches of the kernels.  Device memory is always
// the caller's.
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "proj.h"
#include "sva.h"

namespace {

thread_local std::string g_err;

sva_status fail(sva_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

sva_status ok() {
  g_err.clear();
  return SVA_OK;
}

sva_status cuda_fail(cudaError_t e, const char* what) {
  return fail(SVA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// True when `p` points into device memory of `device`.
bool on_device(const void* p, int device) {
  cudaPointerAttributes attr;
  const cudaError_t e = cudaPointerGetAttributes(&attr, p);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice && attr.device == device;
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

struct Layout {
  int T = 0;
  int Tpad = 0;
  size_t slot_bytes = 0;  // whole slot pool
  size_t tab_t = 0, tab_h = 0, tab_w = 0, tab_ht = 0, tab_wt = 0, status = 0;  // byte offsets
  size_t total = 0;
};

bool geometry_valid(const sva_geometry* g, sva_status* st) {
  *st = SVA_ERR_INVALID_ARGUMENT;
  if (g == nullptr) {
    fail(*st, "geometry is NULL");
    return false;
  }
  if (g->num_heads < 1 || g->num_heads > 128 || g->frames < 1 || g->grid_h < 1 ||
      g->grid_w < 1 || g->num_slots < 1 || g->max_frames < 1 || g->max_frames > (1 << 20)) {
    fail(*st, "geometry out of range (H=%d F=%d Hp=%d Wp=%d slots=%d max_frames=%d)",
         g->num_heads, g->frames, g->grid_h, g->grid_w, g->num_slots, g->max_frames);
    return false;
  }
  const long long T = (long long)g->frames * g->grid_h * g->grid_w;
  if (T > 65536) {
    fail(*st, "T = %lld tokens per chunk exceeds 65536", T);
    return false;
  }
  if (g->head_dim != 64 && g->head_dim != 128) {
    *st = SVA_ERR_UNSUPPORTED;
    fail(*st, "head_dim %d is not 64 or 128", g->head_dim);
    return false;
  }
  if (g->rope_pairs[0] < 0 || g->rope_pairs[1] < 0 || g->rope_pairs[2] < 0 ||
      g->rope_pairs[0] + g->rope_pairs[1] + g->rope_pairs[2] != g->head_dim / 2) {
    fail(*st, "rope_pairs (%d, %d, %d) must be >= 0 and sum to head_dim/2 = %d",
         g->rope_pairs[0], g->rope_pairs[1], g->rope_pairs[2], g->head_dim / 2);
    return false;
  }
  if (!(g->rope_theta > 1.0) || !std::isfinite(g->rope_theta)) {
    fail(*st, "rope_theta must be finite and > 1");
    return false;
  }
  const long long Tpad = (T + sva::kTile - 1) / sva::kTile * sva::kTile;
  const long long rows = (long long)g->num_slots * 2 * g->num_heads * Tpad;
  if (rows >= (1ll << 31)) {
    *st = SVA_ERR_CAPACITY;
    fail(*st, "slot pool has %lld rows; TMA coordinates need < 2^31", rows);
    return false;
  }
  return true;
}

Layout layout_of(const sva_geometry& g) {
  Layout L;
  L.T = g.frames * g.grid_h * g.grid_w;
  L.Tpad = (L.T + sva::kTile - 1) / sva::kTile * sva::kTile;
  L.slot_bytes = (size_t)g.num_slots * 2 * g.num_heads * L.Tpad * g.head_dim * 2;
  size_t off = round_up(L.slot_bytes, 256);
  L.tab_t = off;
  off = round_up(off + (size_t)g.max_frames * g.rope_pairs[0] * sizeof(float2), 256);
  L.tab_h = off;
  off = round_up(off + (size_t)g.grid_h * g.rope_pairs[1] * sizeof(float2), 256);
  L.tab_w = off;
  off = round_up(off + (size_t)g.grid_w * g.rope_pairs[2] * sizeof(float2), 256);
  // the patch-row and patch-column tables again, pair-major ([pair][position]),
  // for readers whose neighbouring threads hold neighbouring tokens
  L.tab_ht = off;
  off = round_up(off + (size_t)g.grid_h * g.rope_pairs[1] * sizeof(float2), 256);
  L.tab_wt = off;
  off = round_up(off + (size_t)g.grid_w * g.rope_pairs[2] * sizeof(float2), 256);
  L.status = off;
  L.total = off + 256;
  return L;
}

struct SlotInfo {
  bool bound = false;
  bool resident = false;
  int32_t seq = 0, chunk = 0, level = 0;
};

using StateKey = std::tuple<int32_t, int32_t, int32_t>;

// (cos, sin) of pos * theta^(-i / pairs) for pos in [0, npos), i in [0, pairs),
// evaluated in fp64 and rounded once to fp32.
std::vector<float2> rope_table(int npos, int pairs, double theta) {
  std::vector<float2> t((size_t)npos * pairs);
  for (int pos = 0; pos < npos; ++pos)
    for (int i = 0; i < pairs; ++i) {
      const double omega = std::pow(theta, -(double)i / (double)pairs);
      const double a = (double)pos * omega;
      t[(size_t)pos * pairs + i] = make_float2((float)std::cos(a), (float)std::sin(a));
    }
  return t;
}

sva_status encode_2d_kv(CUtensorMap* m, void* base, const sva_geometry& g, const Layout& L) {
  auto fn = encode_fn();
  if (!fn) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  const cuuint64_t rows = (cuuint64_t)g.num_slots * 2 * g.num_heads * L.Tpad;
  cuuint64_t dims[2] = {(cuuint64_t)g.head_dim, rows};
  cuuint64_t strides[1] = {(cuuint64_t)g.head_dim * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)sva::kTile};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(kv) failed: %d", (int)r);
  return SVA_OK;
}

sva_status encode_4d_q(CUtensorMap* m, const void* q, const sva_geometry& g, int T, int n_nodes) {
  auto fn = encode_fn();
  if (!fn) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  const cuuint64_t d = (cuuint64_t)g.head_dim, H = (cuuint64_t)g.num_heads;
  cuuint64_t dims[4] = {d, H, (cuuint64_t)T, (cuuint64_t)n_nodes};
  cuuint64_t strides[3] = {d * 2, H * d * 2, (cuuint64_t)T * H * d * 2};
  cuuint32_t box[4] = {64, 1, (cuuint32_t)sva::kTile, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(q), dims, strides, box,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(q) failed: %d", (int)r);
  return SVA_OK;
}

int phi(int policy, int j, int r) {
  switch (policy) {
    case SVA_POLICY_CLEAN:
      return 0;
    case SVA_POLICY_SAME:
      return j;
    case SVA_POLICY_PROG:
      return j - r > 0 ? j - r : 0;
  }
  return -1;
}

}  // namespace

struct sva_cache {
  sva_geometry g{};
  Layout L;
  char* base = nullptr;
  int device = 0;
  int num_sms = 0;
  std::vector<SlotInfo> slots;
  std::map<StateKey, int32_t> index;
  std::vector<int32_t> free_slots;  // stack, lowest slot on top
  CUtensorMap tmap_kv{};
  const void* q_cached = nullptr;
  int q_cached_n = -1;
  CUtensorMap tmap_q{};
  int fault_mode = 0;  // one-shot test hook, see sva_debug_inject
  uint64_t timeout_ns = sva::kDefaultWaitTimeoutNs;
  char* ws = nullptr;  // caller's split workspace (sva_cache_set_workspace), or null
};

namespace {

sva_status check_device(const sva_cache* c) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != c->device)
    return fail(SVA_ERR_INVALID_ARGUMENT, "cache lives on device %d but device %d is current",
                c->device, dev);
  return SVA_OK;
}

// Validates that slot `s` is bound to (seq, chunk, level) and resident.
sva_status check_own(const sva_cache* c, const sva_node& n, int i, bool need_resident) {
  if (n.own_slot < 0 || n.own_slot >= c->g.num_slots)
    return fail(SVA_ERR_INVALID_ARGUMENT, "node %d: own_slot %d out of range", i, n.own_slot);
  const SlotInfo& s = c->slots[n.own_slot];
  if (!s.bound || s.seq != n.seq || s.chunk != n.chunk || s.level != n.level)
    return fail(SVA_ERR_INVALID_ARGUMENT,
                "node %d: own_slot %d is not bound to (seq %d, chunk %d, level %d)", i, n.own_slot,
                n.seq, n.chunk, n.level);
  if (need_resident && !s.resident)
    return fail(SVA_ERR_NOT_RESIDENT, "node %d: own_slot %d has not been written", i, n.own_slot);
  return SVA_OK;
}

// Split workspace: room for 4 waves of split work items (one per SM and
// wave), each 256 query rows x (d + 2) fp32, after one arrival counter per
// item.
int ws_items(const sva_cache* c) { return 4 * c->num_sms; }
size_t ws_item_bytes(const sva_cache* c) { return (size_t)256 * (c->g.head_dim + 2) * 4; }
size_t ws_counter_bytes(const sva_cache* c) { return round_up((size_t)ws_items(c) * 4, 256); }
size_t ws_total_bytes(const sva_cache* c) {
  return ws_counter_bytes(c) + (size_t)ws_items(c) * ws_item_bytes(c);
}

// Fewest key tiles a work unit of node i walks: all of its slots' tiles,
// except under frame causality, where a pair of query tiles skips the own
// chunk's tiles past its last row's frame (the first pair skips the most).
int key_tiles_walked(const sva_cache* c, const sva::AttnNode& n, int nt_slot) {
  int own = nt_slot;
  if (n.frame_causal) {
    const int frame_tokens = c->g.grid_h * c->g.grid_w;
    const int last_row = std::min(2 * sva::kTile, c->L.T) - 1;
    const int frame_end = (last_row / frame_tokens + 1) * frame_tokens;
    own = std::min((frame_end + sva::kTile - 1) / sva::kTile, nt_slot);
  }
  return (n.n_kv - 1) * nt_slot + own;
}

// Splits per work unit: the smallest s in 1..kMaxSplit minimising the wave
// count per split, ceil(units * s / SMs) / s, subject to room for the split
// items (`cap` of them; none without scratch) and to at least 4 key tiles
// per split.
int choose_split(const sva_cache* c, long long units, int min_tiles, long long cap) {
  const long long sms = c->num_sms;
  double best = (double)((units + sms - 1) / sms);
  int best_s = 1;
  for (int s = 2; s <= sva::kMaxSplit; ++s) {
    const long long items = units * s;
    if (items > cap || min_tiles / s < 4) break;
    const double cost = (double)((items + sms - 1) / sms) / s;
    if (cost < best - 1e-9) {
      best = cost;
      best_s = s;
    }
  }
  return best_s;
}

// The split plan of a launch: units 0..n_full-1 unsplit, the rest split
// n_split ways, with at most `cap` split items.  When the units fill some
// whole waves of one CTA per SM, those waves run unsplit and only the partial
// last wave is split; that has the makespan of splitting every unit (when it
// is no longer) with fewer CTAs, fewer prologues and epilogues and fewer
// partials to merge, and needs room for fewer split items.
void plan_split(const sva_cache* c, long long units, int min_tiles, long long cap,
                long long* n_full, int* n_split) {
  const long long sms = c->num_sms;
  const int s_all = choose_split(c, units, min_tiles, cap);
  *n_full = 0;
  *n_split = s_all;
  if (units < sms) return;
  const long long full = units / sms * sms, rest = units - full;
  const int s_rest = choose_split(c, rest, min_tiles, cap);
  const double cost_all = (double)((units * s_all + sms - 1) / sms) / s_all;
  const double cost_mixed =
      (double)(full / sms) + (double)((rest * s_rest + sms - 1) / sms) / s_rest;
  if (cost_mixed <= cost_all + 1e-9) {
    *n_full = full;
    *n_split = s_rest;
  }
}

}  // namespace

extern "C" {

size_t sva_cache_bytes(const sva_geometry* g) {
  sva_status st;
  if (!geometry_valid(g, &st)) return 0;
  return layout_of(*g).total;
}

sva_status sva_cache_create(const sva_geometry* g, void* dev_buf, size_t bytes, sva_cache** out) {
  sva_status st;
  if (out == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "out is NULL");
  *out = nullptr;
  if (!geometry_valid(g, &st)) return st;
  if (dev_buf == nullptr || (reinterpret_cast<uintptr_t>(dev_buf) & 255u) != 0)
    return fail(SVA_ERR_INVALID_ARGUMENT, "dev_buf must be a non-NULL, 256-byte aligned device pointer");
  const Layout L = layout_of(*g);
  if (bytes < L.total)
    return fail(SVA_ERR_INVALID_ARGUMENT, "buffer of %zu bytes is smaller than the %zu needed",
                bytes, L.total);
  cudaPointerAttributes attr;
  cudaError_t e = cudaPointerGetAttributes(&attr, dev_buf);
  if (e != cudaSuccess || attr.type != cudaMemoryTypeDevice) {
    cudaGetLastError();
    return fail(SVA_ERR_INVALID_ARGUMENT, "dev_buf is not device memory");
  }
  sva_cache* c = new sva_cache();
  c->g = *g;
  c->L = L;
  c->base = static_cast<char*>(dev_buf);
  c->device = attr.device;
  int cur = -1;
  cudaGetDevice(&cur);
  if (cur != c->device) {
    delete c;
    return fail(SVA_ERR_INVALID_ARGUMENT, "dev_buf is on device %d, current device is %d",
                attr.device, cur);
  }
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
  if (c->num_sms <= 0) c->num_sms = 1;
  c->slots.assign(g->num_slots, SlotInfo());
  for (int32_t s = g->num_slots - 1; s >= 0; --s) c->free_slots.push_back(s);

  // Zero the pad rows [T, Tpad) of every (slot, K|V, head): the attention
  // kernel reads them inside each slot's last key tile and masks them.
  const size_t d = g->head_dim;
  if (L.Tpad > L.T) {
    e = cudaMemset2D(c->base + (size_t)L.T * d * 2, (size_t)L.Tpad * d * 2, 0,
                     (size_t)(L.Tpad - L.T) * d * 2, (size_t)g->num_slots * 2 * g->num_heads);
    if (e != cudaSuccess) {
      delete c;
      return cuda_fail(e, "cudaMemset2D(pad rows)");
    }
  }
  auto tt = rope_table(g->max_frames, g->rope_pairs[0], g->rope_theta);
  auto th = rope_table(g->grid_h, g->rope_pairs[1], g->rope_theta);
  auto tw = rope_table(g->grid_w, g->rope_pairs[2], g->rope_theta);
  auto transpose = [](const std::vector<float2>& t, int n_pos, int n_pair) {
    std::vector<float2> r(t.size());
    for (int i = 0; i < n_pos; ++i)
      for (int j = 0; j < n_pair; ++j) r[(size_t)j * n_pos + i] = t[(size_t)i * n_pair + j];
    return r;
  };
  auto tht = transpose(th, g->grid_h, g->rope_pairs[1]);
  auto twt = transpose(tw, g->grid_w, g->rope_pairs[2]);
  struct Up {
    size_t off;
    const std::vector<float2>* v;
  } ups[5] = {{L.tab_t, &tt}, {L.tab_h, &th}, {L.tab_w, &tw}, {L.tab_ht, &tht}, {L.tab_wt, &twt}};
  for (auto& u : ups) {
    if (u.v->empty()) continue;
    e = cudaMemcpy(c->base + u.off, u.v->data(), u.v->size() * sizeof(float2),
                   cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
      delete c;
      return cuda_fail(e, "cudaMemcpy(rope table)");
    }
  }
  e = cudaMemset(c->base + L.status, 0, 256);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    delete c;
    return cuda_fail(e, "cache initialisation");
  }
  st = encode_2d_kv(&c->tmap_kv, c->base, *g, L);
  if (st != SVA_OK) {
    delete c;
    return st;
  }
  *out = c;
  return ok();
}

sva_status sva_cache_bind(sva_cache* c, int32_t seq, int32_t chunk, int32_t level, int32_t* slot) {
  if (c == nullptr || slot == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  if (level < 0) return fail(SVA_ERR_INVALID_ARGUMENT, "level %d < 0", level);
  const StateKey k{seq, chunk, level};
  if (c->index.count(k))
    return fail(SVA_ERR_INVALID_ARGUMENT, "(seq %d, chunk %d, level %d) is already bound to slot %d",
                seq, chunk, level, c->index[k]);
  if (c->free_slots.empty())
    return fail(SVA_ERR_CAPACITY, "all %d slots are bound", c->g.num_slots);
  const int32_t s = c->free_slots.back();
  c->free_slots.pop_back();
  SlotInfo& si = c->slots[s];
  si.bound = true;
  si.resident = false;
  si.seq = seq;
  si.chunk = chunk;
  si.level = level;
  c->index[k] = s;
  *slot = s;
  return ok();
}

sva_status sva_cache_lookup(const sva_cache* c, int32_t seq, int32_t chunk, int32_t level,
                            int32_t* slot) {
  if (c == nullptr || slot == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  auto it = c->index.find(StateKey{seq, chunk, level});
  if (it == c->index.end())
    return fail(SVA_ERR_NOT_RESIDENT, "(seq %d, chunk %d, level %d) is not in the cache", seq,
                chunk, level);
  *slot = it->second;
  return ok();
}

sva_status sva_cache_release(sva_cache* c, int32_t seq, int32_t chunk, int32_t level) {
  if (c == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  auto it = c->index.find(StateKey{seq, chunk, level});
  if (it == c->index.end())
    return fail(SVA_ERR_NOT_RESIDENT, "(seq %d, chunk %d, level %d) is not in the cache", seq,
                chunk, level);
  const int32_t s = it->second;
  c->index.erase(it);
  c->slots[s] = SlotInfo();
  c->free_slots.push_back(s);
  return ok();
}

sva_status sva_select_context(int32_t policy, int32_t K, int32_t W, int32_t chunk, int32_t level,
                              int32_t cap, int32_t* chunks, int32_t* levels, int32_t* n) {
  if (chunks == nullptr || levels == nullptr || n == nullptr)
    return fail(SVA_ERR_INVALID_ARGUMENT, "NULL output");
  if (policy < SVA_POLICY_CLEAN || policy > SVA_POLICY_PROG)
    return fail(SVA_ERR_INVALID_ARGUMENT, "unknown policy %d", policy);
  if (K < 1 || level < 0 || level > K || W < 0)
    return fail(SVA_ERR_INVALID_ARGUMENT, "need K >= 1, 0 <= level <= K, W >= 0 (K=%d level=%d W=%d)",
                K, level, W);
  const long long window = (long long)chunk - 1;
  const int32_t count = (int32_t)std::max(0ll, std::min<long long>(W, window));
  *n = count;
  if (count > cap)
    return fail(SVA_ERR_CAPACITY, "selection has %d states, cap is %d", count, cap);
  for (int32_t r = 1; r <= count; ++r) {
    chunks[r - 1] = chunk - r;
    levels[r - 1] = phi(policy, level, r);
  }
  return ok();
}

sva_status sva_pipeline_round(int32_t K, int32_t B, int32_t round, int32_t cap, int32_t* chunks,
                              int32_t* levels, int32_t* count) {
  if (chunks == nullptr || levels == nullptr || count == nullptr)
    return fail(SVA_ERR_INVALID_ARGUMENT, "NULL output");
  if (K < 1 || B < 0) return fail(SVA_ERR_INVALID_ARGUMENT, "need K >= 1 and B >= 0");
  int32_t m = 0;
  for (int32_t j = K; j >= 1; --j) {
    const long long b = (long long)round - K + j;
    if (b >= 1 && b <= B) ++m;
  }
  *count = m;
  if (m > cap) return fail(SVA_ERR_CAPACITY, "round has %d states, cap is %d", m, cap);
  int32_t w = 0;
  for (int32_t j = K; j >= 1; --j) {
    const long long b = (long long)round - K + j;
    if (b >= 1 && b <= B) {
      chunks[w] = (int32_t)b;
      levels[w] = j;
      ++w;
    }
  }
  return ok();
}

sva_status sva_check_pipeline(int32_t K, int32_t level, int32_t chunk, int32_t n,
                              const int32_t* chunks, const int32_t* levels) {
  if (n < 0 || (n > 0 && (chunks == nullptr || levels == nullptr)))
    return fail(SVA_ERR_INVALID_ARGUMENT, "bad list");
  if (K < 1 || level < 0 || level > K)
    return fail(SVA_ERR_INVALID_ARGUMENT, "need K >= 1 and 0 <= level <= K");
  for (int32_t i = 0; i < n; ++i) {
    const long long r = (long long)chunk - chunks[i];
    if (r < 1)
      return fail(SVA_ERR_CAUSALITY, "entry %d: chunk %d is not before chunk %d", i, chunks[i],
                  chunk);
    if (levels[i] < 0 || levels[i] > K)
      return fail(SVA_ERR_INVALID_ARGUMENT, "entry %d: level %d outside 0..%d", i, levels[i], K);
    const long long reached = std::max(0ll, (long long)level - r);
    if (levels[i] < reached)
      return fail(SVA_ERR_UNAVAILABLE,
                  "entry %d: chunk %d has only reached level %lld when chunk %d is at level %d; "
                  "level %d is not available (Eq. 7)",
                  i, chunks[i], reached, chunk, level, levels[i]);
  }
  return ok();
}

}  // extern "C"

namespace {

// sva_rope_kv_write and sva_rope_kv_write_qknorm: gamma_k == NULL means no norm.
sva_status rope_write(sva_cache* c, const sva_node* nodes, int32_t n_nodes, const void* k_new,
                      const void* v_new, void* q_inout, const float* gamma_k,
                      const float* gamma_q, float eps, sva_stream s) {
  if (c == nullptr || nodes == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  if (n_nodes < 1) return fail(SVA_ERR_INVALID_ARGUMENT, "n_nodes %d < 1", n_nodes);
  if (n_nodes > SVA_MAX_NODES)
    return fail(SVA_ERR_CAPACITY, "n_nodes %d > SVA_MAX_NODES (%d)", n_nodes, SVA_MAX_NODES);
  if (k_new == nullptr || v_new == nullptr || !aligned16(k_new) || !aligned16(v_new) ||
      (q_inout != nullptr && !aligned16(q_inout)))
    return fail(SVA_ERR_INVALID_ARGUMENT, "k_new/v_new/q_inout must be non-NULL (q may be NULL) and 16-byte aligned");
  sva_status st = check_device(c);
  if (st != SVA_OK) return st;
  const sva_geometry& g = c->g;
  sva::RopeParams p{};
  for (int i = 0; i < n_nodes; ++i) {
    const sva_node& n = nodes[i];
    st = check_own(c, n, i, false);
    if (st != SVA_OK) return st;
    for (int k = 0; k < i; ++k)
      if (nodes[k].own_slot == n.own_slot)
        return fail(SVA_ERR_INVALID_ARGUMENT, "nodes %d and %d write the same slot %d", k, i,
                    n.own_slot);
    const long long t0 = (long long)g.frames * n.chunk;
    if (t0 < 0 || t0 + g.frames > g.max_frames)
      return fail(SVA_ERR_CAPACITY,
                  "node %d: chunk %d covers frames [%lld, %lld), outside the RoPE table [0, %d)", i,
                  n.chunk, t0, t0 + g.frames, g.max_frames);
    p.nodes[i].slot = n.own_slot;
    p.nodes[i].t_base = (int32_t)t0;
  }
  p.k_new = k_new;
  p.v_new = v_new;
  p.q = q_inout;
  p.cache = c->base;
  p.tab_t = reinterpret_cast<const float2*>(c->base + c->L.tab_t);
  p.tab_h = reinterpret_cast<const float2*>(c->base + c->L.tab_h);
  p.tab_w = reinterpret_cast<const float2*>(c->base + c->L.tab_w);
  p.T = c->L.T;
  p.H = g.num_heads;
  p.d = g.head_dim;
  p.Tpad = c->L.Tpad;
  p.Hp = g.grid_h;
  p.Wp = g.grid_w;
  p.P0 = g.rope_pairs[0];
  p.P1 = g.rope_pairs[1];
  p.P2 = g.rope_pairs[2];
  p.n_nodes = n_nodes;
  p.gamma_k = gamma_k;
  p.gamma_q = gamma_k != nullptr && q_inout != nullptr ? gamma_q : nullptr;
  p.norm_eps = eps;
  const long long tokens = (long long)n_nodes * p.T;  // one warp per token, 8 warps per block
  const long long blocks = (tokens + 7) / 8;
  p.grid_blocks = (int)std::min<long long>(blocks, (long long)c->num_sms * 16);
  cudaError_t e = sva::launch_rope_kv(p, c->num_sms, reinterpret_cast<cudaStream_t>(s));
  if (e != cudaSuccess) return cuda_fail(e, "rope_kv launch");
  for (int i = 0; i < n_nodes; ++i) c->slots[nodes[i].own_slot].resident = true;
  return ok();
}

}  // namespace

extern "C" {

sva_status sva_rope_kv_write(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                             const void* k_new, const void* v_new, void* q_inout, sva_stream s) {
  return rope_write(c, nodes, n_nodes, k_new, v_new, q_inout, nullptr, nullptr, 0.0f, s);
}

sva_status sva_rope_kv_write_qknorm(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                    const void* k_new, const void* v_new, void* q_inout,
                                    const float* gamma_k, const float* gamma_q, float eps,
                                    sva_stream s) {
  if (gamma_k == nullptr || !aligned16(gamma_k) ||
      (q_inout != nullptr && (gamma_q == nullptr || !aligned16(gamma_q))))
    return fail(SVA_ERR_INVALID_ARGUMENT,
                "gamma_k (and gamma_q when q_inout is given) must be non-NULL and 16-byte aligned");
  if (!std::isfinite(eps) || !(eps > 0.0f))
    return fail(SVA_ERR_INVALID_ARGUMENT, "eps must be finite and > 0");
  return rope_write(c, nodes, n_nodes, k_new, v_new, q_inout, gamma_k, gamma_q, eps, s);
}

}  // extern "C"

namespace {

// Where the key-range split partials of an attention launch go.
enum class Scratch {
  kWorkspace,  // the caller's workspace (sva_cache_set_workspace), if attached
  kStatic,     // the library's static device array (sva_attend_nodes_noalloc)
};

// sva_attend_nodes, _sparse, _masked and _noalloc: the checks, the launch
// parameters, the split plan and the launch.  tile_mask, own_mask and
// hist_mask NULL is
// the dense mask.  Every check runs before anything is enqueued.
sva_status attend(sva_cache* c, const sva_node* nodes, int32_t n_nodes, const void* q, void* out,
                  float* lse, float scale, const uint32_t* tile_mask, int32_t mask_words,
                  const uint32_t* own_mask, int32_t own_words, const uint32_t* hist_mask,
                  int32_t hist_states, int32_t hist_words, sva_stream s, Scratch scratch) {
  if (c == nullptr || nodes == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  if (n_nodes < 1) return fail(SVA_ERR_INVALID_ARGUMENT, "n_nodes %d < 1", n_nodes);
  if (n_nodes > SVA_MAX_NODES)
    return fail(SVA_ERR_CAPACITY, "n_nodes %d > SVA_MAX_NODES (%d)", n_nodes, SVA_MAX_NODES);
  if (q == nullptr || out == nullptr || !aligned16(q) || !aligned16(out) ||
      (lse != nullptr && (reinterpret_cast<uintptr_t>(lse) & 3u) != 0))
    return fail(SVA_ERR_INVALID_ARGUMENT, "q/out must be non-NULL and 16-byte aligned, lse 4-byte aligned");
  if (!std::isfinite(scale) || !(scale > 0.0f))
    return fail(SVA_ERR_INVALID_ARGUMENT, "scale must be finite and > 0");
  sva_status st = check_device(c);
  if (st != SVA_OK) return st;
  const sva_geometry& g = c->g;

  static thread_local sva::AttnParams p;  // ~5 KB: kept off the stack
  std::memset(&p, 0, sizeof(p));
  for (int i = 0; i < n_nodes; ++i) {
    const sva_node& n = nodes[i];
    st = check_own(c, n, i, true);
    if (st != SVA_OK) return st;
    if (n.n_ctx < 0 || n.n_ctx > SVA_MAX_CTX)
      return fail(SVA_ERR_CAPACITY, "node %d: n_ctx %d outside 0..%d", i, n.n_ctx, SVA_MAX_CTX);
    if (n.within != SVA_WITHIN_BIDIRECTIONAL && n.within != SVA_WITHIN_FRAME_CAUSAL)
      return fail(SVA_ERR_INVALID_ARGUMENT, "node %d: unknown within-chunk mode %d", i, n.within);
    sva::AttnNode& a = p.nodes[i];
    a.q_index = i;
    a.frame_causal = n.within == SVA_WITHIN_FRAME_CAUSAL ? 1 : 0;
    a.slot[0] = n.own_slot;
    a.src[0] = 0;
    int nkv = 1;
    for (int k = 0; k < n.n_ctx; ++k) {
      const int32_t cs = n.ctx_slot[k];
      if (cs < 0 || cs >= g.num_slots)
        return fail(SVA_ERR_INVALID_ARGUMENT, "node %d ctx %d: slot %d out of range", i, k, cs);
      const SlotInfo& si = c->slots[cs];
      if (!si.bound || !si.resident)
        return fail(SVA_ERR_NOT_RESIDENT, "node %d ctx %d: slot %d is %s", i, k, cs,
                    si.bound ? "bound but not written" : "not bound");
      if (si.seq != n.seq || si.chunk >= n.chunk)
        return fail(SVA_ERR_CAUSALITY,
                    "node %d (seq %d, chunk %d) ctx %d: slot %d holds (seq %d, chunk %d), not a "
                    "past chunk of the same sequence",
                    i, n.seq, n.chunk, k, cs, si.seq, si.chunk);
      if (cs == n.own_slot)
        return fail(SVA_ERR_INVALID_ARGUMENT, "node %d ctx %d repeats the own slot", i, k);
      for (int k2 = 0; k2 < k; ++k2)
        if (n.ctx_slot[k2] == cs)
          return fail(SVA_ERR_INVALID_ARGUMENT, "node %d: slot %d listed twice", i, cs);
      if (n.ctx_visible[k]) {
        a.src[nkv] = (uint8_t)(1 + k);
        a.slot[nkv++] = cs;
      }
    }
    a.n_kv = nkv;
  }
  p.n_qt = (c->L.T + sva::kTile - 1) / sva::kTile;
  p.nt_slot = c->L.Tpad / sva::kTile;
  if (tile_mask != nullptr) {
    if ((reinterpret_cast<uintptr_t>(tile_mask) & 3u) != 0)
      return fail(SVA_ERR_INVALID_ARGUMENT, "tile_mask must be 4-byte aligned");
    for (int i = 0; i < n_nodes; ++i) {
      const long long bits = (long long)(1 + nodes[i].n_ctx) * p.nt_slot;
      if (bits > 32LL * sva::kMaskWords)
        return fail(SVA_ERR_CAPACITY, "node %d: %lld key tiles exceed the %d a tile mask covers",
                    i, bits, 32 * sva::kMaskWords);
      if (mask_words < (bits + 31) / 32)
        return fail(SVA_ERR_INVALID_ARGUMENT,
                    "node %d: words_per_row %d < %lld needed for %lld key tiles", i, mask_words,
                    (bits + 31) / 32, bits);
    }
    p.tile_mask = tile_mask;
    p.mask_words = mask_words;
  }
  if (own_mask != nullptr) {
    if ((reinterpret_cast<uintptr_t>(own_mask) & 3u) != 0)
      return fail(SVA_ERR_INVALID_ARGUMENT, "own_mask must be 4-byte aligned");
    if (own_words < (c->L.T + 31) / 32)
      return fail(SVA_ERR_INVALID_ARGUMENT, "own_words %d < %d needed for %d tokens", own_words,
                  (c->L.T + 31) / 32, c->L.T);
    p.own_mask = own_mask;
    p.own_words = own_words;
  }
  if (hist_mask != nullptr) {
    if ((reinterpret_cast<uintptr_t>(hist_mask) & 3u) != 0)
      return fail(SVA_ERR_INVALID_ARGUMENT, "hist_mask must be 4-byte aligned");
    if (hist_words < (c->L.T + 31) / 32)
      return fail(SVA_ERR_INVALID_ARGUMENT, "hist_words %d < %d needed for %d tokens", hist_words,
                  (c->L.T + 31) / 32, c->L.T);
    if (hist_states < 1)
      return fail(SVA_ERR_INVALID_ARGUMENT, "hist_states %d < 1", hist_states);
    for (int i = 0; i < n_nodes; ++i)
      if (nodes[i].n_ctx > hist_states)
        return fail(SVA_ERR_INVALID_ARGUMENT, "node %d has %d context states, hist_states is %d",
                    i, nodes[i].n_ctx, hist_states);
    p.hist_mask = hist_mask;
    p.hist_states = hist_states;
    p.hist_words = hist_words;
  }
  p.masked = (tile_mask != nullptr || own_mask != nullptr || hist_mask != nullptr) ? 1 : 0;
  if (p.masked)  // the masked kernel keeps a bitmap of the node's key tiles
    for (int i = 0; i < n_nodes; ++i)
      if ((long long)p.nodes[i].n_kv * p.nt_slot > 32LL * sva::kMaskWords)
        return fail(SVA_ERR_CAPACITY, "node %d: %lld key tiles exceed the %d a masked launch covers",
                    i, (long long)p.nodes[i].n_kv * p.nt_slot, 32 * sva::kMaskWords);

  // The split plan.  The static scratch takes the plan a full caller
  // workspace would get, so both entry points compute the same result, and
  // refuses a plan whose partials do not fit the array.
  int min_tiles = 1 << 30;
  for (int i = 0; i < n_nodes; ++i)
    min_tiles = std::min(min_tiles, key_tiles_walked(c, p.nodes[i], p.nt_slot));
  p.n_qp = (p.n_qt + 1) / 2;
  const long long units = (long long)g.num_heads * n_nodes * p.n_qp;
  const long long cap = (scratch == Scratch::kStatic || c->ws != nullptr) ? ws_items(c) : 0;
  long long n_full = 0;
  int n_split = 1;
  plan_split(c, units, min_tiles, cap, &n_full, &n_split);
  char* split_base = c->ws;
  size_t counter_bytes = ws_counter_bytes(c);
  if (scratch == Scratch::kStatic) {
    split_base = nullptr;
    if (n_split > 1) {
      const long long split_units = units - n_full;
      counter_bytes = round_up((size_t)split_units * 4, 256);
      const size_t need = counter_bytes + (size_t)split_units * n_split * ws_item_bytes(c);
      if (need > sva::kStaticScratchBytes)
        return fail(SVA_ERR_CAPACITY,
                    "this launch splits %lld work units %d ways and needs %zu bytes of scratch; the "
                    "library's static scratch holds %zu bytes (use sva_attend_nodes with a "
                    "workspace for launches this large)",
                    split_units, n_split, need, sva::kStaticScratchBytes);
      void* addr = nullptr;
      cudaError_t e = sva::static_split_scratch(c->device, &addr);
      if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(split scratch)");
      split_base = static_cast<char*>(addr);
    }
  }

  if (c->q_cached != q || c->q_cached_n != n_nodes) {
    st = encode_4d_q(&c->tmap_q, q, g, c->L.T, n_nodes);
    if (st != SVA_OK) {
      c->q_cached = nullptr;
      return st;
    }
    c->q_cached = q;
    c->q_cached_n = n_nodes;
  }
  p.tmap_q = c->tmap_q;
  p.tmap_kv = c->tmap_kv;
  p.out = out;
  p.lse = lse;
  p.status = reinterpret_cast<int*>(c->base + c->L.status);
  p.scale_log2 = scale * 1.4426950408889634f;
  p.T = c->L.T;
  p.Tpad = c->L.Tpad;
  p.H = g.num_heads;
  p.n_nodes = n_nodes;
  p.valid_last = c->L.T - (p.nt_slot - 1) * sva::kTile;
  p.frame_tokens = g.grid_h * g.grid_w;
  p.fault_mode = scratch == Scratch::kStatic ? 0 : c->fault_mode;
  p.timeout_ns = c->timeout_ns;
  if (scratch != Scratch::kStatic) c->fault_mode = 0;
  p.n_full = (int32_t)n_full;
  p.n_split = n_split;
  if (n_split > 1) {
    p.ws_count = reinterpret_cast<int*>(split_base);
    p.ws = reinterpret_cast<float*>(split_base + counter_bytes);
    if (scratch == Scratch::kStatic) {
      // the arrival counters must start at zero; the array keeps whatever the
      // previous call left in it
      cudaError_t e = cudaMemsetAsync(split_base, 0, counter_bytes, reinterpret_cast<cudaStream_t>(s));
      if (e != cudaSuccess) return cuda_fail(e, "clearing the split counters");
    }
  }
  const long long grid = n_full + (units - n_full) * n_split;
  cudaError_t e = sva::launch_attend(p, g.head_dim, (int)grid, reinterpret_cast<cudaStream_t>(s));
  if (e != cudaSuccess) return cuda_fail(e, "attend launch");
  return ok();
}

}  // namespace

extern "C" {

sva_status sva_attend_nodes(sva_cache* c, const sva_node* nodes, int32_t n_nodes, const void* q,
                            void* out, float* lse, float scale, sva_stream s) {
  return attend(c, nodes, n_nodes, q, out, lse, scale, nullptr, 0, nullptr, 0, nullptr, 0, 0, s,
                Scratch::kWorkspace);
}

}  // extern "C"

namespace {

// sva_qkv_project, and with `nodes` non-NULL sva_qkv_project_rope (k, v are
// then unused: K' and V go to the nodes' own slots).
sva_status project(sva_cache* c, const sva_node* nodes, int32_t n_nodes, const void* x,
                   int32_t rows, int32_t in_features, const void* weight, const float* bias,
                   void* q, void* k, void* v, sva_stream s) {
  if (c == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL cache");
  if (rows < 1 || in_features < 8 || in_features % 8 != 0)
    return fail(SVA_ERR_INVALID_ARGUMENT,
                "rows %d must be >= 1 and in_features %d a positive multiple of 8", rows,
                in_features);
  const bool rope = nodes != nullptr;
  if (x == nullptr || weight == nullptr || q == nullptr || !aligned16(x) || !aligned16(weight) ||
      !aligned16(q) || (!rope && (k == nullptr || v == nullptr || !aligned16(k) || !aligned16(v))) ||
      (bias != nullptr && !aligned16(bias)))
    return fail(SVA_ERR_INVALID_ARGUMENT,
                rope ? "x, weight, q_out (and bias if given) must be non-NULL and 16-byte aligned"
                     : "x, weight, q, k, v (and bias if given) must be non-NULL and 16-byte aligned");
  sva_status st = check_device(c);
  if (st != SVA_OK) return st;
  {
    // every operand must be memory of the cache's device: the tensor maps and
    // the epilogue's stores address it directly
    const void* ptrs[6] = {x, weight, bias, q, k, v};
    const char* names[6] = {"x", "weight", "bias", rope ? "q_out" : "q", "k", "v"};
    for (int i = 0; i < 6; ++i)
      if (ptrs[i] != nullptr && !on_device(ptrs[i], c->device))
        return fail(SVA_ERR_INVALID_ARGUMENT, "%s is not device memory of the cache's device %d",
                    names[i], c->device);
  }
  const sva_geometry& g = c->g;
  const int N = g.num_heads * g.head_dim;
  if (N % 128 != 0)
    return fail(SVA_ERR_UNSUPPORTED, "num_heads * head_dim = %d is not a multiple of 128", N);
  const int bn = (N % 256 == 0) ? 256 : 128;
  auto fn = encode_fn();
  if (!fn) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  static thread_local sva::ProjParams p;
  std::memset(&p, 0, sizeof(p));
  cuuint32_t es[2] = {1, 1};
  {
    cuuint64_t dims[2] = {(cuuint64_t)in_features, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)in_features * 2};
    cuuint32_t box[2] = {64, 128};
    CUresult r = fn(&p.tmap_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims,
                    strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(x) failed: %d", (int)r);
  }
  for (int half = 0; half < 2; ++half) {
    // one CTA's half of the W rows of a whole item (BN / 2 rows) and of a
    // half-width item (BN / 4)
    cuuint64_t dims[2] = {(cuuint64_t)in_features, (cuuint64_t)3 * N};
    cuuint64_t strides[1] = {(cuuint64_t)in_features * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)(half ? bn / 4 : bn / 2)};
    CUresult r = fn(half ? &p.tmap_wh : &p.tmap_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                    const_cast<void*>(weight), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
      return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(weight) failed: %d", (int)r);
  }
  {
    // the epilogue's tile stores: 32 rows x 32 columns (64 bytes), staged in
    // shared memory in the 64-byte swizzle; rows past `rows` are not written
    void* outs[3] = {q, k, v};
    for (int i = 0; i < (rope ? 1 : 3); ++i) {
      cuuint64_t dims[2] = {(cuuint64_t)N, (cuuint64_t)rows};
      cuuint64_t strides[1] = {(cuuint64_t)N * 2};
      cuuint32_t box[2] = {32, 32};
      CUresult r = fn(&p.tmap_out[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, outs[i], dims, strides,
                      box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                      CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS)
        return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(output %d) failed: %d", i, (int)r);
    }
    if (rope) {
      // K' and V into the slot pool: rows of one (slot, K|V, head) are the
      // tokens [0, T) of that slot (the padding rows up to Tpad untouched)
      const sva_geometry& g0 = c->g;
      cuuint64_t dims[3] = {(cuuint64_t)g0.head_dim, (cuuint64_t)c->L.T,
                            (cuuint64_t)g0.num_slots * 2 * g0.num_heads};
      cuuint64_t strides[2] = {(cuuint64_t)g0.head_dim * 2, (cuuint64_t)c->L.Tpad * g0.head_dim * 2};
      cuuint32_t box[3] = {32, 32, 1};
      cuuint32_t es3[3] = {1, 1, 1};
      CUresult r = fn(&p.tmap_out[1], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, c->base, dims, strides,
                      box, es3, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                      CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS)
        return fail(SVA_ERR_CUDA, "cuTensorMapEncodeTiled(slot pool) failed: %d", (int)r);
    }
  }
  if (rope) {
    // the same node checks as sva_rope_kv_write
    for (int i = 0; i < n_nodes; ++i) {
      const sva_node& n = nodes[i];
      st = check_own(c, n, i, false);
      if (st != SVA_OK) return st;
      for (int j = 0; j < i; ++j)
        if (nodes[j].own_slot == n.own_slot)
          return fail(SVA_ERR_INVALID_ARGUMENT, "nodes %d and %d write the same slot %d", j, i,
                      n.own_slot);
      const long long t0 = (long long)g.frames * n.chunk;
      if (t0 < 0 || t0 + g.frames > g.max_frames)
        return fail(SVA_ERR_CAPACITY,
                    "node %d: chunk %d covers frames [%lld, %lld), outside the RoPE table [0, %d)",
                    i, n.chunk, t0, t0 + g.frames, g.max_frames);
      p.rope.nodes[i].slot = n.own_slot;
      p.rope.nodes[i].t_base = (int32_t)t0;
    }
    p.rope_on = 1;
    p.rope.cache = c->base;
    p.rope.tab_t = reinterpret_cast<const float2*>(c->base + c->L.tab_t);
    p.rope.tab_h = reinterpret_cast<const float2*>(c->base + c->L.tab_ht);  // pair-major
    p.rope.tab_w = reinterpret_cast<const float2*>(c->base + c->L.tab_wt);  // pair-major
    p.rope.T = c->L.T;
    p.rope.H = g.num_heads;
    p.rope.d = g.head_dim;
    p.rope.Tpad = c->L.Tpad;
    p.rope.Hp = g.grid_h;
    p.rope.Wp = g.grid_w;
    p.rope.P0 = g.rope_pairs[0];
    p.rope.P1 = g.rope_pairs[1];
    p.rope.P2 = g.rope_pairs[2];
    p.rope.n_nodes = n_nodes;
  }
  p.bias = bias;
  p.out[0] = q;
  p.out[1] = k;
  p.out[2] = v;
  p.status = reinterpret_cast<int*>(c->base + c->L.status);
  p.rows = rows;
  p.C = in_features;
  p.N = N;
  p.n_mtiles = (rows + 255) / 256;
  p.n_ntiles = 3 * N / bn;
  p.n_kblocks = (in_features + 63) / 64;
  p.timeout_ns = c->timeout_ns;
  // One pair of CTAs per two SMs walks the items.  The tiles of a partial
  // last round are split into two half-width items when the halves fit one
  // round (and, for the fused RoPE epilogue, still cover whole heads), so
  // that the last round takes half as long.
  int max_pairs = 0;
  cudaError_t e = sva::qkv_project_max_pairs(bn, &max_pairs);
  if (e != cudaSuccess) return cuda_fail(e, "qkv_project occupancy");
  const long long pairs = std::max(1, std::min(max_pairs, c->num_sms / 2));
  const long long tiles = (long long)p.n_mtiles * p.n_ntiles;
  if (tiles > INT32_MAX / 2) return fail(SVA_ERR_CAPACITY, "%lld output tiles", tiles);
  const long long rest = tiles % pairs;
  const bool split_tail = rest > 0 && 2 * rest <= pairs && (!rope || (bn / 2) % g.head_dim == 0);
  p.n_whole = (int32_t)(split_tail ? tiles - rest : tiles);
  p.n_items = (int32_t)(split_tail ? tiles + rest : tiles);
  const int grid = 2 * (int)std::min<long long>(p.n_items, pairs);
  e = sva::launch_qkv_project(p, bn, grid, reinterpret_cast<cudaStream_t>(s));
  if (e != cudaSuccess) return cuda_fail(e, "qkv_project launch");
  if (rope)
    for (int i = 0; i < n_nodes; ++i) c->slots[nodes[i].own_slot].resident = true;
  return ok();
}

}  // namespace

extern "C" {

sva_status sva_qkv_project(sva_cache* c, const void* x, int32_t rows, int32_t in_features,
                           const void* weight, const float* bias, void* q, void* k, void* v,
                           sva_stream s) {
  return project(c, nullptr, 0, x, rows, in_features, weight, bias, q, k, v, s);
}

sva_status sva_qkv_project_rope(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                const void* x, int32_t in_features, const void* weight,
                                const float* bias, void* q_out, sva_stream s) {
  if (c == nullptr || nodes == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  if (n_nodes < 1) return fail(SVA_ERR_INVALID_ARGUMENT, "n_nodes %d < 1", n_nodes);
  if (n_nodes > SVA_MAX_NODES)
    return fail(SVA_ERR_CAPACITY, "n_nodes %d > SVA_MAX_NODES (%d)", n_nodes, SVA_MAX_NODES);
  const long long rows = (long long)n_nodes * c->L.T;
  if (rows > INT32_MAX) return fail(SVA_ERR_CAPACITY, "n_nodes * T = %lld rows", rows);
  return project(c, nodes, n_nodes, x, (int32_t)rows, in_features, weight, bias, q_out, nullptr,
                 nullptr, s);
}

sva_status sva_attend_nodes_sparse(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                   const void* q, void* out, float* lse, float scale,
                                   const uint32_t* tile_mask, int32_t words_per_row,
                                   sva_stream s) {
  if (tile_mask == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "tile_mask is NULL");
  return attend(c, nodes, n_nodes, q, out, lse, scale, tile_mask, words_per_row, nullptr, 0,
                nullptr, 0, 0, s, Scratch::kWorkspace);
}

sva_status sva_attend_nodes_masked(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                   const void* q, void* out, float* lse, float scale,
                                   const sva_attn_mask* mask, sva_stream s) {
  if (mask == nullptr)
    return attend(c, nodes, n_nodes, q, out, lse, scale, nullptr, 0, nullptr, 0, nullptr, 0, 0, s,
                  Scratch::kWorkspace);
  return attend(c, nodes, n_nodes, q, out, lse, scale, mask->tile_mask, mask->tile_words,
                mask->own_mask, mask->own_words, mask->hist_mask, mask->hist_states,
                mask->hist_words, s, Scratch::kWorkspace);
}

// Attention with the split scratch taken from the library's own device
// array instead of a caller-attached workspace (see include/sva.h): the same
// checks, the same split plan and the same kernel as sva_attend_nodes with a
// workspace attached.
sva_status sva_attend_nodes_noalloc(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                    const void* q, void* out, float* lse, float scale,
                                    sva_stream s) {
  return attend(c, nodes, n_nodes, q, out, lse, scale, nullptr, 0, nullptr, 0, nullptr, 0, 0, s,
                Scratch::kStatic);
}

sva_status sva_poll_device_status(sva_cache* c, sva_stream s) {
  if (c == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  sva_status st = check_device(c);
  if (st != SVA_OK) return st;
  cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(s));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int word = 0;
  e = cudaMemcpy(&word, c->base + c->L.status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the status word");
  if (word != 0) {
    e = cudaMemset(c->base + c->L.status, 0, sizeof(int));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "clearing the status word");
    if (c->ws != nullptr) {
      // a timed-out split unit may have left its arrival counter non-zero
      e = cudaMemset(c->ws, 0, ws_counter_bytes(c));
      if (e == cudaSuccess) e = cudaDeviceSynchronize();
      if (e != cudaSuccess) return cuda_fail(e, "clearing the split counters");
    }
    if (word == SVA_ERR_DEVICE_TIMEOUT)
      return fail(SVA_ERR_DEVICE_TIMEOUT, "a kernel gave up a bounded wait; its outputs are invalid");
    return fail(SVA_ERR_CUDA, "device status word %d", word);
  }
  return ok();
}

size_t sva_attend_workspace_bytes(const sva_cache* c) {
  if (c == nullptr) return 0;
  return ws_total_bytes(c);
}

sva_status sva_cache_set_workspace(sva_cache* c, void* dev_buf, size_t bytes) {
  if (c == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL cache");
  if (dev_buf == nullptr) {
    c->ws = nullptr;
    return ok();
  }
  if ((reinterpret_cast<uintptr_t>(dev_buf) & 255u) != 0)
    return fail(SVA_ERR_INVALID_ARGUMENT, "workspace must be 256-byte aligned");
  if (bytes < ws_total_bytes(c))
    return fail(SVA_ERR_INVALID_ARGUMENT, "workspace of %zu bytes is smaller than the %zu needed",
                bytes, ws_total_bytes(c));
  cudaPointerAttributes attr;
  cudaError_t e = cudaPointerGetAttributes(&attr, dev_buf);
  if (e != cudaSuccess || attr.type != cudaMemoryTypeDevice || attr.device != c->device) {
    cudaGetLastError();
    return fail(SVA_ERR_INVALID_ARGUMENT, "workspace is not device memory of the cache's device");
  }
  e = cudaMemset(dev_buf, 0, ws_counter_bytes(c));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "zeroing the workspace counters");
  c->ws = static_cast<char*>(dev_buf);
  return ok();
}

sva_status sva_debug_inject(sva_cache* c, int32_t mode, double timeout_s) {
  if (c == nullptr) return fail(SVA_ERR_INVALID_ARGUMENT, "NULL argument");
  if (mode < 0 || mode > 1) return fail(SVA_ERR_INVALID_ARGUMENT, "unknown fault mode %d", mode);
  if (!(timeout_s >= 1e-3 && timeout_s <= 60.0))
    return fail(SVA_ERR_INVALID_ARGUMENT, "timeout must be in [1 ms, 60 s]");
  c->fault_mode = mode;
  c->timeout_ns = (uint64_t)(timeout_s * 1e9);
  return ok();
}

sva_status sva_destroy(sva_cache* c) {
  delete c;
  return ok();
}

const char* sva_last_error(void) { return g_err.c_str(); }

}  // extern "C"
