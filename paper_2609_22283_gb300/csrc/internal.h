// Parameter blocks passed from the host runtime (sva_api.cpp) to the
// attention and RoPE kernels (the projection's are in proj.h), by value as
// __grid_constant__ kernel parameters, so a launch needs no host-to-device
// copy of its node list.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "sva.h"

namespace sva {

constexpr int kTile = 128;  // query rows per Q tile and key rows per K/V tile
constexpr int kMaxSplit = 4;  // key-range splits of one work unit
constexpr uint64_t kDefaultWaitTimeoutNs = 1000000000ull;  // bounded device waits: 1 s
constexpr int kMaskWords = 128;  // block-sparse launches: at most 32 * 128 key tiles per node

// Device status word values (a subset of sva_status).
constexpr int kStatusOk = 0;
constexpr int kStatusTimeout = SVA_ERR_DEVICE_TIMEOUT;

// One node of an attention launch: its index in q/out/lse and the cache
// slots it attends, own slot first, then the visible context slots.
struct AttnNode {
  int32_t q_index;
  int32_t n_kv;
  int32_t frame_causal;  // own-chunk keys of later latent frames masked
  int32_t slot[1 + SVA_MAX_CTX];
  // key state (0 = own, 1 + j = the caller's ctx_slot[j]) of each entry of
  // `slot`: the row index of its tiles in a block-sparse tile mask
  uint8_t src[1 + SVA_MAX_CTX];
};

struct alignas(128) AttnParams {
  CUtensorMap tmap_q;   // q as 4D (d, H, T, n_nodes), box (64, 1, 128, 1), 128B swizzle
  CUtensorMap tmap_kv;  // slot pool as 2D (d, num_slots*2*H*Tpad), box (64, 128), 128B swizzle
  void* out;            // bf16 [n_nodes][T][H][d]
  float* lse;           // fp32 [n_nodes][H][T] or null
  int* status;          // device status word
  float scale_log2;     // logit scale * log2(e)
  int32_t T;            // tokens per chunk
  int32_t Tpad;         // T rounded up to kTile: rows per (slot, K|V, head)
  int32_t H;
  int32_t n_qt;         // query tiles per node = ceil(T / kTile)
  int32_t n_qp;         // work units per (node, head): query-tile pairs = ceil(n_qt / 2)
  int32_t n_nodes;
  int32_t nt_slot;      // key tiles per slot = Tpad / kTile
  int32_t valid_last;   // valid key rows in the last tile of a slot
  int32_t frame_tokens; // tokens per latent frame (Hp * Wp)
  int32_t fault_mode;   // 0 in production; see sva_api.cpp
  int32_t n_split;      // key-range splits per split work unit (1 = no split)
  int32_t n_full;       // units 0..n_full-1 run unsplit (one CTA each); the
                        // rest are split n_split ways (CTAs after them)
  float* ws;            // split partials [unit][split][(d + 2) * 256] fp32, or null
  int* ws_count;        // per-unit arrival counters, zero between launches, or null
  uint64_t timeout_ns;
  const uint32_t* tile_mask;  // block-sparse visibility [n_nodes][n_qt][mask_words], or null
  int32_t mask_words;
  const uint32_t* own_mask;   // token visibility in the own chunk [n_nodes][T][own_words], or null
  int32_t own_words;
  // token visibility of the context states [n_nodes][T][hist_states][hist_words]
  // (state j = the caller's ctx_slot[j]), or null
  const uint32_t* hist_mask;
  int32_t hist_states;
  int32_t hist_words;
  int32_t masked;             // a tile or token mask given: a masked kernel instance
  AttnNode nodes[SVA_MAX_NODES];
};

struct RopeNode {
  int32_t slot;    // own slot the node's K', V go to
  int32_t t_base;  // absolute latent-frame position of the chunk's first frame (F * chunk)
};

struct RopeParams {
  const void* k_new;  // bf16 [n_nodes][T][H][d]
  const void* v_new;  // bf16 [n_nodes][T][H][d]
  void* q;            // bf16 [n_nodes][T][H][d], rotated in place; may be null
  void* cache;        // slot pool base, bf16 [num_slots][2][H][Tpad][d]
  const float2* tab_t;  // (cos, sin) [max_frames][P0]
  const float2* tab_h;  // (cos, sin) [Hp][P1]
  const float2* tab_w;  // (cos, sin) [Wp][P2]
  int32_t T, H, d, Tpad, Hp, Wp, P0, P1, P2;
  int32_t n_nodes;
  int32_t grid_blocks;
  // Optional RMSNorm of each token's K (and Q) vector of H*d elements before
  // the rotation: x * gamma / sqrt(mean(x^2) + eps).  Null gammas: no norm.
  const float* gamma_k;
  const float* gamma_q;
  float norm_eps;
  RopeNode nodes[SVA_MAX_NODES];
};

// Size of the library-owned split scratch used by sva_attend_nodes_noalloc.
constexpr size_t kStaticScratchBytes = (size_t)32 << 20;

// Device address of that scratch on `device` (the current device); the
// first call on a device looks it up.  Defined in attend_noalloc.cu.
cudaError_t static_split_scratch(int device, void** ptr);

// Launchers (defined in the .cu files).  They return the launch error.
cudaError_t launch_attend(const AttnParams& p, int head_dim, int grid, cudaStream_t s);
cudaError_t launch_rope_kv(const RopeParams& p, int num_sms, cudaStream_t s);

}  // namespace sva
