// Policy-indexed chunk-causal attention (Eq. 4, Section 3.2) for a batch of
// denoising nodes on sm_103a.
//
// For node n, head h and query u of the node's own chunk:
//   O[u] = sum_v softmax_v(scale * q_u . k_v + M(u, v)) v_v,
// where M is 0 on every key of the node's own slot (bidirectional inside the
// chunk) and of its visible context slots, and -inf everywhere else.  Keys
// outside those slots are never read, so the mask costs nothing except on the
// zero pad rows of each slot's last tile, which get -inf explicitly.
//
// One CTA computes one work unit: (node, head, a pair of 128-query tiles Q0,
// Q1) and streams every key tile of every slot the node reads; each K/V tile
// in shared memory serves both query tiles.
//   warp 0     TMA producer: Q0/Q1 once, then K and V tiles of the slot list
//              into rings of shared-memory stages (128B swizzle);
//   warps 1, 3 MMA issuers, warp 1 for query tile 0 and warp 3 for query
//              tile 1 (each whole warp runs its loop, one elected lane
//              issues); warp 1 also owns TMEM;
//   warps 4-11 softmax, all eight warps on one query tile at a time (Q0 then
//              Q1 of every key tile): two threads per query row, 64 keys
//              each; S from TMEM, fp32 online softmax in the log2 domain with
//              a lazy rescale of O, P written back over S as bf16; then the
//              epilogue (O / l to bf16 global, optional LSE).
// TMEM columns: S0 [0,128), S1 [128,256), O0 [256, 256+d), O1 [384, 384+d).
// Each issuer's order per key tile i is PV_b,i then S_b,i+1, so the softmax of
// either query tile has the other tile's PV and S (two 128x128x128 MMAs) to
// hide behind.  A tcgen05.mma costs its issuing warp nearly as long as the
// tensor pipe takes to run it (about 60 of 64 cycles while the softmax warps
// share the SM), so one issuer for both tiles left the pipe idle whenever it
// waited on a barrier; two issuers on different sub-partitions each have half
// the MMAs to issue.  A commit that completes S_b of tile i also implies PV_b
// of tile i-1 is complete (one issuer per tile, MMAs of a thread execute in
// issue order), so the rescale of O_b needs no extra barrier.
// A unit may be split into n_split contiguous key ranges (when there are too
// few units to fill the GPU's waves): each split CTA writes its normalised
// partial O with its row max and sum to the workspace and bumps the unit's
// arrival counter; the last to arrive merges the partials (the usual
// log-sum-exp combination) and writes the output, then resets the counter.
// All waits are bounded (1 s by default): on expiry the CTA records
// SVA_ERR_DEVICE_TIMEOUT in the status word, drains its own copies and MMAs,
// frees TMEM and exits.
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "ptx.cuh"

namespace sva {
namespace {

using namespace ptx;

template <int D>
struct AttnCfg {
  static_assert(D == 64 || D == 128, "head_dim");
  static constexpr int kBoxBytes = kTile * 64 * 2;   // one 128-row x 64-column bf16 box
  static constexpr int kBoxes = D / 64;
  static constexpr int kTileBytes = kBoxBytes * kBoxes;
  static constexpr int kKStages = (D == 128) ? 3 : 4;
  static constexpr int kVStages = (D == 128) ? 2 : 4;
  static constexpr int kOffQ0 = 0;
  static constexpr int kOffQ1 = kTileBytes;
  static constexpr int kOffK = 2 * kTileBytes;
  static constexpr int kOffV = kOffK + kKStages * kTileBytes;
  static constexpr int kSmemBytes = kOffV + kVStages * kTileBytes + 1024;  // + alignment slack
  static constexpr uint32_t kTmemCols = 512;
};

// TMEM columns of the S buffers and O accumulators of query tiles 0 and 1.
__device__ __forceinline__ uint32_t col_s(int b) { return b ? 128u : 0u; }
__device__ __forceinline__ uint32_t col_o(int b) { return b ? 384u : 256u; }

// 12 warps: warpgroup 0 = TMA producer (warp 0), MMA issuers (warps 1 and
// 3), warp 2 (the block-sparse mask gather in the prologue, then idle);
// warpgroups 1 and 2 = softmax.  The launch gives every thread
// kLaunchRegs registers; warpgroup 0 then gives registers back
// (setmaxnreg.dec to kRegsLow) and the softmax warpgroups take them
// (setmaxnreg.inc to kRegsHigh).  The split must fit the launch's pool:
// 4*32*kRegsLow + 8*32*kRegsHigh <= 384*kLaunchRegs, checked at launch.
constexpr int kThreads = 384;
constexpr int kLaunchRegs = 168;
constexpr int kRegsLow = 88;
constexpr int kRegsHigh = 208;
static_assert(4 * 32 * kRegsLow + 8 * 32 * kRegsHigh <= kThreads * kLaunchRegs, "register split");
// Lazy rescale of O: a row's running max m is only moved (and O, l scaled)
// when a tile's max exceeds it by more than this many log2 units, so P =
// 2^(x - m) <= 2^64 between rescales.  Then l <= 2^(64 + 16) for up to 2^16
// keys and |O| <= 2^86 for |V| <= 2^6, far below the fp32 and bf16 limit of
// 2^128, while bf16 keeps P's relative precision at any magnitude.  With
// x10 outliers in q and k a row's max keeps jumping by more than 2^8 long
// into the key sequence, and each jump cost the warp a TMEM round trip of O
// on the softmax's critical path (stress14b: 2^64 instead of 2^8 is 1.8%
// faster).
constexpr float kRescaleThreshold = 64.0f;

template <int N>
__device__ __forceinline__ void regs_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

template <int N>
__device__ __forceinline__ void regs_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ uint64_t f2u(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}

__device__ __forceinline__ void u2f(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}

// (a0, a1) * bb + cc, two lanes in one instruction
__device__ __forceinline__ void ffma2(float& o0, float& o1, float a0, float a1, uint64_t bb,
                                      uint64_t cc) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(f2u(a0, a1)), "l"(bb), "l"(cc));
  u2f(r, o0, o1);
}

__device__ __forceinline__ uint64_t fadd2(uint64_t a, float b0, float b1) {
  uint64_t r;
  asm("add.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(f2u(b0, b1)));
  return r;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&r);
}

struct Bars {
  uint64_t q_full;
  uint64_t s_full[2];
  uint64_t p_full[2];
  uint64_t o_final;
  uint64_t drain;
  uint64_t k_full[4];
  uint64_t k_empty[4];
  uint64_t v_full[4];
  uint64_t v_empty[4];
};

// Block-sparse launches: a role's walk over the key tiles that either query
// tile of the unit may attend (bitmaps in the kernel's tile order).  The
// current word's remaining bits stay in a register, so a step reads shared
// memory only when it moves to the next word.  start() takes a set bit (or
// n_all); the first next() returns it, each later one the following tile of
// the walk, or n_all past the last.
template <int W>
struct TileWalk {
  const uint32_t (*tm)[W];
  int n_all, w;
  uint32_t u;
  __device__ __forceinline__ void start(const uint32_t (*tm_)[W], int from, int n_all_) {
    tm = tm_;
    n_all = n_all_;
    w = from >> 5;
    u = from < n_all ? (tm[0][w] | tm[1][w]) & (~0u << (from & 31)) : 0u;
  }
  __device__ __forceinline__ int next() {
    const int words = (n_all + 31) >> 5;
    while (u == 0u) {
      if (++w >= words) return n_all;
      u = tm[0][w] | tm[1][w];
    }
    const int k = (w << 5) + __ffs(u) - 1;
    u &= u - 1u;
    return k;
  }
};

__device__ __forceinline__ void record_timeout(const AttnParams& p, volatile int* abort_flag) {
  *abort_flag = 1;
  atomicCAS(p.status, kStatusOk, kStatusTimeout);
}

// Instances: kSparse = a block-sparse tile mask is walked (all ones when the
// caller gives none); kOwn = a token-level mask inside the own chunk is
// applied (only with kSparse).  Each extra feature costs the per-tile loop,
// so a launch takes the leanest instance that covers it.
template <int D, bool kSparse, bool kOwn>
__global__ void __launch_bounds__(kThreads, 1) attend_kernel(const __grid_constant__ AttnParams p) {
  using C = AttnCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ Bars bars;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;
  __shared__ int last_split;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // Work unit, head-major so the CTAs that share a head's K/V run together.
  // The first n_full units run unsplit (one CTA each, the full waves); the
  // others are split n_split ways, the splits of a unit adjacent.
  const bool whole = (int)blockIdx.x < p.n_full;
  const int ns = whole ? 1 : p.n_split;  // key ranges of this unit
  const int split = whole ? 0 : (int)(blockIdx.x - p.n_full) % p.n_split;
  const int unit = whole ? (int)blockIdx.x : p.n_full + (int)(blockIdx.x - p.n_full) / p.n_split;
  const int sunit = unit - p.n_full;     // index among the split units
  const int qp = unit % p.n_qp;
  const int rest = unit / p.n_qp;
  const int ni = rest % p.n_nodes;
  const int h = rest / p.n_nodes;
  const AttnNode& nd = p.nodes[ni];
  const int n_all = nd.n_kv * p.nt_slot;  // key tiles of the node
  const int qt0 = 2 * qp;
  const bool has_q1 = qt0 + 1 < p.n_qt;
  // Under frame causality the own chunk's key tiles past the frame of the
  // pair's last query row hold no key that either query tile may see: the
  // node's key tiles [gap_lo, gap_hi) are skipped.
  int gap_lo = n_all, gap_hi = n_all;
  if (nd.frame_causal) {
    const int last_row = min((qt0 + (has_q1 ? 2 : 1)) * kTile, p.T) - 1;
    const int frame_end = (last_row / p.frame_tokens + 1) * p.frame_tokens;
    gap_lo = min((frame_end + kTile - 1) / kTile, p.nt_slot);
    gap_hi = p.nt_slot;
  }
  // the key tile after kt in this CTA's walk (dense instances)
  auto next_kt = [gap_lo, gap_hi](int kt) { return kt + 1 == gap_lo ? gap_hi : kt + 1; };
  // Key tiles of this CTA: a contiguous range of the node's tiles that are
  // not skipped, or under a block-sparse mask a contiguous range of the
  // tiles either query tile may attend (set in the prologue below).
  constexpr bool sparse = kSparse;  // a launch with a block-sparse tile mask
  const int n_eff = n_all - (gap_hi - gap_lo);
  int t_begin = (int)((long long)split * n_eff / ns);
  int n_tiles = (int)((long long)(split + 1) * n_eff / ns) - t_begin;
  if (t_begin >= gap_lo) t_begin += gap_hi - gap_lo;
  // per query tile, bit i = kernel key tile i (block-sparse instances only)
  __shared__ uint32_t tmask[2][kSparse ? kMaskWords : 1];
  __shared__ int sp_first, sp_count;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(&bars.q_full, 1);
    mbar_init(&bars.o_final, 2);  // one commit per MMA issuer
    mbar_init(&bars.drain, 2);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars.s_full[b], 1);
      mbar_init(&bars.p_full[b], 256);
    }
    for (int s = 0; s < C::kKStages; ++s) {
      mbar_init(&bars.k_full[s], 1);
      mbar_init(&bars.k_empty[s], 1);
    }
    for (int s = 0; s < C::kVStages; ++s) {
      mbar_init(&bars.v_full[s], 1);
      mbar_init(&bars.v_empty[s], 1);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_sh, C::kTmemCols);
    tmem_relinquish();
  }
  if constexpr (sparse) if (warp == 2) {
    // Gather the caller's mask rows of the two query tiles into the kernel's
    // key tile order (slot list without hidden context slots), then take
    // this split's share of the union's set bits.  Without a tile mask every
    // key tile is kept.
    const int words = (n_all + 31) >> 5;  // <= kMaskWords, checked on the host
    const uint32_t* row0 =
        p.tile_mask ? p.tile_mask + ((size_t)nd.q_index * p.n_qt + qt0) * p.mask_words : nullptr;
    const uint32_t* row1 = row0 ? row0 + p.mask_words : nullptr;
    int total = 0;
    for (int w = 0; w < words; ++w) {
      const int i = (w << 5) + lane;
      bool b0 = false, b1 = false;
      if (i < n_all && (i < gap_lo || i >= gap_hi)) {
        const int s = i / p.nt_slot;
        const int k = nd.src[s] * p.nt_slot + (i - s * p.nt_slot);
        b0 = row0 ? ((row0[k >> 5] >> (k & 31)) & 1u) != 0u : true;
        if (has_q1) b1 = row1 ? ((row1[k >> 5] >> (k & 31)) & 1u) != 0u : true;
      }
      const uint32_t m0 = __ballot_sync(0xffffffffu, b0);
      const uint32_t m1 = __ballot_sync(0xffffffffu, b1);
      if (lane == 0) {
        tmask[0][w] = m0;
        tmask[1][w] = m1;
      }
      total += __popc(m0 | m1);
    }
    if (lane == 0) {
      const int lo = (int)((long long)split * total / ns);
      const int hi = (int)((long long)(split + 1) * total / ns);
      int first = n_all, seen = 0;
      for (int w = 0; hi > lo && w < words; ++w) {
        uint32_t u = tmask[0][w] | tmask[1][w];
        const int cnt = __popc(u);
        if (seen + cnt > lo) {
          for (int r = lo - seen; r > 0; --r) u &= u - 1;  // drop the bits before the lo-th
          first = (w << 5) + __ffs(u) - 1;
          break;
        }
        seen += cnt;
      }
      sp_first = first;
      sp_count = hi - lo;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if constexpr (sparse) {
    t_begin = sp_first;
    n_tiles = sp_count;
  }
  const uint32_t tbase = tmem_base_sh;
  const uint64_t tmo = p.timeout_ns;

  uint8_t* sQ0 = smem + C::kOffQ0;
  uint8_t* sQ1 = smem + C::kOffQ1;
  uint8_t* sK = smem + C::kOffK;
  uint8_t* sV = smem + C::kOffV;
  int k_issued = 0, v_issued = 0;  // producer: tiles whose K / V copies were started

  if (warp < 4) {
    regs_dec<kRegsLow>();
    if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      prefetch_tmap(&p.tmap_q);
      prefetch_tmap(&p.tmap_kv);
      mbar_arrive_expect_tx(&bars.q_full, (has_q1 ? 2 : 1) * C::kTileBytes);
#pragma unroll
      for (int b = 0; b < C::kBoxes; ++b) {
        tma_load_4d(sQ0 + b * C::kBoxBytes, &p.tmap_q, &bars.q_full, b * 64, h, qt0 * kTile,
                    nd.q_index);
        if (has_q1)
          tma_load_4d(sQ1 + b * C::kBoxBytes, &p.tmap_q, &bars.q_full, b * 64, h,
                      (qt0 + 1) * kTile, nd.q_index);
      }
      const uint64_t keep = l2_policy_evict_last();
      TileWalk<kSparse ? kMaskWords : 1> walk;
      if constexpr (sparse) walk.start(tmask, t_begin, n_all);
      int i = sparse ? walk.next() : t_begin;  // key tile of the node
      for (int j = 0; j < n_tiles; ++j, i = sparse ? walk.next() : next_kt(i)) {
        const int ks = j % C::kKStages;
        const int vs = j % C::kVStages;
        const int slot = nd.slot[i / p.nt_slot];
        const int t = i - (i / p.nt_slot) * p.nt_slot;
        const int row_k = ((slot * 2 + 0) * p.H + h) * p.Tpad + t * kTile;
        const int row_v = row_k + p.H * p.Tpad;
        if (!mbar_wait(&bars.k_empty[ks], ((uint32_t)(j / C::kKStages) & 1u) ^ 1u, &abort_flag,
                       tmo)) {
          record_timeout(p, &abort_flag);
          break;
        }
        mbar_arrive_expect_tx(&bars.k_full[ks], C::kTileBytes);
#pragma unroll
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d_hint(sK + ks * C::kTileBytes + b * C::kBoxBytes, &p.tmap_kv,
                           &bars.k_full[ks], b * 64, row_k, keep);
        k_issued = j + 1;
        if (!mbar_wait(&bars.v_empty[vs], ((uint32_t)(j / C::kVStages) & 1u) ^ 1u, &abort_flag,
                       tmo)) {
          record_timeout(p, &abort_flag);
          break;
        }
        // fault_mode 1 (test hook): withhold the V copy of the second tile,
        // so the MMA issuer's bounded wait on it expires.
        if (!(p.fault_mode == 1 && j == 1)) {
          mbar_arrive_expect_tx(&bars.v_full[vs], C::kTileBytes);
#pragma unroll
          for (int b = 0; b < C::kBoxes; ++b)
            tma_load_2d_hint(sV + vs * C::kTileBytes + b * C::kBoxBytes, &p.tmap_kv,
                             &bars.v_full[vs], b * 64, row_v, keep);
        }
        v_issued = j + 1;
      }
    }
  } else if (warp == 1 || warp == 3) {
    // ------------------------------------------------------------ MMA issuers
    // The whole warp runs the loop (waits are voted warp-wide so every lane
    // takes the same branch); one elected lane issues each MMA and commit.
    {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, true);
      // Base descriptors are built once; an MMA's operand descriptor is its
      // base plus a compile-time offset (the start-address field holds
      // address >> 4 and every operand lies below 256 KB, so the add never
      // carries out of the field).  Rebuilding descriptors per MMA costs the
      // issuing warp about as long as the MMA itself takes.
      const uint64_t dQ[2] = {sdesc_sw128(smem_u32(sQ0), 16, 1024),
                              sdesc_sw128(smem_u32(sQ1), 16, 1024)};
      const uint64_t dK = sdesc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t dV = sdesc_sw128(smem_u32(sV), C::kBoxBytes, 1024);
      constexpr uint64_t kTileStep = (uint64_t)(C::kTileBytes >> 4);
      // Under a block-sparse mask a query tile may skip a key tile the other
      // query tile attends: its S and PV MMAs are then not issued (the S
      // barrier is still committed, so every barrier completes once per
      // tile), and its first issued PV starts the accumulator.
      auto vis = [&](int b, int kt) {
        return !sparse || ((tmask[b][kt >> 5] >> (kt & 31)) & 1u) != 0u;
      };
      bool pv_started = false;  // this issuer's query tile has a PV in O
      // S_b = Q_b K_i^T into TMEM buffer b
      auto issue_s = [&](int b, int i, bool v) {
        if (v) {
          const uint64_t kb = dK + (uint64_t)(i % C::kKStages) * kTileStep;
          const uint64_t qb = b == 0 ? dQ[0] : dQ[1];
          const uint32_t dcol = tbase + col_s(b);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t off = (uint64_t)(((kk >> 2) * C::kBoxBytes + (kk & 3) * 32) >> 4);
            mma_ss_warp(dcol, qb + off, kb + off, idesc_qk, kk > 0 ? 1u : 0u);
          }
        }
        mma_commit_warp(&bars.s_full[b]);
      };
      // O_b += P_b V_i with P_b read from TMEM over S_b
      auto issue_pv = [&](int b, int i) {
        const uint64_t vb = dV + (uint64_t)(i % C::kVStages) * kTileStep;
        const uint32_t ocol = tbase + col_o(b);
        const uint32_t pcol = tbase + col_s(b);
        const uint32_t acc0 = (sparse ? pv_started : i > 0) ? 1u : 0u;
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk)
          mma_ts_warp(ocol, pcol + kk * 8, vb + (uint64_t)((kk * 2048) >> 4), idesc_pv,
                 kk > 0 ? 1u : acc0);
        if (sparse) pv_started = true;
      };
      auto wait = [&](uint64_t* bar, uint32_t parity) {
        return __all_sync(0xffffffffu, mbar_wait(bar, parity, &abort_flag, tmo));
      };
      auto wait_k = [&](int i) {
        return wait(&bars.k_full[i % C::kKStages], (uint32_t)(i / C::kKStages) & 1u);
      };
      const int bq = warp == 1 ? 0 : 1;  // the query tile this warp issues for
      bool ok = wait(&bars.q_full, 0);
      if (bq == 0 || has_q1) {
        TileWalk<kSparse ? kMaskWords : 1> walk;
        if constexpr (sparse) walk.start(tmask, t_begin, n_all);
        int kt = sparse ? walk.next() : t_begin;  // key tile of the node at iteration i
        if (n_tiles > 0) {  // a block-sparse range may be empty: then only o_final is committed
          ok = ok && wait_k(0);
          if (ok) {
            tc_fence_after();
            issue_s(bq, 0, vis(bq, kt));
          }
        }
        for (int i = 0; ok && i < n_tiles; ++i) {
          const uint32_t par = (uint32_t)i & 1u;
          const bool more = i + 1 < n_tiles;
          const int kt_next = !more ? kt : (sparse ? walk.next() : next_kt(kt));
          const bool vis_cur = vis(bq, kt), vis_next = more && vis(bq, kt_next);
          // V_i and K_{i+1} normally land before the softmax hands over P_b,
          // so their waits go first, off the path from P_b to the next MMA.
          if (!wait(&bars.v_full[i % C::kVStages], (uint32_t)(i / C::kVStages) & 1u) ||
              (more && !wait_k(i + 1)) || !wait(&bars.p_full[bq], par)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (vis_cur) issue_pv(bq, i);
          if (more) issue_s(bq, i + 1, vis_next);
          kt = kt_next;
        }
      }
      if (ok) {
        mma_commit_warp(&bars.o_final);
      } else if (lane == 0) {
        record_timeout(p, &abort_flag);
      }
    }
    }
    // ---------------------------------------------------------------- teardown (warpgroup 0)
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (abort_flag) {
      // Some wait expired.  Before the CTA exits, wait (bounded, ignoring
      // the abort flag) for what this CTA still has in flight: the TMA
      // copies the producer started (a stage's barrier cannot run ahead of
      // the last copy started into it) and every MMA the issuers started.
      const int zero = 0;
      if (warp == 0 && lane == 0) {
        mbar_wait(&bars.q_full, 0, &zero, tmo);
        for (int i = (k_issued > C::kKStages ? k_issued - C::kKStages : 0); i < k_issued; ++i)
          mbar_wait(&bars.k_full[i % C::kKStages], (uint32_t)(i / C::kKStages) & 1u, &zero, tmo);
        for (int i = (v_issued > C::kVStages ? v_issued - C::kVStages : 0); i < v_issued; ++i) {
          if (p.fault_mode == 1 && i == 1) continue;  // the copy the test hook withheld
          mbar_wait(&bars.v_full[i % C::kVStages], (uint32_t)(i / C::kVStages) & 1u, &zero, tmo);
        }
      } else if (warp == 1 || warp == 3) {
        mma_commit_warp(&bars.drain);  // the same elected lane that issued the MMAs
        mbar_wait(&bars.drain, 0, &zero, tmo);
      }
    }
    __syncwarp();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tbase, C::kTmemCols);
    }
  } else {
    regs_inc<kRegsHigh>();
    // ------------------------------------------------------------ softmax + epilogue
    // All eight softmax warps work on one query tile at a time (tile 0, then
    // tile 1, of every key tile).  A warp covers 16 rows, half of its TMEM
    // lane quarter, with two threads per row (16x32bx2 shape): thread t < 16
    // holds keys 0..63 of its row, thread t + 16 keys 64..127 of the same
    // row.  Both threads of a row keep the same running max (the two halves'
    // maxima are exchanged with one shuffle) and each its part of the sum,
    // so each thread exponentiates 64 keys per tile instead of 128 and the
    // two warps sharing a sub-partition overlap their MUFU and FMA work.
    constexpr int DH = D / 2;                      // output columns per thread
    const int q4 = warp & 3;                       // TMEM lane quarter this warp may access
    const int hi = warp >> 3;                      // which 16 lanes of the quarter
    const int half = lane >> 4;                    // which 64 keys, which D/2 columns
    const int row = q4 * 32 + hi * 16 + (lane & 15);  // query row inside a tile
    const uint32_t lane_off = (uint32_t)(q4 * 32 + hi * 16) << 16;
    const int nb = has_q1 ? 2 : 1;
    const float sl2 = p.scale_log2;
    const uint64_t sl2x2 = f2u(sl2, sl2);
    const int frame_causal = nd.frame_causal;
    bool o_has[2] = {false, false};       // O_b holds a PV (some key tile was attended)
    float m[2] = {-INFINITY, -INFINITY};  // running max of scale*log2(e)*logit per query tile
    float l[2] = {0.0f, 0.0f};            // this thread's part of the running sum of 2^(x - m)
    // first token of the latent frame after this row's (frame-causal mask)
    int frame_end[2];
#pragma unroll
    for (int b = 0; b < 2; ++b)
      frame_end[b] = ((qt0 + b) * kTile + row) / p.frame_tokens * p.frame_tokens + p.frame_tokens;
    // The softmax sees S_0 and then S_1 of key tile i complete.  S_b,i
    // follows PV_b,i-1 in its issuer's order, so once both are seen every
    // MMA that reads K stage i or V stage i-1 has completed, and one softmax
    // thread hands both stages back to the producer when it sees the last S
    // of the tile (S_1, or S_0 without a second query tile).  The MMA warps
    // then commit only to their S barriers (a commit costs an issuer about
    // as long as an MMA).
    const bool releaser = warp == 4 && lane == 0;
    bool ok = true;
    TileWalk<kSparse ? kMaskWords : 1> walk;
    if constexpr (sparse) walk.start(tmask, t_begin, n_all);
    int kt = sparse ? walk.next() : t_begin;  // key tile of the node
    int kt_next = kt;
    for (int i = 0; ok && i < n_tiles; ++i, kt = kt_next) {
      // The next tile of the walk and, under a tile mask, which query tiles
      // attend this one: read from shared memory before the S wait, so their
      // latency is not added to the path from S to P.
      kt_next = sparse ? walk.next() : next_kt(kt);
      const uint32_t attends = sparse ? ((tmask[0][kt >> 5] >> (kt & 31)) & 1u) |
                                            (((tmask[1][kt >> 5] >> (kt & 31)) & 1u) << 1)
                                      : 3u;
      const int t = kt % p.nt_slot;  // key tile inside its slot
      const int valid_tile = (t == p.nt_slot - 1) ? p.valid_last : kTile;
      const bool own_fc = frame_causal && kt < p.nt_slot;
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        if (b == 1 && !has_q1) break;
        // token-level mask (token-mask instance): this thread's 64 bits of its
        // row for this key tile, from the own-chunk mask or from the history
        // mask of the tile's key state (the caller's context index); fetched
        // before the wait so that the load hides behind it
        const int kst = kOwn ? kt / p.nt_slot : 0;  // key state: 0 own, then the visible contexts
        const bool own_tile = kOwn && (kst == 0 ? p.own_mask : p.hist_mask) != nullptr;
        uint32_t ow[2] = {~0u, ~0u};
        if (own_tile) {
          const int u = (qt0 + b) * kTile + row;
          if (u < p.T) {  // rows past T are never stored
            const size_t qrow = (size_t)nd.q_index * p.T + u;
            const uint32_t* mrow =
                kst == 0 ? p.own_mask + qrow * p.own_words
                         : p.hist_mask + (qrow * p.hist_states + (nd.src[kst] - 1)) * p.hist_words;
            const int words = kst == 0 ? p.own_words : p.hist_words;
            const int wi = (kt - kst * p.nt_slot) * 4 + half * 2;  // key 128 t + 64 half of the state
            ow[0] = wi < words ? __ldg(mrow + wi) : 0u;
            ow[1] = wi + 1 < words ? __ldg(mrow + wi + 1) : 0u;
          }
        }
        ok = mbar_wait(&bars.s_full[b], (uint32_t)i & 1u, &abort_flag, tmo);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        if (releaser && b == nb - 1) {
          mbar_arrive(&bars.k_empty[i % C::kKStages]);
          if (i > 0) mbar_arrive(&bars.v_empty[(i - 1) % C::kVStages]);
        }
        if (sparse && !((attends >> b) & 1u)) {
          // query tile b skips this key tile: no S was computed, no P is due
          mbar_arrive(&bars.p_full[b]);
          continue;
        }
        tc_fence_after();
        const uint32_t scol = tbase + lane_off + col_s(b);
        const uint32_t ocol = tbase + lane_off + col_o(b);
        // own-chunk tile under frame causality: keys up to the end of this
        // row's latent frame are visible (tile 0, frame 0, always is)
        const int valid = own_fc ? min(valid_tile, frame_end[b] - t * kTile) : valid_tile;
        const int vrel = valid - half * 64;  // visible keys among this thread's 64
        // The loads also reduce each 32-column chunk to its maximum, so a
        // full tile needs no max tree; a tile with masked keys (the ragged
        // last tile of a slot, frame causality) takes the max over what is
        // left after masking.
        uint32_t s[2][32];
        float cmax[2];
        tmem_ld16x2_32_max<64>(scol, s[0], cmax[0]);
        tmem_ld16x2_32_max<64>(scol + 32, s[1], cmax[1]);
        tmem_wait_ld(s[0]);
        tmem_wait_ld(s[1]);
        tmem_wait_ld_max2(cmax);
        float m_part = fmaxf(cmax[0], cmax[1]);
        // Tiles that can hold masked keys (a slot's ragged last tile, the own
        // chunk under frame causality) take the masked path; the test is the
        // same for every thread, so it needs no vote.
        if (valid_tile < kTile || own_fc || own_tile) {
          float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (c * 32 + e >= vrel || !((ow[c] >> e) & 1u)) s[c][e] = __float_as_uint(-INFINITY);
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 32; e += 8) {
              const int k = (c & 1) * 2 + (e >> 4);
              mx[k] = max3(mx[k], __uint_as_float(s[c][e]), __uint_as_float(s[c][e + 1]));
              mx[k] = max3(mx[k], __uint_as_float(s[c][e + 2]), __uint_as_float(s[c][e + 3]));
              mx[k] = max3(mx[k], __uint_as_float(s[c][e + 4]), __uint_as_float(s[c][e + 5]));
              mx[k] = max3(mx[k], __uint_as_float(s[c][e + 6]), __uint_as_float(s[c][e + 7]));
            }
          m_part = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        }
        const float m_tile = fmaxf(m_part, __shfl_xor_sync(0xffffffffu, m_part, 16)) * sl2;
        const float m_new = fmaxf(m[b], m_tile);
        const bool need = m_new > m[b] + kRescaleThreshold;
        if (__any_sync(0xffffffffu, need)) {
          // 0 when the row's first visible keys arrive (m = -inf); 1 for a row
          // of the warp whose max did not move (also when it is still -inf:
          // -inf - -inf would be NaN)
          const float alpha = m_new > m[b] ? ex2(m[b] - m_new) : 1.0f;
          if (sparse ? o_has[b] : i > 0) {
            // O_b holds the sum over earlier tiles: the commit that completed
            // S_b of this tile came after PV_b of the previous one.
#pragma unroll
            for (int c = 0; c < DH / 32; ++c) {
              uint32_t o[32];
              tmem_ld16x2_32<DH>(ocol + c * 32, o);
              tmem_wait_ld(o);
#pragma unroll
              for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
              tmem_st16x2_32<DH>(ocol + c * 32, o);
            }
            tmem_wait_st();
          }
          l[b] *= alpha;
          m[b] = m_new;
        }
        // m stays -inf while a row has seen no visible key (possible in a key
        // range that starts past a row's frame under frame causality); its
        // scores are then all -inf and must give P = 0, not NaN.
        const float m_sub = (m[b] == -INFINITY) ? 0.0f : m[b];
        const uint64_t negm = f2u(-m_sub, -m_sub);
        uint64_t acc[4] = {0, 0, 0, 0};
        // P of 32 keys packs into 16 words, written over the first half of
        // the same registers (word e/2 is written after elements e, e+1 are
        // read); the two halves make one 32-column store over S (keys
        // 0..63 of the row at columns 0..31, keys 64..127 at 32..63).
#pragma unroll
        for (int c = 0; c < 2; ++c) {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float x0, x1;
            ffma2(x0, x1, __uint_as_float(s[c][e]), __uint_as_float(s[c][e + 1]), sl2x2, negm);
            const float p0 = ex2(x0);
            const float p1 = ex2(x1);
            acc[(e >> 1) & 3] = fadd2(acc[(e >> 1) & 3], p0, p1);
            s[c][e >> 1] = pack_bf16(p0, p1);
          }
        }
        tmem_st16x2_32_halves<32>(scol, s[0], s[1]);
        float a0, a1, a2, a3, a4, a5, a6, a7;
        u2f(acc[0], a0, a1);
        u2f(acc[1], a2, a3);
        u2f(acc[2], a4, a5);
        u2f(acc[3], a6, a7);
        l[b] += ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&bars.p_full[b]);
        if (sparse) o_has[b] = true;
      }
    }
    if (ok) {
      ok = mbar_wait(&bars.o_final, 0, &abort_flag, tmo);
      ok = __all_sync(0xffffffffu, ok);
    }
    if (!ok) record_timeout(p, &abort_flag);
    float l_row[2];  // the row's whole sum: both halves, under the same max
#pragma unroll
    for (int b = 0; b < 2; ++b) l_row[b] = l[b] + __shfl_xor_sync(0xffffffffu, l[b], 16);
    if (ns == 1) {
      if (ok) {
        tc_fence_after();
#pragma unroll
        for (int b = 0; b < 2; ++b) {
          if (b == 1 && !has_q1) break;
          const int token = (qt0 + b) * kTile + row;
          const bool in_range = token < p.T;
          __nv_bfloat16* orow = static_cast<__nv_bfloat16*>(p.out) +
                                (((size_t)nd.q_index * p.T + token) * p.H + h) * D + DH * half;
          const float inv_l = l_row[b] > 0.0f ? 1.0f / l_row[b] : 0.0f;  // no visible key: O = 0
#pragma unroll
          for (int c = 0; c < DH / 32; ++c) {
            uint32_t o[32];
            if (sparse ? o_has[b] : n_tiles > 0) {  // some key tile was attended
              tmem_ld16x2_32<DH>(tbase + lane_off + col_o(b) + c * 32, o);
              tmem_wait_ld(o);
            } else {  // no key tile attended in this range (block-sparse): no MMA wrote O
#pragma unroll
              for (int e = 0; e < 32; ++e) o[e] = 0u;
            }
            if (in_range) {
              uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
              for (int v = 0; v < 4; ++v) {
                uint4 w;
                w.x = pack_bf16(__uint_as_float(o[v * 8 + 0]) * inv_l, __uint_as_float(o[v * 8 + 1]) * inv_l);
                w.y = pack_bf16(__uint_as_float(o[v * 8 + 2]) * inv_l, __uint_as_float(o[v * 8 + 3]) * inv_l);
                w.z = pack_bf16(__uint_as_float(o[v * 8 + 4]) * inv_l, __uint_as_float(o[v * 8 + 5]) * inv_l);
                w.w = pack_bf16(__uint_as_float(o[v * 8 + 6]) * inv_l, __uint_as_float(o[v * 8 + 7]) * inv_l);
                dst[v] = w;
              }
            }
          }
          if (p.lse != nullptr && in_range && half == 0)
            p.lse[((size_t)nd.q_index * p.H + h) * p.T + token] =
                (m[b] + __log2f(l_row[b])) * 0.69314718055994531f;
        }
      }
    } else {
      // Split unit.  Partial layout per (unit, split): O as [D/4][256]
      // float4 (rows of both query tiles), then m[256], then l[256].
      constexpr size_t kItem = (size_t)256 * (D + 2);
      float* part = p.ws + ((size_t)sunit * ns + split) * kItem;
      if (ok) {
        tc_fence_after();
        float4* part4 = reinterpret_cast<float4*>(part);
#pragma unroll
        for (int b = 0; b < 2; ++b) {
          if (b == 1 && !has_q1) break;
          const int r = b * 128 + row;
          const float inv_l = l_row[b] > 0.0f ? 1.0f / l_row[b] : 0.0f;  // no visible key here
#pragma unroll
          for (int c = 0; c < DH / 32; ++c) {
            uint32_t o[32];
            if (sparse ? o_has[b] : n_tiles > 0) {  // some key tile was attended
              tmem_ld16x2_32<DH>(tbase + lane_off + col_o(b) + c * 32, o);
              tmem_wait_ld(o);
            } else {  // no key tile attended in this range (block-sparse): no MMA wrote O
#pragma unroll
              for (int e = 0; e < 32; ++e) o[e] = 0u;
            }
#pragma unroll
            for (int v = 0; v < 8; ++v)
              part4[(DH * half / 4 + c * 8 + v) * 256 + r] =
                  make_float4(__uint_as_float(o[v * 4 + 0]) * inv_l, __uint_as_float(o[v * 4 + 1]) * inv_l,
                              __uint_as_float(o[v * 4 + 2]) * inv_l, __uint_as_float(o[v * 4 + 3]) * inv_l);
          }
          if (half == 0) {
            part[D * 256 + r] = m[b];
            part[D * 256 + 256 + r] = l_row[b];
          }
        }
      }
      __threadfence();
      // Every softmax thread of the CTA passes both barriers, whatever its
      // wait results were, so none can be left waiting here.
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (threadIdx.x == 128) {
        int last = 0;
        if (!abort_flag) last = atomicAdd(&p.ws_count[sunit], 1) == ns - 1;
        last_split = last;
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (last_split) {
        __threadfence();
        const float* base = p.ws + (size_t)sunit * ns * kItem;
#pragma unroll
        for (int b = 0; b < 2; ++b) {
          if (b == 1 && !has_q1) break;
          const int r = b * 128 + row;
          const int token = (qt0 + b) * kTile + row;
          if (token >= p.T) continue;
          float mk[kMaxSplit], wk[kMaxSplit];
          float M = -INFINITY;
#pragma unroll
          for (int k = 0; k < kMaxSplit; ++k) {
            mk[k] = k < ns ? __ldcg(base + k * kItem + D * 256 + r) : -INFINITY;
            M = fmaxf(M, mk[k]);
          }
          const float M_sub = (M == -INFINITY) ? 0.0f : M;  // every range empty: O = 0
          float L = 0.0f;
#pragma unroll
          for (int k = 0; k < kMaxSplit; ++k) {
            wk[k] = k < ns
                        ? __ldcg(base + k * kItem + D * 256 + 256 + r) * ex2(mk[k] - M_sub)
                        : 0.0f;
            L += wk[k];
          }
          const float inv_L = L > 0.0f ? 1.0f / L : 0.0f;
#pragma unroll
          for (int k = 0; k < kMaxSplit; ++k) wk[k] *= inv_L;
          uint4* orow4 = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(p.out) +
                                                  (((size_t)nd.q_index * p.T + token) * p.H + h) * D);
          // Loads of absent splits are predicated off rather than broken out
          // of, so every load of an iteration is in flight at once (a loop
          // that waited for each L2 round trip in turn took ~9 us per CTA).
#pragma unroll 2
          for (int c8 = half * (D / 16); c8 < (half + 1) * (D / 16); ++c8) {
            float4 x[kMaxSplit], y[kMaxSplit];
#pragma unroll
            for (int k = 0; k < kMaxSplit; ++k) {
              const float4* b4 = reinterpret_cast<const float4*>(base + k * kItem);
              x[k] = k < ns ? __ldcg(b4 + (c8 * 2 + 0) * 256 + r) : make_float4(0.f, 0.f, 0.f, 0.f);
              y[k] = k < ns ? __ldcg(b4 + (c8 * 2 + 1) * 256 + r) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int k = 0; k < kMaxSplit; ++k) {
              a[0] += wk[k] * x[k].x; a[1] += wk[k] * x[k].y; a[2] += wk[k] * x[k].z; a[3] += wk[k] * x[k].w;
              a[4] += wk[k] * y[k].x; a[5] += wk[k] * y[k].y; a[6] += wk[k] * y[k].z; a[7] += wk[k] * y[k].w;
            }
            uint4 w;
            w.x = pack_bf16(a[0], a[1]);
            w.y = pack_bf16(a[2], a[3]);
            w.z = pack_bf16(a[4], a[5]);
            w.w = pack_bf16(a[6], a[7]);
            orow4[c8] = w;
          }
          if (p.lse != nullptr && half == 0)
            p.lse[((size_t)nd.q_index * p.H + h) * p.T + token] = (M + __log2f(L)) * 0.69314718055994531f;
        }
        if (threadIdx.x == 128) p.ws_count[sunit] = 0;  // ready for the next launch
      }
    }
    // ---------------------------------------------------------------- teardown (softmax)
    __syncwarp();
    tc_fence_before();
    __syncthreads();
  }
}

// One-time per-device set-up of the kernel instances (shared-memory limit,
// register check), done under a lock so that two host threads launching on
// the same device for the first time cannot race.
template <int D>
cudaError_t configure_d(int dev) {
  using C = AttnCfg<D>;
  static std::mutex mu;
  static bool configured[64] = {};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (configured[dev]) return cudaSuccess;
  cudaError_t e;
  for (auto k : {attend_kernel<D, false, false>, attend_kernel<D, true, false>,
                 attend_kernel<D, true, true>}) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
    if (e != cudaSuccess) return e;
  }
  // setmaxnreg.inc waits until the block's register pool can serve it: a
  // build whose launch register count leaves the split short would never
  // proceed, so such a build is refused here.
  for (auto k : {attend_kernel<D, false, false>, attend_kernel<D, true, false>,
                 attend_kernel<D, true, true>}) {
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, k);
    if (e != cudaSuccess) return e;
    if (fa.numRegs * kThreads < 4 * 32 * kRegsLow + 8 * 32 * kRegsHigh)
      return cudaErrorInvalidConfiguration;
  }
  configured[dev] = true;
  return cudaSuccess;
}

template <int D>
cudaError_t launch_d(const AttnParams& p, int grid, cudaStream_t s) {
  using C = AttnCfg<D>;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = configure_d<D>(dev);
  if (e != cudaSuccess) return e;
  if (p.masked && (p.own_mask != nullptr || p.hist_mask != nullptr))
    attend_kernel<D, true, true><<<grid, kThreads, C::kSmemBytes, s>>>(p);
  else if (p.masked)
    attend_kernel<D, true, false><<<grid, kThreads, C::kSmemBytes, s>>>(p);
  else
    attend_kernel<D, false, false><<<grid, kThreads, C::kSmemBytes, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attend(const AttnParams& p, int head_dim, int grid, cudaStream_t s) {
  if (head_dim == 128) return launch_d<128>(p, grid, s);
  if (head_dim == 64) return launch_d<64>(p, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace sva
