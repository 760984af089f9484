// The linear projection in front of the attention layer: for every token row
// of x, y = x W^T + b, split into the q, k and v tensors that
// sva_rope_kv_write consumes (token-major [rows][H*d] each).  A dense
// contraction, so it runs on the tensor cores:
//
//   bf16 x [rows][C] (A, K-major) times bf16 W [3N][C] (B, K-major) into an
//   fp32 accumulator in TMEM, 256 x BN output tiles (BN = 256, or 128 when
//   N = H*d is not a multiple of 256), 64-wide K blocks through a TMA ring.
//
// Each tile is computed by a pair of CTAs (a cluster of two) with two-SM
// MMAs (tcgen05 cta_group::2, M = 256): CTA r of the pair loads rows
// [128 r, 128 r + 128) of the tile's x rows and rows [r BN/2, (r+1) BN/2) of
// its W rows into the same shared-memory offsets, the even CTA issues the
// MMAs, and each CTA's tensor memory receives its own 128 accumulator rows.
// Per SM a K block then brings 16 KB of x and BN/2 x 64 of W from L2 (32 KB
// at BN = 256) for 512 tensor cycles, against 48 KB for a one-SM 128 x 256
// tile.  Both CTAs' copies count toward the even CTA's stage barrier; the
// MMA commits free the stage in each CTA and hand the accumulator to each
// CTA's epilogue; the odd CTA's epilogue warps arrive remotely on the even
// CTA's accumulator-free barrier.
//
// Persistent pairs (one CTA per SM) walk a list of work items; two TMEM
// accumulators let the epilogue of one item (TMEM -> + bias -> bf16 ->
// global) overlap the main loop of the next.  Items are output tiles in
// groups of up to 16 row tiles, the row tile varying fastest inside a group:
// the pairs running at one time share each W column tile through L2, and a
// group's x rows (at most 16 x 256 rows) stay in L2 while the group sweeps
// the columns, so that W is read from HBM once per group even where it does
// not fit in L2.  When the tiles do not fill the last round of pairs, the
// tiles of that round are split into two half-width items (BN / 2 columns),
// so that the last round takes half as long.
//   warp 0      TMA producer (x and W tiles, 128-byte swizzle);
//   warp 1      TMEM owner (both CTAs) and MMA issuer (even CTA; whole warp,
//               one elected lane);
//   warps 4-11  epilogue: two warps per TMEM lane quarter, one output row per
//               thread, the two warps of a quarter taking alternate 32-column
//               chunks.  Each chunk (32 rows x 64 bytes) is staged in the
//               warp's shared-memory buffers and leaves by one TMA tile store
//               (two buffers per warp, reused once the store has read them):
//               a per-thread store would touch 32 rows per warp instruction.
// An item never straddles q, k and v (N is a multiple of BN), so its epilogue
// writes into one tensor.  With the fused RoPE epilogue (sva_qkv_project_rope)
// each thread rotates the pairs of its row's q and k columns in fp32 at the
// token's (t, h, w) position before the one bf16 rounding; Q' leaves token-
// major by tile store, K' and V by tile stores into the node's own cache
// slot (a 3D map of the slot pool that clips rows past T); a chunk whose 32
// rows belong to two nodes is scattered by the warp reading it back, eight
// whole 64-byte cache rows per store instruction.  Rows past `rows` read
// zeros (TMA fill) and are not stored; K past C reads zeros on both
// operands.  All waits are bounded: on expiry the CTA records
// SVA_ERR_DEVICE_TIMEOUT, drains its own copies and MMAs, frees TMEM and
// exits.
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "proj.h"
#include "ptx.cuh"

namespace sva {
namespace {

using namespace ptx;

constexpr int kProjThreads = 384;
constexpr int kMaxStages = 8;
constexpr int kBM = 128;       // accumulator rows per CTA (a pair's tile has 256)
constexpr int kBK = 64;
constexpr int kEpiWarps = 8;
constexpr int kGroupM = 16;    // row tiles per raster group
constexpr int kChunkBytes = 32 * 64;  // one staged 32 x 32 bf16 output chunk

template <int BN>
struct ProjCfg {
  static constexpr int kABytes = kBM * kBK * 2;        // 16 KB of x rows per CTA
  static constexpr int kBBytes = (BN / 2) * kBK * 2;   // this CTA's half of the W rows
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = BN == 256 ? 6 : 8;
  static constexpr int kOutBytes = kEpiWarps * 2 * kChunkBytes;  // output staging, 32 KB
  static constexpr int kSmemBytes = kStages * kStageBytes + kOutBytes + 1024;  // + alignment slack
  static constexpr uint32_t kTmemCols = 2 * BN;                   // two accumulators
  static_assert(kStages <= kMaxStages, "stage barriers");
  static_assert(kSmemBytes + 256 <= 227 * 1024, "shared memory per CTA");
};

struct ProjBars {
  uint64_t full[kMaxStages];   // even CTA: both CTAs' copies of a stage landed
  uint64_t empty[kMaxStages];  // this CTA's stage was read by the MMAs
  uint64_t acc_full[2];        // the accumulator of an item is complete
  uint64_t acc_empty[2];       // even CTA: both CTAs' epilogues read it (16 arrivals)
  uint64_t drain;
};

__device__ __forceinline__ uint32_t pack2_bf16(float lo, float hi) {
  __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&r);
}

__device__ __forceinline__ uint32_t rotate2_bf16(float x, float y, float2 cs) {
  const float rx = __fmaf_rn(x, cs.x, -(y * cs.y));
  const float ry = __fmaf_rn(x, cs.y, y * cs.x);
  return pack2_bf16(rx, ry);
}

// Tile store shared -> global through a 3D tensor map (bulk-group
// completion); elements outside the tensor's extent are not written.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int32_t c0,
                                             int32_t c1, int32_t c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(src), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

// ---------------------------------------------------------------- CTA pairs
//
// Two-SM MMAs (cta_group::2): a cluster of two CTAs on neighbouring SMs; the
// even-ranked CTA issues the MMAs, each reading its A rows and its half of
// B from the shared memory of its own CTA (the same offsets in both), and
// each CTA's tensor memory receives its own 128 accumulator rows.  Signals
// between the two CTAs go to barriers named by their shared::cluster
// address (mapa), one barrier per signal.

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// The shared::cluster address of the variable at `addr` (a shared::cta
// address of this CTA) in the CTA of rank `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Arrives once on a barrier of either CTA of the cluster (release at
// cluster scope: this thread's earlier writes are visible to the waiter).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}

// tma_load_2d whose completion is counted on a barrier that may belong to
// the peer CTA of the pair (`bar` is a shared::cluster address); the data
// lands in this CTA's shared memory.
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, uint32_t bar,
                                                 int32_t c0, int32_t c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}

// Tensor-memory allocation for a CTA pair: one warp of each of the two CTAs
// executes it; both get the same column base.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// D[tmem of both CTAs] (+)= A[smem of both] * B[smem of both], M = 256 rows
// (128 per CTA); issued by the even CTA only, warp-wide with one elected lane.
__device__ __forceinline__ void mma_ss_pair_warp(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n"
      " .reg .pred p, e;\n"
      " setp.ne.b32 p, %4, 0;\n"
      " elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on the barrier at shared::cluster address `bar` (this CTA's
// or the peer's) when every tcgen05 operation this thread issued so far has
// completed; warp-wide, one elected lane.
__device__ __forceinline__ void mma_commit_pair_warp(uint32_t bar) {
  asm volatile(
      "{\n"
      " .reg .pred e;\n"
      " elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];\n"
      "}\n" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void proj_timeout(const ProjParams& p, volatile int* abort_flag) {
  *abort_flag = 1;
  atomicCAS(p.status, kStatusOk, kStatusTimeout);
}

// Work item i: output tile (m, n), whole (half = -1) or its column half
// `half` (items past n_whole, two per tile).
struct Item {
  int m, n, half;
};

__device__ __forceinline__ Item item_of(const ProjParams& p, int i) {
  Item it;
  int t = i;
  it.half = -1;
  if (i >= p.n_whole) {
    t = p.n_whole + ((i - p.n_whole) >> 1);
    it.half = (i - p.n_whole) & 1;
  }
  // tile t of the raster: groups of kGroupM row tiles (the last may be
  // smaller), the row tile varying fastest inside a group
  const int per_group = kGroupM * p.n_ntiles;
  const int g = t / per_group;
  const int r = t - g * per_group;
  const int gm = min(kGroupM, p.n_mtiles - g * kGroupM);
  const int n = r / gm;
  it.m = g * kGroupM + (r - n * gm);
  it.n = n;
  return it;
}

template <int BN>
__global__ void __launch_bounds__(kProjThreads, 1) qkv_project_kernel(const __grid_constant__ ProjParams p) {
  using C = ProjCfg<BN>;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ ProjBars bars;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();  // 0: issues the MMAs of the pair
  const int pair = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bars.full[s], 1);
      mbar_init(&bars.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars.acc_full[b], 1);
      mbar_init(&bars.acc_empty[b], 2 * kEpiWarps);
    }
    mbar_init(&bars.drain, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(&tmem_base_sh, C::kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  // both CTAs' barriers are initialised before either signals the other's
  cluster_sync();
  tc_fence_after();
  const uint32_t tbase = tmem_base_sh;
  const uint64_t tmo = p.timeout_ns;
  int issued = 0;  // producer: K blocks whose copies were started

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      prefetch_tmap(&p.tmap_x);
      prefetch_tmap(&p.tmap_w);
      prefetch_tmap(&p.tmap_wh);
      const uint32_t full0 = mapa_shared(smem_u32(&bars.full[0]), 0);  // even CTA's barriers
      for (int i = pair; i < p.n_items; i += n_pairs) {
        const Item it = item_of(p, i);
        const bool half = it.half >= 0;
        // this CTA's part of the stage: its 128 x rows and its half of the W rows
        const uint32_t bytes = C::kABytes + (half ? C::kBBytes / 2 : C::kBBytes);
        const int x_row = it.m * 2 * kBM + (int)rank * kBM;
        const int w_row = it.n * BN + (half ? it.half * (BN / 2) + (int)rank * (BN / 4)
                                            : (int)rank * (BN / 2));
        bool ok = true;
        for (int kb = 0; kb < p.n_kblocks; ++kb, ++issued) {
          const int s = issued % kStages;
          const uint32_t ph = (uint32_t)(issued / kStages) & 1u;
          if (!mbar_wait(&bars.empty[s], ph ^ 1u, &abort_flag, tmo)) {
            proj_timeout(p, &abort_flag);
            ok = false;
            break;
          }
          uint8_t* sa = smem + s * C::kStageBytes;
          const uint32_t full = full0 + (uint32_t)(s * sizeof(uint64_t));
          if (rank == 0) mbar_arrive_expect_tx(&bars.full[s], 2 * bytes);  // both CTAs' bytes
          tma_load_2d_pair(sa, &p.tmap_x, full, kb * kBK, x_row);
          tma_load_2d_pair(sa + C::kABytes, half ? &p.tmap_wh : &p.tmap_w, full, kb * kBK, w_row);
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (rank == 0) {
      constexpr uint32_t idesc_whole = idesc_bf16_f32(2 * kBM, BN, false);
      constexpr uint32_t idesc_half = idesc_bf16_f32(2 * kBM, BN / 2, false);
      const uint64_t dA = sdesc_sw128(smem_u32(smem), 16, 1024);
      const uint64_t dB = sdesc_sw128(smem_u32(smem + C::kABytes), 16, 1024);
      constexpr uint64_t kStageStep = (uint64_t)(C::kStageBytes >> 4);
      const uint32_t empty_own = smem_u32(&bars.empty[0]);
      const uint32_t empty_peer = mapa_shared(empty_own, 1);
      const uint32_t accf_own = smem_u32(&bars.acc_full[0]);
      const uint32_t accf_peer = mapa_shared(accf_own, 1);
      auto wait = [&](uint64_t* bar, uint32_t parity) {
        return __all_sync(0xffffffffu, mbar_wait(bar, parity, &abort_flag, tmo));
      };
      bool ok = true;
      int k_it = 0, tc = 0;
      for (int i = pair; ok && i < p.n_items; i += n_pairs, ++tc) {
        const uint32_t idesc = item_of(p, i).half >= 0 ? idesc_half : idesc_whole;
        const int acc = tc & 1;
        if (!wait(&bars.acc_empty[acc], ((uint32_t)(tc >> 1) & 1u) ^ 1u)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dcol = tbase + (uint32_t)(acc * BN);
        for (int kb = 0; kb < p.n_kblocks; ++kb, ++k_it) {
          const int s = k_it % kStages;
          if (!wait(&bars.full[s], (uint32_t)(k_it / kStages) & 1u)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a = dA + (uint64_t)s * kStageStep;
          const uint64_t b = dB + (uint64_t)s * kStageStep;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)  // 32 bytes of K per MMA inside the swizzle atom
            mma_ss_pair_warp(dcol, a + (uint64_t)(kk * 2), b + (uint64_t)(kk * 2), idesc,
                             (kb > 0 || kk > 0) ? 1u : 0u);
          // the stage is free in each CTA once these MMAs have read it
          const uint32_t off = (uint32_t)(s * sizeof(uint64_t));
          mma_commit_pair_warp(empty_own + off);
          mma_commit_pair_warp(empty_peer + off);
        }
        if (!ok) break;
        const uint32_t off = (uint32_t)(acc * sizeof(uint64_t));
        mma_commit_pair_warp(accf_own + off);
        mma_commit_pair_warp(accf_peer + off);
      }
      if (!ok && lane == 0) proj_timeout(p, &abort_flag);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ epilogue
    const int q4 = warp & 3;           // TMEM lane quarter this warp may access
    const int part = (warp - 4) >> 2;  // which alternate 32-column chunks
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    // This warp's two staging buffers.  A chunk is 32 rows (one per lane) of
    // 64 bytes; 16-byte piece j of row r sits at piece j ^ ((r >> 1) & 3) (the
    // 64-byte swizzle of the output tensor maps), so that the eight lanes of
    // a shared-memory phase, four row pairs, hit 32 different banks.
    const uint32_t stage0 =
        smem_u32(smem + kStages * C::kStageBytes) + (uint32_t)((warp - 4) * 2 * kChunkBytes);
    int staged = 0;  // chunks this warp has staged
    // This lane's row of a chunk (16 words) into the next buffer, once the
    // bulk store that last read that buffer is done with it; a chunk that
    // will not leave by a bulk store first lets every such store finish
    // reading, whichever buffer it came from.
    auto stage = [&](const uint32_t (&w)[16], bool bulk) -> uint32_t {
      const uint32_t buf = stage0 + (uint32_t)((staged & 1) * kChunkBytes);
      ++staged;
      if (lane == 0) {
        if (bulk)
          bulk_wait_group_read<1>();
        else
          bulk_wait_group_read<0>();
      }
      __syncwarp();
      const uint32_t at = buf + (uint32_t)(lane * 64);
      const int sw = (lane >> 1) & 3;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        st_shared_v4(at + (uint32_t)((j ^ sw) << 4), w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
      return buf;
    };
    // A staged chunk to global by one bulk tensor store: columns [x, x + 32)
    // of rows [y, y + 32) of the map's tensor (rows past its extent are not
    // written).
    auto store_tile = [&](uint32_t buf, const CUtensorMap* map, int x, int y) {
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0 && y < p.rows) {
        tma_store_2d(map, buf, x, y);
        bulk_commit_group();
      }
    };
    // A staged chunk to rows scattered in the cache: row j * 8 + lane / 4 to
    // rowp[j] + off (rows with a null pointer are skipped); four lanes per
    // 64-byte row, eight whole rows per store instruction.
    auto store_rows = [&](uint32_t buf, const uint64_t (&rowp)[4], size_t off) {
      __syncwarp();
      const int piece = lane & 3;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int r = j * 8 + (lane >> 2);
        const uint4 v = ld_shared_v4(buf + (uint32_t)(r * 64 + ((piece ^ ((r >> 1) & 3)) << 4)));
        if (rowp[j] != 0)
          *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(rowp[j]) + off + piece * 8) = v;
      }
    };
    bool ok = true;
    int tc = 0;
    const uint32_t acce0 = mapa_shared(smem_u32(&bars.acc_empty[0]), 0);  // even CTA's
    for (int i = pair; ok && i < p.n_items; i += n_pairs, ++tc) {
      const Item it = item_of(p, i);
      const int width = it.half >= 0 ? BN / 2 : BN;  // output columns of this item
      const int acc = tc & 1;
      // Waits for this item's accumulator; what depends only on the item is
      // worked out (and fetched) before, while the MMAs still run.
      auto wait_acc = [&]() {
        const bool got = __all_sync(0xffffffffu, mbar_wait(&bars.acc_full[acc], (uint32_t)(tc >> 1) & 1u,
                                                            &abort_flag, tmo));
        tc_fence_after();
        return got;
      };
      const int col = it.n * BN + (it.half > 0 ? BN / 2 : 0);  // output column in [0, 3N)
      const int tensor = col / p.N;      // q, k or v
      const int c0 = col - tensor * p.N;  // column inside that tensor
      const int y0 = it.m * 2 * kBM + (int)rank * kBM + q4 * 32;  // first output row of this warp
      // 32 accumulator columns of this row: TMEM -> registers, plus the bias
      auto load_chunk = [&](int c, uint32_t (&r)[32], float (&bv)[32]) {
        tmem_ld32(tbase + lane_off + (uint32_t)(acc * BN + c * 32), r);
        tmem_wait_ld(r);
        if (p.bias != nullptr) {
          const float4* b4 = reinterpret_cast<const float4*>(p.bias + col + c * 32);
#pragma unroll
          for (int v = 0; v < 8; ++v) {
            const float4 x = __ldg(b4 + v);
            bv[4 * v] = x.x; bv[4 * v + 1] = x.y; bv[4 * v + 2] = x.z; bv[4 * v + 3] = x.w;
          }
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e) bv[e] = 0.0f;
        }
      };
      if (p.rope_on) {
        // Fused RoPE: this row's node, token and position, and where K' / V go
        const RopeParams& rp = p.rope;
        const long long grow = (long long)it.m * 2 * kBM + (int)rank * kBM + row;
        int tpos = 0, hh = 0, ww = 0;
        uint64_t cdst = 0;  // (slot, K or V, head 0, token u, dim 0) of the cache; 0 past `rows`
        if (grow < p.rows) {
          const int node = (int)(grow / rp.T);
          const int u = (int)(grow - (long long)node * rp.T);
          const int HpWp = rp.Hp * rp.Wp;
          const int f = u / HpWp;
          hh = (u - f * HpWp) / rp.Wp;
          ww = u - f * HpWp - hh * rp.Wp;
          tpos = rp.nodes[node].t_base + f;
          cdst = reinterpret_cast<uint64_t>(
              static_cast<__nv_bfloat16*>(rp.cache) +
              ((((size_t)rp.nodes[node].slot * 2 + (tensor == 2 ? 1 : 0)) * rp.H) * rp.Tpad + u) * rp.d);
        }
        uint64_t rowp[4];  // the cache rows this lane writes in store_rows
#pragma unroll
        for (int j = 0; j < 4; ++j) rowp[j] = __shfl_sync(0xffffffffu, cdst, j * 8 + (lane >> 2));
        // K' and V: when this warp's 32 rows are tokens of one node (rows past
        // that node's T, only possible for the last node, are clipped by the
        // slot-pool map), a chunk leaves by one tile store at (column, token
        // u0, (slot, K|V, head)); a chunk whose rows straddle two nodes goes
        // row by row.
        int u0 = 0, kv_plane = -1;  // first token; (slot * 2 + K|V) * H, or -1: row by row
        if (tensor != 0 && y0 < p.rows) {
          const int n0 = y0 / rp.T;
          u0 = y0 - n0 * rp.T;
          if (u0 + 32 <= rp.T || n0 == rp.n_nodes - 1)
            kv_plane = (rp.nodes[n0].slot * 2 + (tensor == 2 ? 1 : 0)) * rp.H;
        }
        // The 32-column chunk ci of every head in the item uses the same 16
        // (cos, sin) pairs, fetched once per chunk index (the next one while
        // the current one is rotated); this warp takes the chunk indices of
        // its parity.  Pairs [0, P0) rotate with the frame index, [P0, P0+P1)
        // with the patch row, the rest with the patch column (the values and
        // split of the RoPE + cache write); the patch-row and patch-column
        // tables here are the pair-major copies, so the 32 tokens of a warp
        // read neighbouring entries.  An item covers whole heads (the host
        // splits a tile only when its halves do).
        const int cpd = rp.d / 32;  // chunks per head (even: d is 64 or 128)
        const int heads = width / rp.d;
        const float2* pt = rp.tab_t + (size_t)tpos * rp.P0;  // this token's frame row
        auto load_cs = [&](int ci, float2 (&cs)[16]) {
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int pi = ci * 16 + e;
            const float2* a =
                pi < rp.P0 ? pt + pi
                           : (pi < rp.P0 + rp.P1 ? rp.tab_h + (size_t)(pi - rp.P0) * rp.Hp + hh
                                                 : rp.tab_w + (size_t)(pi - rp.P0 - rp.P1) * rp.Wp + ww);
            cs[e] = __ldg(a);
          }
        };
        float2 cs_next[16];
        if (tensor != 2) load_cs(part, cs_next);
        ok = wait_acc();
        if (!ok) break;
#pragma unroll 1
        for (int ci = part; ci < cpd; ci += 2) {
          float2 cs[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) cs[e] = cs_next[e];
          if (tensor != 2 && ci + 2 < cpd) load_cs(ci + 2, cs_next);
#pragma unroll 1
          for (int hb = 0; hb < heads; ++hb) {
            const int c = hb * cpd + ci;
            uint32_t r[32];
            float bv[32];
            load_chunk(c, r, bv);  // warp-collective: every thread, in range or not
            uint32_t w[16];
            if (tensor == 2) {
#pragma unroll
              for (int e = 0; e < 16; ++e)
                w[e] = pack2_bf16(__uint_as_float(r[2 * e]) + bv[2 * e], __uint_as_float(r[2 * e + 1]) + bv[2 * e + 1]);
            } else {
#pragma unroll
              for (int e = 0; e < 16; ++e)
                w[e] = rotate2_bf16(__uint_as_float(r[2 * e]) + bv[2 * e],
                                    __uint_as_float(r[2 * e + 1]) + bv[2 * e + 1], cs[e]);
            }
            if (tensor == 0) {
              store_tile(stage(w, true), &p.tmap_out[0], c0 + c * 32, y0);  // Q' token-major
            } else {
              const int head = (c0 + c * 32) / rp.d;
              if (kv_plane >= 0) {
                const uint32_t buf = stage(w, true);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                  tma_store_3d(&p.tmap_out[1], buf, ci * 32, u0, kv_plane + head);
                  bulk_commit_group();
                }
              } else {
                store_rows(stage(w, false), rowp, (size_t)head * rp.Tpad * rp.d + (size_t)ci * 32);
              }
            }
          }
        }
      } else {
        ok = wait_acc();
        if (!ok) break;
#pragma unroll 1
        for (int c = part; c < width / 32; c += 2) {
          uint32_t r[32];
          float bv[32];
          load_chunk(c, r, bv);  // warp-collective: every thread, in range or not
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; ++e)
            w[e] = pack2_bf16(__uint_as_float(r[2 * e]) + bv[2 * e], __uint_as_float(r[2 * e + 1]) + bv[2 * e + 1]);
          store_tile(stage(w, true), &p.tmap_out[tensor], c0 + c * 32, y0);
        }
      }
      // The MMA warp may overwrite this accumulator once every epilogue warp
      // of both CTAs has read its part (each thread waited for its own TMEM
      // loads).
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acce0 + (uint32_t)(acc * sizeof(uint64_t)));
    }
    // the bulk stores read this CTA's shared memory and must be complete
    // before it exits
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
    if (!ok) proj_timeout(p, &abort_flag);
  }

  // ---------------------------------------------------------------- teardown
  // Every MMA that reads this CTA's stages has completed, and its commits
  // have arrived here, once the last round of this CTA's stages is free
  // again (bounded wait).  After a timeout the even CTA also waits for its
  // stage barriers, whose phases count both CTAs' copies, and for every MMA
  // it issued.
  if (warp == 0 && lane == 0) {
    const int zero = 0;
    for (int i = (issued > kStages ? issued - kStages : 0); i < issued; ++i) {
      mbar_wait(&bars.empty[i % kStages], (uint32_t)(i / kStages) & 1u, &zero, tmo);
      if (abort_flag && rank == 0)
        mbar_wait(&bars.full[i % kStages], (uint32_t)(i / kStages) & 1u, &zero, tmo);
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (abort_flag && rank == 0 && warp == 1) {
    const int zero = 0;
    mma_commit_pair_warp(smem_u32(&bars.drain));
    mbar_wait(&bars.drain, 0, &zero, tmo);
  }
  __syncwarp();
  tc_fence_before();
  // neither CTA leaves (or frees tensor memory) while the other may still
  // signal its barriers or have MMAs read its shared memory
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tbase, C::kTmemCols);
  }
}

// One-time per-device set-up of a kernel instance (its shared-memory limit),
// done under a lock so that two host threads launching on the same device
// for the first time cannot race.
template <int BN>
cudaError_t configure_bn(int dev) {
  using C = ProjCfg<BN>;
  static std::mutex mu;
  static bool configured[64] = {};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (configured[dev]) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(qkv_project_kernel<BN>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  configured[dev] = true;
  return cudaSuccess;
}

template <int BN>
void pair_launch_config(cudaLaunchConfig_t* cfg, cudaLaunchAttribute* attr, int grid,
                        cudaStream_t s) {
  *cfg = cudaLaunchConfig_t{};
  cfg->gridDim = dim3((unsigned)grid, 1, 1);
  cfg->blockDim = dim3(kProjThreads, 1, 1);
  cfg->dynamicSmemBytes = ProjCfg<BN>::kSmemBytes;
  cfg->stream = s;
  attr->id = cudaLaunchAttributeClusterDimension;
  attr->val.clusterDim.x = 2;
  attr->val.clusterDim.y = 1;
  attr->val.clusterDim.z = 1;
  cfg->attrs = attr;
  cfg->numAttrs = 1;
}

template <int BN>
cudaError_t launch_bn(const ProjParams& p, int grid, cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = configure_bn<BN>(dev);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr;
  pair_launch_config<BN>(&cfg, &attr, grid, s);
  return cudaLaunchKernelEx(&cfg, qkv_project_kernel<BN>, p);
}

// Clusters of two (one CTA per SM) that can be resident at once on the
// current device, looked up once per device and instance.
template <int BN>
cudaError_t max_pairs_bn(int* out) {
  static std::mutex mu;
  static int pairs[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  e = configure_bn<BN>(dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (pairs[dev] == 0) {
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr;
    pair_launch_config<BN>(&cfg, &attr, 2, nullptr);
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, qkv_project_kernel<BN>, &cfg);
    if (e != cudaSuccess) return e;
    if (n < 1) return cudaErrorInvalidConfiguration;
    pairs[dev] = n;
  }
  *out = pairs[dev];
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_qkv_project(const ProjParams& p, int block_n, int grid, cudaStream_t s) {
  if (grid < 2 || grid % 2 != 0) return cudaErrorInvalidValue;
  if (block_n == 256) return launch_bn<256>(p, grid, s);
  if (block_n == 128) return launch_bn<128>(p, grid, s);
  return cudaErrorInvalidValue;
}

cudaError_t qkv_project_max_pairs(int block_n, int* pairs) {
  if (block_n == 256) return max_pairs_bn<256>(pairs);
  if (block_n == 128) return max_pairs_bn<128>(pairs);
  return cudaErrorInvalidValue;
}

}  // namespace sva
