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
// One CTA computes one work unit (node, head, 128-query tile) and streams
// every key tile of every slot the node reads:
//   warp 0    TMA producer: Q once, then K and V tiles of the slot list into
//             a ring of shared-memory stages (128B swizzle);
//   warp 1    MMA issuer (one thread): S = Q K^T into one of two TMEM
//             buffers, then O += P V with P read from TMEM;
//   warps 2-5 softmax: one query row per thread; S from TMEM, fp32 online
//             softmax in the log2 domain with a lazy rescale of O, P written
//             back into the S buffer as bf16; then the epilogue (O / l to
//             bf16 global, optional LSE).
// TMEM columns: S0 [0,128), S1 [128,256), O [256, 256+d).
// All waits are bounded (1 s by default): on expiry the CTA records
// SVA_ERR_DEVICE_TIMEOUT in the status word, drains its own copies and MMAs,
// frees TMEM and exits.
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
  static constexpr int kStages = (D == 128) ? 3 : 4;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kTileBytes;
  static constexpr int kOffV = kOffK + kStages * kTileBytes;
  static constexpr int kSmemBytes = kOffV + kStages * kTileBytes + 1024;  // + alignment slack
  static constexpr uint32_t kColS = 0;      // S buffers at columns 0 and 128
  static constexpr uint32_t kColO = 256;
  static constexpr uint32_t kTmemCols = 512;
};

constexpr int kThreads = 192;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: P <= 2^8 between rescales

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&r);
}

struct Bars {
  uint64_t q_full;
  uint64_t s_full[2];
  uint64_t p_full[2];
  uint64_t o_ready;
  uint64_t o_final;
  uint64_t drain;
  uint64_t k_full[4];
  uint64_t k_empty[4];
  uint64_t v_full[4];
  uint64_t v_empty[4];
};

__device__ __forceinline__ void record_timeout(const AttnParams& p, volatile int* abort_flag) {
  *abort_flag = 1;
  atomicCAS(p.status, kStatusOk, kStatusTimeout);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) attend_kernel(const __grid_constant__ AttnParams p) {
  using C = AttnCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ Bars bars;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // Work unit, head-major so the CTAs that share a head's K/V run together.
  const int unit = blockIdx.x;
  const int qt = unit % p.n_qt;
  const int rest = unit / p.n_qt;
  const int ni = rest % p.n_nodes;
  const int h = rest / p.n_nodes;
  const AttnNode& nd = p.nodes[ni];
  const int n_tiles = nd.n_kv * p.nt_slot;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(&bars.q_full, 1);
    mbar_init(&bars.o_ready, 1);
    mbar_init(&bars.o_final, 1);
    mbar_init(&bars.drain, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars.s_full[b], 1);
      mbar_init(&bars.p_full[b], 128);
    }
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars.k_full[s], 1);
      mbar_init(&bars.k_empty[s], 1);
      mbar_init(&bars.v_full[s], 1);
      mbar_init(&bars.v_empty[s], 1);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_sh, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = tmem_base_sh;
  const uint64_t tmo = p.timeout_ns;

  uint8_t* sQ = smem + C::kOffQ;
  uint8_t* sK = smem + C::kOffK;
  uint8_t* sV = smem + C::kOffV;
  int k_issued = 0, v_issued = 0;  // producer: tiles whose K / V copies were started

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      prefetch_tmap(&p.tmap_q);
      prefetch_tmap(&p.tmap_kv);
      mbar_arrive_expect_tx(&bars.q_full, C::kTileBytes);
#pragma unroll
      for (int b = 0; b < C::kBoxes; ++b)
        tma_load_4d(sQ + b * C::kBoxBytes, &p.tmap_q, &bars.q_full, b * 64, h, qt * kTile,
                    nd.q_index);
      const uint64_t keep = l2_policy_evict_last();
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % C::kStages;
        const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
        const int slot = nd.slot[i / p.nt_slot];
        const int t = i - (i / p.nt_slot) * p.nt_slot;
        const int row_k = ((slot * 2 + 0) * p.H + h) * p.Tpad + t * kTile;
        const int row_v = row_k + p.H * p.Tpad;
        if (!mbar_wait(&bars.k_empty[st], ph ^ 1u, &abort_flag, tmo)) {
          record_timeout(p, &abort_flag);
          break;
        }
        mbar_arrive_expect_tx(&bars.k_full[st], C::kTileBytes);
#pragma unroll
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d_hint(sK + st * C::kTileBytes + b * C::kBoxBytes, &p.tmap_kv,
                           &bars.k_full[st], b * 64, row_k, keep);
        k_issued = i + 1;
        if (!mbar_wait(&bars.v_empty[st], ph ^ 1u, &abort_flag, tmo)) {
          record_timeout(p, &abort_flag);
          break;
        }
        // fault_mode 1 (test hook): withhold the V copy of tile 1, so the
        // MMA issuer's bounded wait on it expires.
        if (!(p.fault_mode == 1 && i == 1)) {
          mbar_arrive_expect_tx(&bars.v_full[st], C::kTileBytes);
#pragma unroll
          for (int b = 0; b < C::kBoxes; ++b)
            tma_load_2d_hint(sV + st * C::kTileBytes + b * C::kBoxBytes, &p.tmap_kv,
                             &bars.v_full[st], b * 64, row_v, keep);
        }
        v_issued = i + 1;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, true);
      const uint32_t aQ = smem_u32(sQ);
      const uint32_t aK = smem_u32(sK);
      const uint32_t aV = smem_u32(sV);
      bool ok = mbar_wait(&bars.q_full, 0, &abort_flag, tmo);
      tc_fence_after();
      auto issue_qk = [&](int i) -> bool {
        const int st = i % C::kStages;
        const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
        if (!mbar_wait(&bars.k_full[st], ph, &abort_flag, tmo)) return false;
        tc_fence_after();
        const uint32_t dcol = tbase + C::kColS + (uint32_t)(i & 1) * 128u;
        const uint32_t kb = aK + st * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * C::kBoxBytes + (kk & 3) * 32;
          mma_ss(dcol, sdesc_sw128(aQ + off, 16, 1024), sdesc_sw128(kb + off, 16, 1024), idesc_qk,
                 kk > 0 ? 1u : 0u);
        }
        mma_commit(&bars.k_empty[st]);
        mma_commit(&bars.s_full[i & 1]);
        return true;
      };
      if (ok) ok = issue_qk(0);
      for (int i = 0; ok && i < n_tiles; ++i) {
        if (i + 1 < n_tiles && !issue_qk(i + 1)) {
          ok = false;
          break;
        }
        const int st = i % C::kStages;
        const uint32_t ph = (uint32_t)(i / C::kStages) & 1u;
        if (!mbar_wait(&bars.p_full[i & 1], (uint32_t)(i >> 1) & 1u, &abort_flag, tmo) ||
            !mbar_wait(&bars.v_full[st], ph, &abort_flag, tmo)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t pcol = tbase + C::kColS + (uint32_t)(i & 1) * 128u;
        const uint32_t vb = aV + st * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          mma_ts(tbase + C::kColO, pcol + kk * 8, sdesc_sw128(vb + kk * 2048, C::kBoxBytes, 1024),
                 idesc_pv, (i > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&bars.v_empty[st]);
        mma_commit(&bars.o_ready);
      }
      if (ok) {
        mma_commit(&bars.o_final);
      } else {
        record_timeout(p, &abort_flag);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax + epilogue
    const int q4 = warp & 3;                       // TMEM lane quarter this warp may access
    const int row = q4 * 32 + lane;                // query row inside the tile
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const float sl2 = p.scale_log2;
    float m = -INFINITY;  // running max of scale*log2(e)*logit (possibly stale by < threshold)
    float l = 0.0f;       // running sum of 2^(x - m)
    bool ok = true;
    for (int i = 0; i < n_tiles; ++i) {
      const int buf = i & 1;
      ok = mbar_wait(&bars.s_full[buf], (uint32_t)(i >> 1) & 1u, &abort_flag, tmo);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const uint32_t scol = tbase + lane_off + C::kColS + (uint32_t)buf * 128u;
      uint32_t s[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(scol + c * 32, s[c]);
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_wait_ld(s[c]);

      const int t = i % p.nt_slot;
      const int valid = (t == p.nt_slot - 1) ? p.valid_last : kTile;
      if (valid < kTile) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (c * 32 + e >= valid) s[c][e] = __float_as_uint(-INFINITY);
      }
      float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        mx0 = fmaxf(mx0, __uint_as_float(s[0][e]));
        mx1 = fmaxf(mx1, __uint_as_float(s[1][e]));
        mx2 = fmaxf(mx2, __uint_as_float(s[2][e]));
        mx3 = fmaxf(mx3, __uint_as_float(s[3][e]));
      }
      const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sl2;
      const float m_new = fmaxf(m, m_tile);
      const bool need = m_new > m + kRescaleThreshold;
      if (__any_sync(0xffffffffu, need)) {
        const float alpha = ex2(m - m_new);  // 0 on the first tile (m = -inf)
        if (i > 0) {
          // O holds the sum over tiles < i once PV_{i-1} is complete.
          ok = mbar_wait(&bars.o_ready, (uint32_t)(i - 1) & 1u, &abort_flag, tmo);
          ok = __all_sync(0xffffffffu, ok);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            const uint32_t ocol = tbase + lane_off + C::kColO + c * 32;
            tmem_ld32(ocol, o);
            tmem_wait_ld(o);
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st32(ocol, o);
          }
          tmem_wait_st();
        }
        l *= alpha;
        m = m_new;
      }
      float sum0 = 0.f, sum1 = 0.f;
      uint32_t pk[2][32];
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const float p0 = ex2(fmaf(__uint_as_float(s[c][e]), sl2, -m));
          const float p1 = ex2(fmaf(__uint_as_float(s[c][e + 1]), sl2, -m));
          sum0 += p0;
          sum1 += p1;
          pk[c >> 1][(c & 1) * 16 + (e >> 1)] = pack_bf16(p0, p1);
        }
      l += sum0 + sum1;
      tmem_st32(scol, pk[0]);
      tmem_st32(scol + 32, pk[1]);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&bars.p_full[buf]);
    }
    if (ok) {
      ok = mbar_wait(&bars.o_final, 0, &abort_flag, tmo);
      ok = __all_sync(0xffffffffu, ok);
    }
    if (!ok) {
      record_timeout(p, &abort_flag);
    } else {
      tc_fence_after();
      const int token = qt * kTile + row;
      const bool in_range = token < p.T;
      const float inv_l = 1.0f / l;
      __nv_bfloat16* orow = static_cast<__nv_bfloat16*>(p.out) +
                            (((size_t)nd.q_index * p.T + token) * p.H + h) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tbase + lane_off + C::kColO + c * 32, o);
        tmem_wait_ld(o);
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
      if (p.lse != nullptr && in_range) {
        p.lse[((size_t)nd.q_index * p.H + h) * p.T + token] = (m + __log2f(l)) * 0.69314718055994531f;
      }
    }
  }

  // ---------------------------------------------------------------- teardown
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (abort_flag && lane == 0) {
    // Some wait expired.  Before the CTA exits, wait (bounded, ignoring the
    // abort flag) for what this CTA still has in flight: the TMA copies the
    // producer started (a stage's barrier cannot run ahead of the last copy
    // started into it) and every MMA the issuer started.
    const int zero = 0;
    if (warp == 0) {
      mbar_wait(&bars.q_full, 0, &zero, tmo);
      for (int i = (k_issued > C::kStages ? k_issued - C::kStages : 0); i < k_issued; ++i)
        mbar_wait(&bars.k_full[i % C::kStages], (uint32_t)(i / C::kStages) & 1u, &zero, tmo);
      for (int i = (v_issued > C::kStages ? v_issued - C::kStages : 0); i < v_issued; ++i) {
        if (p.fault_mode == 1 && i == 1) continue;  // the copy the test hook withheld
        mbar_wait(&bars.v_full[i % C::kStages], (uint32_t)(i / C::kStages) & 1u, &zero, tmo);
      }
    } else if (warp == 1) {
      mma_commit(&bars.drain);
      mbar_wait(&bars.drain, 0, &zero, tmo);
    }
  }
  __syncwarp();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tbase, C::kTmemCols);
  }
}

template <int D>
cudaError_t launch_d(const AttnParams& p, int grid, cudaStream_t s) {
  using C = AttnCfg<D>;
  static bool configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    e = cudaFuncSetAttribute(attend_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  attend_kernel<D><<<grid, kThreads, C::kSmemBytes, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attend(const AttnParams& p, int head_dim, int grid, cudaStream_t s) {
  if (head_dim == 128) return launch_d<128>(p, grid, s);
  if (head_dim == 64) return launch_d<64>(p, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace sva
