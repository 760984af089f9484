// Fused 3D-RoPE + KV-cache scatter.
//
// Writing a node's keys and values into the (chunk, level)-indexed cache is
// what makes its features available to later nodes and, under progressive
// history, to the other nodes of the same pipeline round (Section 3.3).  The
// rotary embedding is this library's reading of the positional encoding (the
// paper names none): 3D RoPE over (t, h, w) at absolute positions, pairs of
// adjacent head-dimension elements, rotated in fp32 with cos/sin tables that
// the host computed in fp64 and rounded once to fp32.
//
// Bandwidth-bound: each warp moves one token's K, V (and Q) rows for all heads
// as 16-byte vectors, so the position and table work is shared by the heads
// and the three tensors.  Reads are contiguous per token; every store covers
// whole 256-byte (or 128-byte) cache rows per half-warp.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"

namespace sva {
namespace {

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t rotate_pair_f(float x, float y, float c, float s) {
  const float rx = __fmaf_rn(x, c, -(y * s));
  const float ry = __fmaf_rn(x, s, y * c);
  __nv_bfloat162 r = __floats2bfloat162_rn(rx, ry);  // .x (rx) in the low half
  return *reinterpret_cast<uint32_t*>(&r);
}

// bf16 pair (element 2k in the low half) times g0, g1, then rotated
__device__ __forceinline__ uint32_t norm_rotate_pair(uint32_t xy, float g0, float g1, float c,
                                                     float s) {
  return rotate_pair_f(__uint_as_float(xy << 16) * g0, __uint_as_float(xy & 0xFFFF0000u) * g1, c,
                       s);
}

__device__ __forceinline__ float sumsq8(uint4 v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float a = 0.0f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float x = __uint_as_float(w[k] << 16), y = __uint_as_float(w[k] & 0xFFFF0000u);
    a = __fmaf_rn(x, x, a);
    a = __fmaf_rn(y, y, a);
  }
  return a;
}

__device__ __forceinline__ uint32_t rotate_pair(uint32_t xy, float c, float s) {
  const float x = __uint_as_float(xy << 16);
  const float y = __uint_as_float(xy & 0xFFFF0000u);
  const float rx = __fmaf_rn(x, c, -(y * s));
  const float ry = __fmaf_rn(x, s, y * c);
  __nv_bfloat162 r = __floats2bfloat162_rn(rx, ry);  // .x (rx) in the low half
  return *reinterpret_cast<uint32_t*>(&r);
}

// One warp per (node, token).  A token's H*d values are contiguous in the
// token-major inputs, so the warp walks them as 16-byte vectors; lane l always
// holds vector l mod (d/8) of a head row, i.e. the same four pairs for every
// head, so its cos/sin come from the tables once per token.
// Instances: with the RMSNorm of K (and Q), and two without it.  kWave
// holds the kernel to 64 registers (loads in batches of two), so four
// 256-thread blocks fit an SM and a launch of one 4680-token node (585
// blocks) runs in a single wave: such a launch is bound by memory latency,
// and occupancy is what hides it.  Larger launches loop over their tokens
// and do better with batches of four at two blocks per SM.
template <bool kNorm, bool kWave>
__global__ void __launch_bounds__(256, kWave ? 4 : 2) rope_kv_kernel(const __grid_constant__ RopeParams p) {
  const int lane = threadIdx.x & 31;
  const int vpr = p.d >> 3;                        // 16-byte vectors per (token, head) row
  const int vshift = (vpr == 16) ? 4 : 3;
  const int c8 = lane & (vpr - 1);
  const int per_tok = p.H * vpr;                   // vectors per token
  const int HpWp = p.Hp * p.Wp;
  const size_t kv_stride = (size_t)p.H * p.Tpad * p.d;  // elements between K and V of a slot
  const __nv_bfloat16* kin = static_cast<const __nv_bfloat16*>(p.k_new);
  const __nv_bfloat16* vin = static_cast<const __nv_bfloat16*>(p.v_new);
  __nv_bfloat16* qio = static_cast<__nv_bfloat16*>(p.q);
  __nv_bfloat16* cache = static_cast<__nv_bfloat16*>(p.cache);
  const int warps_per_block = blockDim.x >> 5;
  const int n_tok = p.n_nodes * p.T;

  for (int tok = blockIdx.x * warps_per_block + (threadIdx.x >> 5); tok < n_tok;
       tok += gridDim.x * warps_per_block) {
    const int node = tok / p.T;
    const int u = tok - node * p.T;
    const int f = u / HpWp;
    const int hw = u - f * HpWp;
    const int hh = hw / p.Wp;
    const int ww = hw - hh * p.Wp;
    const RopeNode nd = p.nodes[node];
    const int tpos = nd.t_base + f;
    float2 cs[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int pi = c8 * 4 + k;  // pair index within the head dimension
      if (pi < p.P0)
        cs[k] = __ldg(p.tab_t + (size_t)tpos * p.P0 + pi);
      else if (pi < p.P0 + p.P1)
        cs[k] = __ldg(p.tab_h + (size_t)hh * p.P1 + (pi - p.P0));
      else
        cs[k] = __ldg(p.tab_w + (size_t)ww * p.P2 + (pi - p.P0 - p.P1));
    }
    const size_t in_tok = (size_t)tok * per_tok * 8;
    const size_t out_slot = ((size_t)nd.slot * 2 * p.H) * p.Tpad;  // row of (slot, K, head 0)
    // RMSNorm scale of the token's K and Q vectors (pass over the row, then a
    // warp reduction); the second pass below reloads the row from L1/L2.
    float rk = 1.0f, rq = 1.0f;
    constexpr bool norm = kNorm;
    if constexpr (norm) {
      float sk = 0.0f, sq = 0.0f;
      for (int v = lane; v < per_tok; v += 32) {
        const size_t off = in_tok + (size_t)v * 8;
        sk += sumsq8(*reinterpret_cast<const uint4*>(kin + off));
        if (qio) sq += sumsq8(*reinterpret_cast<const uint4*>(qio + off));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        sk += __shfl_xor_sync(0xffffffffu, sk, o);
        sq += __shfl_xor_sync(0xffffffffu, sq, o);
      }
      const float inv_n = 1.0f / (float)(per_tok * 8);
      rk = __frsqrt_rn(__fmaf_rn(sk, inv_n, p.norm_eps));
      rq = __frsqrt_rn(__fmaf_rn(sq, inv_n, p.norm_eps));
    }
    // Batches of kBatch vectors per lane: every load of a batch is issued
    // before any of its stores (q is rotated in place, so without the split
    // the compiler keeps each iteration's loads behind the previous stores).
    // The single-wave instance runs four blocks per SM, so half the batch
    // keeps as many bytes in flight per SM as the others' two blocks.
    constexpr int kBatch = kWave ? 2 : 4;
    for (int v0 = lane; v0 < per_tok; v0 += 32 * kBatch) {
      uint4 kv[kBatch], vv[kBatch], qv[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int v = v0 + 32 * j;
        if (v < per_tok) {
          const size_t in_off = in_tok + (size_t)v * 8;
          kv[j] = ld_stream(kin + in_off);
          vv[j] = ld_stream(vin + in_off);
          qv[j] = qio ? *reinterpret_cast<const uint4*>(qio + in_off) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int v = v0 + 32 * j;
        if (v >= per_tok) break;
        const int h = v >> vshift;
        const size_t in_off = in_tok + (size_t)v * 8;
        uint32_t kw[4] = {kv[j].x, kv[j].y, kv[j].z, kv[j].w};
        uint32_t qw[4] = {qv[j].x, qv[j].y, qv[j].z, qv[j].w};
        if constexpr (norm) {
          const float4* gk = reinterpret_cast<const float4*>(p.gamma_k + (size_t)v * 8);
          const float4 gk0 = __ldg(gk), gk1 = __ldg(gk + 1);
          const float gkk[8] = {gk0.x, gk0.y, gk0.z, gk0.w, gk1.x, gk1.y, gk1.z, gk1.w};
#pragma unroll
          for (int k = 0; k < 4; ++k)
            kw[k] = norm_rotate_pair(kw[k], gkk[2 * k] * rk, gkk[2 * k + 1] * rk, cs[k].x, cs[k].y);
          if (qio) {
            const float4* gq = reinterpret_cast<const float4*>(p.gamma_q + (size_t)v * 8);
            const float4 gq0 = __ldg(gq), gq1 = __ldg(gq + 1);
            const float gqq[8] = {gq0.x, gq0.y, gq0.z, gq0.w, gq1.x, gq1.y, gq1.z, gq1.w};
#pragma unroll
            for (int k = 0; k < 4; ++k)
              qw[k] = norm_rotate_pair(qw[k], gqq[2 * k] * rq, gqq[2 * k + 1] * rq, cs[k].x,
                                       cs[k].y);
          }
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            kw[k] = rotate_pair(kw[k], cs[k].x, cs[k].y);
            qw[k] = rotate_pair(qw[k], cs[k].x, cs[k].y);
          }
        }
        __nv_bfloat16* kdst = cache + ((out_slot + (size_t)h * p.Tpad + u) * p.d + c8 * 8);
        *reinterpret_cast<uint4*>(kdst) = make_uint4(kw[0], kw[1], kw[2], kw[3]);
        *reinterpret_cast<uint4*>(kdst + kv_stride) = vv[j];
        if (qio) *reinterpret_cast<uint4*>(qio + in_off) = make_uint4(qw[0], qw[1], qw[2], qw[3]);
      }
    }
  }
}

}  // namespace

cudaError_t launch_rope_kv(const RopeParams& p, int num_sms, cudaStream_t s) {
  const long long blocks = ((long long)p.n_nodes * p.T + 7) / 8;  // one warp per token
  if (p.gamma_k != nullptr)
    rope_kv_kernel<true, false><<<p.grid_blocks, 256, 0, s>>>(p);
  else if (blocks <= 4LL * num_sms)
    rope_kv_kernel<false, true><<<p.grid_blocks, 256, 0, s>>>(p);
  else
    rope_kv_kernel<false, false><<<p.grid_blocks, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace sva
