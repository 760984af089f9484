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
__global__ void __launch_bounds__(256) rope_kv_kernel(const __grid_constant__ RopeParams p) {
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
#pragma unroll 4
    for (int v = lane; v < per_tok; v += 32) {
      const int h = v >> vshift;
      const size_t in_off = in_tok + (size_t)v * 8;
      const uint4 kv = ld_stream(kin + in_off);
      const uint4 vv = ld_stream(vin + in_off);
      uint4 qv = make_uint4(0, 0, 0, 0);
      if (qio) qv = *reinterpret_cast<const uint4*>(qio + in_off);
      uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w};
      uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        kw[k] = rotate_pair(kw[k], cs[k].x, cs[k].y);
        qw[k] = rotate_pair(qw[k], cs[k].x, cs[k].y);
      }
      __nv_bfloat16* kdst = cache + ((out_slot + (size_t)h * p.Tpad + u) * p.d + c8 * 8);
      *reinterpret_cast<uint4*>(kdst) = make_uint4(kw[0], kw[1], kw[2], kw[3]);
      *reinterpret_cast<uint4*>(kdst + kv_stride) = vv;
      if (qio) *reinterpret_cast<uint4*>(qio + in_off) = make_uint4(qw[0], qw[1], qw[2], qw[3]);
    }
  }
}

}  // namespace

cudaError_t launch_rope_kv(const RopeParams& p, cudaStream_t s) {
  rope_kv_kernel<<<p.grid_blocks, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace sva
