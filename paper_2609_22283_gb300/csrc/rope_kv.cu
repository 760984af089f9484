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
// Bandwidth-bound: every thread owns one 16-byte vector (8 bf16, 4 pairs) of
// one (node, token, head) row and moves it for K, V and optionally Q, so the
// position and table work is shared by the three tensors.  Reads walk the
// token-major inputs linearly; each warp writes two whole 256-byte cache rows.
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

__global__ void __launch_bounds__(256) rope_kv_kernel(const __grid_constant__ RopeParams p) {
  const int vpr = p.d >> 3;                        // 16-byte vectors per (token, head) row
  const long long per_node = (long long)p.T * p.H * vpr;
  const long long total = per_node * p.n_nodes;
  const int HpWp = p.Hp * p.Wp;
  const size_t kv_stride = (size_t)p.H * p.Tpad * p.d;  // elements between K and V of a slot
  const __nv_bfloat16* kin = static_cast<const __nv_bfloat16*>(p.k_new);
  const __nv_bfloat16* vin = static_cast<const __nv_bfloat16*>(p.v_new);
  __nv_bfloat16* qio = static_cast<__nv_bfloat16*>(p.q);
  __nv_bfloat16* cache = static_cast<__nv_bfloat16*>(p.cache);

  for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const int node = (int)(idx / per_node);
    const long long rem = idx - (long long)node * per_node;
    const int c8 = (int)(rem % vpr);
    const long long rh = rem / vpr;
    const int h = (int)(rh % p.H);
    const int u = (int)(rh / p.H);
    const int f = u / HpWp;
    const int hw = u - f * HpWp;
    const int hh = hw / p.Wp;
    const int ww = hw - hh * p.Wp;
    const RopeNode nd = p.nodes[node];
    const int tpos = nd.t_base + f;

    const size_t in_off = (size_t)idx * 8;  // inputs are [node][T][H][d]: linear in idx
    const uint4 kv = ld_stream(kin + in_off);
    const uint4 vv = ld_stream(vin + in_off);
    uint4 qv = make_uint4(0, 0, 0, 0);
    if (qio) qv = *reinterpret_cast<const uint4*>(qio + in_off);

    uint32_t kw[4] = {kv.x, kv.y, kv.z, kv.w};
    uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int pi = c8 * 4 + k;  // pair index within the head dimension
      float2 cs;
      if (pi < p.P0) {
        cs = __ldg(p.tab_t + (size_t)tpos * p.P0 + pi);
      } else if (pi < p.P0 + p.P1) {
        cs = __ldg(p.tab_h + (size_t)hh * p.P1 + (pi - p.P0));
      } else {
        cs = __ldg(p.tab_w + (size_t)ww * p.P2 + (pi - p.P0 - p.P1));
      }
      kw[k] = rotate_pair(kw[k], cs.x, cs.y);
      qw[k] = rotate_pair(qw[k], cs.x, cs.y);
    }

    const size_t row = (((size_t)nd.slot * 2) * p.H + h) * p.Tpad + u;
    __nv_bfloat16* kdst = cache + row * p.d + c8 * 8;
    *reinterpret_cast<uint4*>(kdst) = make_uint4(kw[0], kw[1], kw[2], kw[3]);
    *reinterpret_cast<uint4*>(kdst + kv_stride) = vv;
    if (qio) *reinterpret_cast<uint4*>(qio + in_off) = make_uint4(qw[0], qw[1], qw[2], qw[3]);
  }
}

}  // namespace

cudaError_t launch_rope_kv(const RopeParams& p, cudaStream_t s) {
  rope_kv_kernel<<<p.grid_blocks, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace sva
