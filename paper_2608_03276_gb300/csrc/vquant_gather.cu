// Eq. 2 (Sec. 3.3) per-token V scale and codes (b = 8: int8; b = 4: two per
// byte), and the order-preserving compaction of kept rows into the compressed
// cache (Sec. 3.1).
//
// Both kernels move 16-byte vectors: a row of d bf16 is d/8 lanes wide, so a
// warp covers 32/(d/8) rows per instruction.  The quantisation rule is the
// IEEE one shared with the oracle: gamma = fp32 round-to-nearest(absmax/qmax),
// code = round-half-even of the fp32 quotient v/gamma, clamped; gamma = 0
// gives code 0.  Divisions use __fdiv_rn so that no reciprocal shortcut or
// fused rounding changes a code.
#include <cuda_bf16.h>

#include "tp_device.cuh"

namespace tp {

namespace {

// One row = LPR lanes x 8 bf16.  Rows are processed UNROLL at a time per
// lane group so that several 16-byte loads are in flight per thread.
template <int LPR, int UNROLL>
__global__ void __launch_bounds__(256) tp_vquant_kernel(const uint4* __restrict__ v,
                                                      void* __restrict__ vq,
                                                      float* __restrict__ gamma, int64_t rows,
                                                      float qmax, int bits) {
  constexpr int RPW = 32 / LPR;  // rows per warp instruction
  const int lane = threadIdx.x & 31;
  const int sub = lane / LPR, part = lane % LPR;
  const int64_t warps_total = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  const int64_t gw = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  for (int64_t base = gw * RPW * UNROLL; base < rows; base += warps_total * RPW * UNROLL) {
    uint4 u[UNROLL];
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
      const int64_t row = base + k * RPW + sub;
      u[k] = row < rows ? __ldcs(v + row * LPR + part) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
      const int64_t row = base + k * RPW + sub;
      float f[8];
      bf16x8_to_f32(u[k], f);
      float a = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) a = fmaxf(a, fabsf(f[i]));
#pragma unroll
      for (int o = LPR / 2; o >= 1; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
      const float g = __fdiv_rn(a, qmax);
      if (row < rows) {
        if (vq) {
          if (bits == 8)
            static_cast<uint2*>(vq)[row * LPR + part] = quant8_packed(u[k], g, qmax);
          else
            static_cast<uint32_t*>(vq)[row * LPR + part] = quant4_packed(u[k], g, qmax);
        }
        if (part == 0) gamma[row] = g;
      }
    }
  }
}

// Compaction: a group of LPR lanes moves one (document, head, slot): lane
// `part` copies the 16-byte part `part` of both the K and the V row and forms
// the int8 codes of its 8 V values, so every lane runs the same code.  Each
// lane keeps UNR slots in flight; idx < 0 marks an unused slot
// (zero-filled).  The cache is written with streaming stores (evict-first in
// L2): nothing here reads it again, and the next layer's scales and key scores
// should find L2 room for the selection.
template <int LPR>
__global__ void __launch_bounds__(256) tp_gather_kernel(const __grid_constant__ GatherParams p) {
  constexpr int SPW = 32 / LPR;  // slots per warp instruction
  constexpr int UNR = 2;
  const int lane = threadIdx.x & 31;
  const int part = lane % LPR;
  const int b = blockIdx.z, h = blockIdx.y;
  const int64_t unit = static_cast<int64_t>(b) * p.n_heads_kv + h;
  const int64_t warp_global = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int64_t t0 = warp_global * SPW * UNR + lane / LPR;
  const uint4* kin = reinterpret_cast<const uint4*>(p.k);
  const uint4* vin = reinterpret_cast<const uint4*>(p.v);
  const int64_t tok0 = static_cast<int64_t>(h) * p.n_total + p.off[b];
  grid_dep_launch();  // the next layer's pass 1 may be scheduled now (it waits before storing)
  grid_dep_wait();    // idx comes from the selection kernel
  int32_t j[UNR];
  uint4 kv[UNR], vv[UNR];
  float g[UNR];
#pragma unroll
  for (int u = 0; u < UNR; ++u) {
    const int64_t t = t0 + u * SPW;
    j[u] = t < p.cap ? p.idx[unit * p.cap + t] : -2;
  }
#pragma unroll
  for (int u = 0; u < UNR; ++u) {
    kv[u] = vv[u] = make_uint4(0, 0, 0, 0);
    g[u] = 0.f;
    if (j[u] >= 0) {
      const int64_t tok = tok0 + j[u];
      kv[u] = __ldcs(kin + tok * LPR + part);
      vv[u] = __ldcs(vin + tok * LPR + part);
      g[u] = p.gamma[tok];
    }
  }
#pragma unroll
  for (int u = 0; u < UNR; ++u) {
    if (j[u] == -2) continue;
    const int64_t slot = unit * p.cap + t0 + u * SPW;
    const int64_t dst = slot * LPR + part;
    if (p.kc) __stcs(reinterpret_cast<uint4*>(p.kc) + dst, kv[u]);
    if (p.vc) __stcs(reinterpret_cast<uint4*>(p.vc) + dst, vv[u]);
    if (p.vqc) {
      if (p.bits == 8)
        __stcs(reinterpret_cast<uint2*>(p.vqc) + dst, j[u] >= 0 ? quant8_packed(vv[u], g[u], p.qmax) : make_uint2(0, 0));
      else
        __stcs(reinterpret_cast<unsigned int*>(p.vqc) + dst, j[u] >= 0 ? quant4_packed(vv[u], g[u], p.qmax) : 0u);
    }
    if (p.gammac && part == 0) __stcs(p.gammac + slot, g[u]);
  }
}

// acc[i] += x[i] over n floats: a guide longer than one scoring block adds
// each later block's key scores to the sum of the blocks before it, in block
// order (both buffers 16-byte aligned; a tail of n mod 4 floats one at a time).
__global__ void __launch_bounds__(256) tp_add_kernel(float* __restrict__ acc,
                                                     const float* __restrict__ x, int64_t n) {
  const int64_t n4 = n >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  float4* a4 = reinterpret_cast<float4*>(acc);
  const float4* x4 = reinterpret_cast<const float4*>(x);
  for (int64_t i = t; i < n4; i += stride) {
    float4 a = a4[i];
    const float4 b = x4[i];
    a.x += b.x;
    a.y += b.y;
    a.z += b.z;
    a.w += b.w;
    a4[i] = a;
  }
  for (int64_t i = (n4 << 2) + t; i < n; i += stride) acc[i] += x[i];
}

}  // namespace

cudaError_t launch_add(float* acc, const float* x, int64_t n, int num_sms, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int threads = 256;
  int64_t blocks = ((n >> 2) + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  tp_add_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(acc, x, n);
  return cudaGetLastError();
}

cudaError_t launch_vquant(const uint16_t* v, void* vq, float* gamma, int64_t rows, int head_dim,
                          float qmax, int bits, int num_sms, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  constexpr int kUnroll = 4;
  const int threads = 256;
  const int lpr = head_dim / 8;
  const int64_t rows_per_block = static_cast<int64_t>(threads / 32) * (32 / lpr) * kUnroll;
  int64_t blocks = (rows + rows_per_block - 1) / rows_per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  const uint4* vv = reinterpret_cast<const uint4*>(v);
  if (head_dim == 128)
    tp_vquant_kernel<16, kUnroll><<<static_cast<unsigned>(blocks), threads, 0, s>>>(vv, vq, gamma, rows, qmax, bits);
  else
    tp_vquant_kernel<8, kUnroll><<<static_cast<unsigned>(blocks), threads, 0, s>>>(vv, vq, gamma, rows, qmax, bits);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherParams& p, bool dependent, cudaStream_t s) {
  if (p.cap <= 0) return cudaSuccess;
  const int threads = 128;  // 2 slots per lane, 128 threads: 25 against 27 us at 128K (4 slots, 256)
  const int lpr = p.head_dim / 8;
  const int64_t slots_per_block = (threads / 32) * (32 / lpr) * 2;
  dim3 grid(static_cast<unsigned>((p.cap + slots_per_block - 1) / slots_per_block), p.n_heads_kv,
            p.batch);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(threads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return p.head_dim == 128 ? cudaLaunchKernelEx(&cfg, tp_gather_kernel<16>, p)
                           : cudaLaunchKernelEx(&cfg, tp_gather_kernel<8>, p);
}

}  // namespace tp
