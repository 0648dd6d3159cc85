// Router logits: L[t,e] = sum_h x[t,h] * Wr[e,h] with x bf16, Wr fp32, fp32 accumulation.
//
// The router is the first step of the routed MoE layer (the paper's DeepSeek-V3
// workload routes every token to its experts, Section 4). Kept on the fp32 SIMT
// pipe: the router weights are fp32, so a bf16 tensor-core product would change
// the logits the routing decisions are taken on.
//
// Tiling: a CTA computes a 64-token x 64-expert tile with 256 threads, each
// owning a 4x4 block of outputs; K is staged 32 at a time through shared memory
// (x converted bf16 -> fp32 on the way in). When the tile grid alone cannot
// fill the GPU (decode batches), K is split across CTAs that write fp32
// partials, summed afterwards in split order by a second kernel, so the result
// is deterministic.
#include "common.cuh"

namespace moe {
namespace {

constexpr int BT = 64;   // tokens per tile
constexpr int BE = 64;   // experts per tile
constexpr int BKR = 32;  // K per stage
constexpr int PAD = 4;   // keeps float4 alignment of shared rows

__global__ void __launch_bounds__(256) router_kernel(const uint16_t* __restrict__ x,
                                                     const float* __restrict__ Wr, int T, int H,
                                                     int E, int k_per_split,
                                                     float* __restrict__ out) {
  __shared__ __align__(16) float xs[BKR][BT + PAD];
  __shared__ __align__(16) float ws[BKR][BE + PAD];

  const int tid = threadIdx.x;
  const int t0 = blockIdx.x * BT;
  const int e0 = blockIdx.y * BE;
  const int kbeg = blockIdx.z * k_per_split;
  const int kend = min(H, kbeg + k_per_split);

  const int ty = tid / 16;  // token quad
  const int tx = tid % 16;  // expert quad
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  // loader coordinates: x tile 64 tokens x 32 k = 256 x (8 bf16); Wr tile 64 x 32 = 512 float4
  const int xl_t = tid / 4, xl_k = (tid % 4) * 8;
  for (int kb = kbeg; kb < kend; kb += BKR) {
    {
      const int t = t0 + xl_t;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (t < T) v = *reinterpret_cast<const uint4*>(x + (size_t)t * H + kb + xl_k);
      const uint16_t* hv = reinterpret_cast<const uint16_t*>(&v);
#pragma unroll
      for (int i = 0; i < 8; ++i) xs[xl_k + i][xl_t] = bf16_bits_to_float(hv[i]);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int idx = tid + r * 256;
      const int e = idx / 8, kk = (idx % 8) * 4;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (e0 + e < E) v = *reinterpret_cast<const float4*>(Wr + (size_t)(e0 + e) * H + kb + kk);
      ws[kk + 0][e] = v.x;
      ws[kk + 1][e] = v.y;
      ws[kk + 2][e] = v.z;
      ws[kk + 3][e] = v.w;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BKR; ++kk) {
      const float4 a = *reinterpret_cast<const float4*>(&xs[kk][ty * 4]);
      const float4 b = *reinterpret_cast<const float4*>(&ws[kk][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w};
      const float bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }

  float* dst = out + (size_t)blockIdx.z * T * E;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int t = t0 + ty * 4 + i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + tx * 4 + j;
      if (e < E) dst[(size_t)t * E + e] = acc[i][j];
    }
  }
}

// logits[i] = sum_{s < splits} partials[s][i], in split order.
__global__ void router_reduce_kernel(const float* __restrict__ partials, int splits, size_t n,
                                     float* __restrict__ logits) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int p = 0; p < splits; ++p) s += partials[(size_t)p * n + i];
    logits[i] = s;
  }
}

}  // namespace

int router_splits(const moe_config& c) {
  if (c.T <= 0) return 1;
  const long tiles = (long)((c.T + BT - 1) / BT) * ((c.E + BE - 1) / BE);
  const long want = 2L * 152;  // about two resident CTAs per SM
  long s = (want + tiles - 1) / tiles;
  const long kmax = c.H / 256;  // at least 256 of K per split
  if (s > kmax) s = kmax;
  if (s < 1) s = 1;
  return (int)s;
}

moe_status launch_router(const moe_config& c, const uint16_t* x, const float* Wr, float* logits,
                         float* partials, int splits, cudaStream_t s) {
  if (c.T == 0) return MOE_OK;
  if (splits < 1 || partials == nullptr) splits = 1;
  int kps = (c.H + splits - 1) / splits;
  kps = (kps + BKR - 1) / BKR * BKR;
  splits = (c.H + kps - 1) / kps;
  dim3 grid((c.T + BT - 1) / BT, (c.E + BE - 1) / BE, splits);
  router_kernel<<<grid, 256, 0, s>>>(x, Wr, c.T, c.H, c.E, kps, splits == 1 ? logits : partials);
  note_launch();
  if (splits > 1) {
    const size_t n = (size_t)c.T * c.E;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 4 * num_sms()) blocks = 4 * num_sms();
    router_reduce_kernel<<<blocks, 256, 0, s>>>(partials, splits, n, logits);
    note_launch();
  }
  return launch_status();
}

}  // namespace moe
