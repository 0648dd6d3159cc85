// Router logits: L[t,e] = sum_h x[t,h] * Wr[e,h] with x bf16, Wr fp32, fp32 accumulation.
//
// The router is the first step of the routed MoE layer (the paper's DeepSeek-V3
// workload routes every token to its experts, Section 4). The router weights
// are fp32, so a plain bf16 tensor-core product would change the logits the
// routing decisions are taken on. Two exact forms are provided:
//  * tensor cores (E a multiple of 128): Wr is split into three bf16 planes
//    whose sum is Wr (split_planes_kernel); each x * plane product is exact in
//    the fp32 TMEM accumulator, so the grouped GEMM (three planes summed into
//    one accumulator) yields fp32-accurate logits; K is split across CTAs and
//    the partials are summed in split order (router_reduce_kernel);
//  * the fp32 SIMT kernel below, for any E.
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

// planes[p * n + i] for p = 0, 1, 2: hi = bf16(w), mid = bf16(w - hi),
// lo = bf16(w - hi - mid). Both differences are exact in fp32, so
// hi + mid + lo carries all 24 significant bits of w (to within 2^-24 |w|).
__global__ void split_planes_kernel(const float* __restrict__ w, size_t n,
                                    uint16_t* __restrict__ planes) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    const float v = w[i];
    const uint16_t hi = float_to_bf16_bits(v);
    const float r1 = v - bf16_bits_to_float(hi);
    const uint16_t mid = float_to_bf16_bits(r1);
    const float r2 = r1 - bf16_bits_to_float(mid);
    planes[i] = hi;
    planes[n + i] = mid;
    planes[2 * n + i] = float_to_bf16_bits(r2);
  }
}

}  // namespace

moe_status launch_split_planes(const float* Wr, size_t n, uint16_t* planes, cudaStream_t s) {
  int blocks = (int)((n + 255) / 256);
  if (blocks > 4 * num_sms()) blocks = 4 * num_sms();
  split_planes_kernel<<<blocks, 256, 0, s>>>(Wr, n, planes);
  note_launch();
  return launch_status();
}

moe_status launch_router_reduce(const float* partials, int splits, size_t n, float* logits,
                                cudaStream_t s) {
  int blocks = (int)((n + 255) / 256);
  if (blocks > 4 * num_sms()) blocks = 4 * num_sms();
  router_reduce_kernel<<<blocks, 256, 0, s>>>(partials, splits, n, logits);
  note_launch();
  return launch_status();
}

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

// Scratch of the router: the three bf16 planes of Wr and the per-split partial
// logits (tensor-core path), or the SIMT split-K partials.
size_t router_workspace_bytes(const moe_config& c) {
  if (c.T <= 0) return 0;
  if (c.E % 128 == 0) {
    const size_t planes = align_up((size_t)3 * c.E * c.H * sizeof(uint16_t), 256);
    return planes + (size_t)router_tc_splits(c.T, c.H, c.E) * c.T * c.E * sizeof(float);
  }
  const int s = router_splits(c);
  return s > 1 ? (size_t)s * c.T * c.E * sizeof(float) : 0;
}

moe_status launch_router_auto(const moe_config& c, const uint16_t* x, const float* Wr,
                              float* logits, void* ws, cudaStream_t s) {
  if (c.T == 0) return MOE_OK;
  if (c.E % 128 == 0 && ws) {
    uint16_t* planes = static_cast<uint16_t*>(ws);
    float* partials = reinterpret_cast<float*>(
        static_cast<uint8_t*>(ws) + align_up((size_t)3 * c.E * c.H * sizeof(uint16_t), 256));
    const int ks = router_tc_splits(c.T, c.H, c.E);
    moe_status st = launch_split_planes(Wr, (size_t)c.E * c.H, planes, s);
    if (st != MOE_OK) return st;
    st = launch_router_tc(c.T, c.H, c.E, x, planes, partials, ks, s);
    if (st != MOE_OK) return st;
    return launch_router_reduce(partials, ks, (size_t)c.T * c.E, logits, s);
  }
  return launch_router(c, x, Wr, logits, static_cast<float*>(ws), ws ? router_splits(c) : 1, s);
}

}  // namespace moe
