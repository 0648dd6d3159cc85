// FP8 (e4m3) quantization: the "quantize" stage of the paper's MoE pipeline
// (its host listing quantizes tokens before the dispatch; its Section 4.3 table
// calls the step FP8 quantize), per row or in blocks.
//
// Per row:
// out[r][k] = e4m3(in[r][k] / s_r), s_r = amax_r / 448 (1 for an all-zero row),
// both divisions in fp32, e4m3 rounding to nearest even with saturation at
// +-448. One warp per row, 16-byte loads of 8 bf16 values.
#include <cuda_fp8.h>

#include "common.cuh"

namespace moe {
namespace {

constexpr int Q_WARPS = 8;

__global__ void __launch_bounds__(Q_WARPS * 32) quantize_rows_kernel(
    const uint4* __restrict__ in, long rows, int vpr, uint2* __restrict__ out,
    float* __restrict__ scale) {
  const int lane = threadIdx.x % 32;
  const long r = (long)blockIdx.x * Q_WARPS + threadIdx.x / 32;
  if (r >= rows) return;  // uniform per warp
  const uint4* src = in + r * vpr;
  float amax = 0.f;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 x = src[v];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
#pragma unroll
    for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(bf16_bits_to_float(h[i])));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float s = amax > 0.f ? amax / 448.0f : 1.0f;
  if (lane == 0) scale[r] = s;
  uint2* dst = out + r * vpr;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 x = src[v];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
    uint8_t q[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      q[i] = __nv_cvt_float_to_fp8(bf16_bits_to_float(h[i]) / s, __NV_SATFINITE, __NV_E4M3);
    dst[v] = *reinterpret_cast<const uint2*>(q);
  }
}

// The same for the packed rows of experts [e_begin, e_end) with the e4m3 rows
// written in the tile-packed layout (TiledRow: rows of K / 16 chunks); the
// scales stay indexed by packed row. One warp per row; the row's expert is
// the last e with offsets[e] <= r.
__global__ void __launch_bounds__(Q_WARPS * 32) quantize_rows_tiled_kernel(
    const uint4* __restrict__ in, int vpr, const int32_t* __restrict__ offsets, int e_begin,
    int e_end, int tile, uint2* __restrict__ out, float* __restrict__ scale) {
  const int lane = threadIdx.x % 32;
  const long r = (long)offsets[e_begin] + (long)blockIdx.x * Q_WARPS + threadIdx.x / 32;
  if (r >= offsets[e_end]) return;  // uniform per warp
  int lo = e_begin, hi = e_end - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (offsets[mid] <= r) lo = mid;
    else hi = mid - 1;
  }
  const TiledRow w = tiled_row((int)r, lo, offsets[lo], offsets[lo + 1] - offsets[lo], tile,
                               vpr / 2);
  const uint4* src = in + r * vpr;
  float amax = 0.f;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 x = src[v];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
#pragma unroll
    for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(bf16_bits_to_float(h[i])));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float s = amax > 0.f ? amax / 448.0f : 1.0f;
  if (lane == 0) scale[r] = s;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 x = src[v];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
    uint8_t q[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      q[i] = __nv_cvt_float_to_fp8(bf16_bits_to_float(h[i]) / s, __NV_SATFINITE, __NV_E4M3);
    // 8 bytes = half of 16-byte chunk v / 2 of the e4m3 row
    out[w.chunk16(v >> 1) * 2 + (v & 1)] = *reinterpret_cast<const uint2*>(q);
  }
}

// Block scales (DeepSeek-V3's fine-grained FP8: 1 x 128 blocks of activation
// rows, 128 x 128 blocks of weights) as UE8M0 exponents: k is the smallest
// integer with amax <= 448 * 2^k, read off amax's fp32 bits (amax = f * 2^p,
// f in [1, 2): k = p - 8, plus 1 when f > 1.75, since 448 = 1.75 * 2^8), 0 for
// an all-zero block, clamped to [-127, 127]. The values are e4m3(v * 2^-k): a
// power-of-two product, exact in fp32, then one rounding.
__device__ __forceinline__ int block_exponent(float amax) {
  const uint32_t b = __float_as_uint(amax);
  const int ef = (int)((b >> 23) & 0xFFu);
  if (ef == 0) return (b & 0x7FFFFFu) ? -127 : 0;  // zero; a subnormal amax clamps
  const int k = ef - 127 - 8 + ((b & 0x7FFFFFu) > 0x600000u ? 1 : 0);
  return min(max(k, -127), 127);
}

// 2^-k as an fp32 (k <= 120 for any finite bf16 block, so 127 - k >= 7)
__device__ __forceinline__ float inv_pow2(int k) {
  return __uint_as_float((uint32_t)(127 - min(k, 126)) << 23);
}

__device__ __forceinline__ uint2 quantize8(const uint4& x, float inv) {
  const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
  uint8_t q[8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
    q[i] = __nv_cvt_float_to_fp8(bf16_bits_to_float(h[i]) * inv, __NV_SATFINITE, __NV_E4M3);
  return *reinterpret_cast<const uint2*>(q);
}

__device__ __forceinline__ float amax8(const uint4& x) {
  const uint16_t* h = reinterpret_cast<const uint16_t*>(&x);
  float m = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) m = fmaxf(m, fabsf(bf16_bits_to_float(h[i])));
  return m;
}

// 1 x 128 blocks: one warp per row, each half-warp one block (16 lanes x 8 values).
__global__ void __launch_bounds__(Q_WARPS * 32) quantize_blocks_kernel(
    const uint4* __restrict__ in, long rows, int nblk, uint2* __restrict__ out,
    uint8_t* __restrict__ sf, long sf_ld) {
  const int lane = threadIdx.x % 32, hl = lane & 15;
  const long r = (long)blockIdx.x * Q_WARPS + threadIdx.x / 32;
  if (r >= rows) return;  // uniform per warp
  const uint4* src = in + r * nblk * 16;
  uint2* dst = out + r * nblk * 16;
  for (int b0 = 0; b0 < nblk; b0 += 2) {
    const int b = b0 + (lane >> 4);
    const bool act = b < nblk;  // uniform per half-warp
    const uint4 x = act ? src[b * 16 + hl] : make_uint4(0u, 0u, 0u, 0u);
    float m = amax8(x);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    const int k = block_exponent(m);
    if (act) {
      dst[b * 16 + hl] = quantize8(x, inv_pow2(k));
      if (hl == 0) sf[(size_t)r * sf_ld + b] = (uint8_t)(k + 127);
    }
  }
}

// 128 x 128 blocks: one CTA of 256 threads per block, 8 x 16 bytes per thread.
__global__ void __launch_bounds__(256) quantize_weight_blocks_kernel(
    const uint4* __restrict__ in, int vpr, uint2* __restrict__ out, uint8_t* __restrict__ sf) {
  __shared__ float red[8];
  const int cb = blockIdx.x, rb = blockIdx.y;
  uint4 v[8];
  size_t at[8];
  float m = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int i = threadIdx.x + 256 * j;  // row i / 16 of the block, 16-byte column i % 16
    at[j] = (size_t)(rb * 128 + (i >> 4)) * vpr + cb * 16 + (i & 15);
    v[j] = in[at[j]];
    m = fmaxf(m, amax8(v[j]));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (threadIdx.x % 32 == 0) red[threadIdx.x / 32] = m;
  __syncthreads();
#pragma unroll
  for (int w = 0; w < 8; ++w) m = fmaxf(m, red[w]);
  const int k = block_exponent(m);
  const float inv = inv_pow2(k);
#pragma unroll
  for (int j = 0; j < 8; ++j) out[at[j]] = quantize8(v[j], inv);
  if (threadIdx.x == 0) sf[(size_t)rb * gridDim.x + cb] = (uint8_t)(k + 127);
}

}  // namespace

moe_status launch_quantize_blocks(const uint16_t* in, long rows, int K, uint8_t* out, uint8_t* sf,
                                  long sf_ld, cudaStream_t s) {
  if (rows == 0) return MOE_OK;
  const long blocks = (rows + Q_WARPS - 1) / Q_WARPS;
  quantize_blocks_kernel<<<(unsigned)blocks, Q_WARPS * 32, 0, s>>>(
      reinterpret_cast<const uint4*>(in), rows, K / 128, reinterpret_cast<uint2*>(out), sf, sf_ld);
  note_launch();
  return launch_status();
}

moe_status launch_quantize_weight_blocks(const uint16_t* in, long rows, int K, uint8_t* out,
                                         uint8_t* sf, cudaStream_t s) {
  if (rows == 0) return MOE_OK;
  quantize_weight_blocks_kernel<<<dim3((unsigned)(K / 128), (unsigned)(rows / 128)), 256, 0, s>>>(
      reinterpret_cast<const uint4*>(in), K / 8, reinterpret_cast<uint2*>(out), sf);
  note_launch();
  return launch_status();
}

moe_status launch_quantize_rows(const uint16_t* in, long rows, int K, uint8_t* out, float* scale,
                                cudaStream_t s, const int32_t* offsets, int e_begin, int e_end,
                                int tile) {
  if (rows == 0) return MOE_OK;
  const long blocks = (rows + Q_WARPS - 1) / Q_WARPS;
  if (tile > 0) {
    if (e_end <= e_begin) return MOE_OK;
    quantize_rows_tiled_kernel<<<(unsigned)blocks, Q_WARPS * 32, 0, s>>>(
        reinterpret_cast<const uint4*>(in), K / 8, offsets, e_begin, e_end, tile,
        reinterpret_cast<uint2*>(out), scale);
    note_launch();
    return launch_status();
  }
  quantize_rows_kernel<<<(unsigned)blocks, Q_WARPS * 32, 0, s>>>(
      reinterpret_cast<const uint4*>(in), rows, K / 8, reinterpret_cast<uint2*>(out), scale);
  note_launch();
  return launch_status();
}

}  // namespace moe
