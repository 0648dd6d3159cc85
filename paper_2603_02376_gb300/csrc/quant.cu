// FP8 (e4m3) row quantization: the "quantize" stage of the paper's MoE pipeline
// (its host listing quantizes tokens before the dispatch; its Section 4.3 table
// calls the step FP8 quantize).
//
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

}  // namespace

moe_status launch_quantize_rows(const uint16_t* in, long rows, int K, uint8_t* out, float* scale,
                                cudaStream_t s) {
  if (rows == 0) return MOE_OK;
  const long blocks = (rows + Q_WARPS - 1) / Q_WARPS;
  quantize_rows_kernel<<<(unsigned)blocks, Q_WARPS * 32, 0, s>>>(
      reinterpret_cast<const uint4*>(in), rows, K / 8, reinterpret_cast<uint2*>(out), scale);
  note_launch();
  return launch_status();
}

}  // namespace moe
