// Gate + group-limited top-k: one warp routes one token.
//
// The routing rule is the DeepSeek-V3 one of the layer the paper's MoE
// workload reproduces (Appendix "Workload Details"): sigmoid (or softmax)
// scores, a selection bias, groups scored by the sum of their two best
// selection scores, the top groups kept, the top-k experts picked among them,
// and the unbiased scores of the picked experts normalised and scaled.
//
// Lane l holds experts e = l + 32 i. Every decision is taken on fp32 values;
// ties go to the lower expert (or group) index, and slot j of the output holds
// the j-th best expert, so the result is a deterministic function of the fp32
// logits.
#include <math_constants.h>

#include "common.cuh"

namespace moe {
namespace {

constexpr int GATE_WARPS = 8;

__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

template <int NPL>  // experts per lane = ceil(E / 32)
__global__ void __launch_bounds__(GATE_WARPS * 32) gate_kernel(
    const float* __restrict__ logits, const float* __restrict__ bias, int T, int E, int k, int G,
    int KG, int gate, int normalize, float scale, int32_t* __restrict__ out_idx,
    float* __restrict__ out_w) {
  extern __shared__ float gate_smem[];  // [GATE_WARPS][E] selection scores
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int t = blockIdx.x * GATE_WARPS + warp;
  if (t >= T) return;  // uniform per warp
  float* ssel = gate_smem + (size_t)warp * E;
  const float* L = logits + (size_t)t * E;

  float sc[NPL], sel[NPL];
  float mx = -CUDART_INF_F;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int e = lane + 32 * i;
    sc[i] = e < E ? L[e] : -CUDART_INF_F;
    mx = fmaxf(mx, sc[i]);
  }
  if (gate == MOE_GATE_SOFTMAX) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const int e = lane + 32 * i;
      sc[i] = e < E ? expf(sc[i] - mx) : 0.f;
      sum += sc[i];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
#pragma unroll
    for (int i = 0; i < NPL; ++i) sc[i] = sc[i] / sum;
  } else {
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const int e = lane + 32 * i;
      sc[i] = e < E ? 1.0f / (1.0f + expf(-sc[i])) : 0.f;
    }
  }
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int e = lane + 32 * i;
    if (e < E) {
      sel[i] = bias ? sc[i] + bias[e] : sc[i];
      ssel[e] = sel[i];
    } else {
      sel[i] = -CUDART_INF_F;
    }
  }
  __syncwarp();

  // group limit: lanes g < G score group g, then rank the G groups
  if (G > 1 && KG < G) {
    const int gs = E / G;
    float gscore = -CUDART_INF_F;
    if (lane < G) {
      float b1 = -CUDART_INF_F, b2 = -CUDART_INF_F;
      for (int q = 0; q < gs; ++q) {
        const float v = ssel[lane * gs + q];
        if (v > b1) {
          b2 = b1;
          b1 = v;
        } else if (v > b2) {
          b2 = v;
        }
      }
      gscore = gs > 1 ? b1 + b2 : b1;
    }
    int rank = 0;
    for (int g2 = 0; g2 < G; ++g2) {
      const float o = __shfl_sync(0xffffffffu, gscore, g2);
      if (lane < G && better(o, g2, gscore, lane)) ++rank;
    }
    const unsigned keep = __ballot_sync(0xffffffffu, lane < G && rank < KG);
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const int e = lane + 32 * i;
      if (e < E && !((keep >> (e / gs)) & 1u)) sel[i] = -CUDART_INF_F;
    }
  }

  // top-k by repeated warp argmax; the winner's lane retires it
  int my_idx = 0;
  float my_s = 0.f;
  for (int j = 0; j < k; ++j) {
    float bv = -CUDART_INF_F;
    int be = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const int e = lane + 32 * i;
      if (e < E && better(sel[i], e, bv, be)) {
        bv = sel[i];
        be = e;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oe = __shfl_xor_sync(0xffffffffu, be, o);
      if (better(ov, oe, bv, be)) {
        bv = ov;
        be = oe;
      }
    }
    float s_win = 0.f;
    if (lane == (be & 31)) {
#pragma unroll
      for (int i = 0; i < NPL; ++i) {
        if (lane + 32 * i == be) {
          s_win = sc[i];
          sel[i] = -CUDART_INF_F;
        }
      }
    }
    s_win = __shfl_sync(0xffffffffu, s_win, be & 31);
    if (lane == j) {
      my_idx = be;
      my_s = s_win;
    }
  }

  float w = my_s;
  if (normalize) {
    float tot = 0.f;
    for (int j = 0; j < k; ++j) tot += __shfl_sync(0xffffffffu, my_s, j);
    w = my_s / tot;
  }
  w *= scale;
  if (lane < k) {
    out_idx[(size_t)t * k + lane] = my_idx;
    out_w[(size_t)t * k + lane] = w;
  }
}

template <int NPL>
void launch_gate_t(const moe_config& c, const float* logits, const float* bias, int32_t* idx,
                   float* w, cudaStream_t s) {
  const int blocks = (c.T + GATE_WARPS - 1) / GATE_WARPS;
  const size_t smem = (size_t)GATE_WARPS * c.E * sizeof(float);
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(gate_kernel<NPL>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  gate_kernel<NPL><<<blocks, GATE_WARPS * 32, smem, s>>>(logits, bias, c.T, c.E, c.k, c.n_groups,
                                                         c.topk_groups, c.gate, c.normalize,
                                                         c.route_scale, idx, w);
  note_launch();
}

}  // namespace

moe_status launch_gate(const moe_config& c, const float* logits, const float* bias, int32_t* idx,
                       float* w, cudaStream_t s) {
  if (c.T == 0) return MOE_OK;
  const int npl = (c.E + 31) / 32;
  if (npl <= 1) launch_gate_t<1>(c, logits, bias, idx, w, s);
  else if (npl <= 2) launch_gate_t<2>(c, logits, bias, idx, w, s);
  else if (npl <= 4) launch_gate_t<4>(c, logits, bias, idx, w, s);
  else if (npl <= 8) launch_gate_t<8>(c, logits, bias, idx, w, s);
  else if (npl <= 16) launch_gate_t<16>(c, logits, bias, idx, w, s);
  else launch_gate_t<32>(c, logits, bias, idx, w, s);
  return launch_status();
}

}  // namespace moe
