// A stack of consecutive MoE layers, and its capture into a CUDA graph.
//
// The paper's multi-layer study (Section 4.3, "Multi-layer scaling") runs
// L = 1..16 consecutive MoE layers and reports the per-layer time. Here layer
// l + 1 reads layer l's bf16 output, optionally RMS-normalized per token (the
// unit-gain form of the RMSNorm in front of a DeepSeek-V3 MoE block: without
// it the outputs of chained bare MoE layers drift away from unit scale and the
// routing of later layers collapses onto a few experts). The activations
// between layers ping-pong between two [T, H] bf16 buffers carved after the
// layer workspace, which all layers share (they run one after another on the
// same stream).
//
// moe_graph_create_stack records the whole stack once, through stream capture
// on a private stream, into an executable CUDA graph: one cudaGraphLaunch then
// replays every kernel, memset, copy and cross-stream event of all L layers
// with the pointers and shapes given at creation.
#include <vector>

#include "common.cuh"

struct moe_graph_s {
  cudaGraphExec_t exec = nullptr;
  uint64_t kernels = 0;  // library kernels per replay
};

namespace {

constexpr int NORM_WARPS = 8;

// x[r] = bf16(x[r] / sqrt(mean(x[r]^2) + 1e-6)) in place, fp32 arithmetic; one
// warp per row, 16-byte vectors of 8 bf16.
__global__ void __launch_bounds__(NORM_WARPS * 32) rms_norm_rows_kernel(uint4* __restrict__ x,
                                                                        long rows, int vpr) {
  const int lane = threadIdx.x % 32;
  const long r = (long)blockIdx.x * NORM_WARPS + threadIdx.x / 32;
  if (r >= rows) return;  // uniform per warp
  uint4* row = x + r * vpr;
  float ss = 0.f;
  for (int v = lane; v < vpr; v += 32) {
    const uint4 q = row[v];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&q);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float f = moe::bf16_bits_to_float(h[i]);
      ss = fmaf(f, f, ss);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = rsqrtf(ss / (float)(vpr * 8) + 1e-6f);
  for (int v = lane; v < vpr; v += 32) {
    uint4 q = row[v];
    uint16_t* h = reinterpret_cast<uint16_t*>(&q);
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = moe::float_to_bf16_bits(moe::bf16_bits_to_float(h[i]) * inv);
    row[v] = q;
  }
}

moe_status rms_norm_rows(uint16_t* x, long rows, int H, cudaStream_t s) {
  if (rows == 0) return MOE_OK;
  rms_norm_rows_kernel<<<(unsigned)((rows + NORM_WARPS - 1) / NORM_WARPS), NORM_WARPS * 32, 0,
                         s>>>(reinterpret_cast<uint4*>(x), rows, H / 8);
  moe::note_launch();
  return moe::launch_status();
}

size_t act_bytes(const moe_config& c) { return moe::align_up((size_t)c.T * c.H * 2, 256); }

bool valid_stack(const moe_config* cfg, const moe_exec* ex, const moe_weights* layers,
                 int32_t n_layers) {
  if (moe_validate_config(cfg) != MOE_OK || !ex || !layers) return false;
  if (n_layers < 1 || n_layers > 4096) return false;
  if (ex->out_fp32 != 0) return false;  // layers chain through bf16 activations
  return moe_workspace_size(cfg, ex) > 0;
}

}  // namespace

extern "C" {

moe_status moe_rms_norm(int64_t rows, int32_t H, const uint16_t* x, uint16_t* out, void* stream) {
  if (rows < 0 || rows > (1LL << 31) || H < 8 || H % 8 || H > 65536) return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!x || !out || !moe::aligned16(x) || !moe::aligned16(out)) return MOE_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (x != out &&
      cudaMemcpyAsync(out, x, (size_t)rows * H * 2, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return MOE_ERR_CUDA;
  return rms_norm_rows(out, rows, H, s);
}

size_t moe_stack_workspace_size(const moe_config* cfg, const moe_exec* ex) {
  if (moe_validate_config(cfg) != MOE_OK || !ex || ex->out_fp32 != 0) return 0;
  const size_t layer = moe_workspace_size(cfg, ex);
  if (layer == 0) return 0;
  return moe::align_up(layer, 256) + 2 * act_bytes(*cfg);
}

moe_status moe_stack_forward(const moe_config* cfg, const moe_exec* ex, const moe_weights* layers,
                             int32_t n_layers, int32_t rms_norm, const uint16_t* x, uint16_t* out,
                             void* ws, size_t ws_bytes, void* stream, void* aux_stream) {
  if (!valid_stack(cfg, ex, layers, n_layers) || (rms_norm != 0 && rms_norm != 1))
    return MOE_ERR_INVALID_ARG;
  if (cfg->T == 0) return MOE_OK;
  if (!x || !out || !moe::aligned16(x) || !moe::aligned16(out)) return MOE_ERR_INVALID_ARG;
  const size_t layer = moe::align_up(moe_workspace_size(cfg, ex), 256);
  if (!ws || ws_bytes < moe_stack_workspace_size(cfg, ex) || ((uintptr_t)ws & 255))
    return MOE_ERR_WORKSPACE;
  uint8_t* base = static_cast<uint8_t*>(ws);
  uint16_t* act[2] = {reinterpret_cast<uint16_t*>(base + layer),
                      reinterpret_cast<uint16_t*>(base + layer + act_bytes(*cfg))};
  const uint16_t* in = x;
  for (int l = 0; l < n_layers; ++l) {
    uint16_t* dst = l == n_layers - 1 ? out : act[l % 2];
    moe_status st = moe_layer_forward(cfg, ex, &layers[l], in, dst, nullptr, base, layer, stream,
                                      aux_stream);
    if (st == MOE_OK && rms_norm && l < n_layers - 1)
      st = rms_norm_rows(dst, cfg->T, cfg->H, static_cast<cudaStream_t>(stream));
    if (st != MOE_OK) return st;
    in = dst;
  }
  return MOE_OK;
}

moe_status moe_graph_create_stack(const moe_config* cfg, const moe_exec* ex,
                                  const moe_weights* layers, int32_t n_layers, int32_t rms_norm,
                                  const uint16_t* x, uint16_t* out, void* ws, size_t ws_bytes,
                                  void* stream, moe_graph* graph) {
  if (!graph) return MOE_ERR_INVALID_ARG;
  *graph = nullptr;
  if (!valid_stack(cfg, ex, layers, n_layers) || (rms_norm != 0 && rms_norm != 1))
    return MOE_ERR_INVALID_ARG;
  if (ex->stage_events) return MOE_ERR_INVALID_ARG;  // tracing events are not replayable
  if (cfg->T > 0 && (!ws || ws_bytes < moe_stack_workspace_size(cfg, ex)))
    return MOE_ERR_WORKSPACE;
  cudaStream_t cs = nullptr;
  if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) return MOE_ERR_CUDA;
  // The private stream starts after the caller's prior work on `stream` (x
  // may still be being written there).
  cudaEvent_t ready = nullptr;
  moe_status st = MOE_OK;
  if (cudaEventCreateWithFlags(&ready, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventRecord(ready, static_cast<cudaStream_t>(stream)) != cudaSuccess ||
      cudaStreamWaitEvent(cs, ready, 0) != cudaSuccess)
    st = MOE_ERR_CUDA;
  // One eager forward first: lazily created internal streams, events and
  // kernel attributes are then in place before the capture.
  if (st == MOE_OK)
    st = moe_stack_forward(cfg, ex, layers, n_layers, rms_norm, x, out, ws, ws_bytes, cs, nullptr);
  if (st == MOE_OK && cudaStreamSynchronize(cs) != cudaSuccess) st = MOE_ERR_CUDA;
  cudaGraph_t g = nullptr;
  const uint64_t k0 = moe_launch_count();
  if (st == MOE_OK) {
    if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
      st = MOE_ERR_CUDA;
    } else {
      st = moe_stack_forward(cfg, ex, layers, n_layers, rms_norm, x, out, ws, ws_bytes, cs,
                             nullptr);
      const cudaError_t e = cudaStreamEndCapture(cs, &g);  // always ends the capture
      if (st == MOE_OK && e != cudaSuccess) st = MOE_ERR_CUDA;
    }
  }
  const uint64_t kernels = moe_launch_count() - k0;
  cudaGraphExec_t exec = nullptr;
  if (st == MOE_OK && cudaGraphInstantiate(&exec, g, 0) != cudaSuccess) st = MOE_ERR_CUDA;
  if (g) cudaGraphDestroy(g);
  if (ready) cudaEventDestroy(ready);
  cudaStreamDestroy(cs);
  cudaGetLastError();  // a failed capture leaves no sticky error behind
  if (st != MOE_OK) {
    if (exec) cudaGraphExecDestroy(exec);
    return st;
  }
  *graph = new moe_graph_s{exec, kernels};
  return MOE_OK;
}

moe_status moe_graph_launch(moe_graph graph, void* stream) {
  if (!graph || !graph->exec) return MOE_ERR_INVALID_ARG;
  if (cudaGraphLaunch(graph->exec, static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MOE_ERR_CUDA;
  moe::note_launch(static_cast<int>(graph->kernels));
  return MOE_OK;
}

uint64_t moe_graph_kernel_count(moe_graph graph) { return graph ? graph->kernels : 0; }

void moe_graph_destroy(moe_graph graph) {
  if (!graph) return;
  if (graph->exec) cudaGraphExecDestroy(graph->exec);
  delete graph;
}

}  // extern "C"
