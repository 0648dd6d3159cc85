// C ABI of the MoE layer forward: host-side validation, workspace layout,
// entry points and the stage orchestration (sequential or two-stream
// pipelined), in the stage order of the paper's MoE pipeline (host MoE
// listing, Appendix "Static Analysis Example"; two-stream dispatch hiding,
// Section 4.3).
#include <atomic>
#include <cmath>
#include <mutex>
#include <vector>

#include "common.cuh"

// The device error word: latched by kernels whose bounded waits expire.
__device__ int g_moe_device_error = 0;

namespace moe {
namespace {

constexpr int MAX_DEVICES = 64;
std::atomic<uint64_t> g_launches{0};
std::mutex g_mu;
int* g_err_addr[MAX_DEVICES] = {};
int g_sms[MAX_DEVICES] = {};

struct DeviceStreams {
  cudaStream_t pack = nullptr;
  std::vector<cudaEvent_t> events;
};
DeviceStreams g_streams[MAX_DEVICES];
// Pipelined forwards of one device share its internal events: their host-side
// enqueue is serialised (a wait captures the event's record at the time of the
// wait call, so a later re-record by another call cannot reach back into it).
std::mutex g_pipe_mu[MAX_DEVICES];

int current_device() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= MAX_DEVICES) return 0;
  return d;
}

}  // namespace

void note_launch(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

int* device_error_word() {
  const int d = current_device();
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_err_addr[d]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_moe_device_error) == cudaSuccess) g_err_addr[d] = (int*)p;
  }
  return g_err_addr[d];
}

int num_sms() {
  const int d = current_device();
  if (!g_sms[d]) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, d);
    g_sms[d] = v > 0 ? v : 1;
  }
  return g_sms[d];
}

namespace {

// ---------------------------------------------------------------- validation

bool valid_config(const moe_config* c) {
  if (!c) return false;
  if (c->T < 0 || c->H < 128 || c->H % 128 || c->H > 65536) return false;
  if (c->E < 1 || c->E > 1024 || c->k < 1 || c->k > 32 || c->k > c->E) return false;
  if (c->I < 128 || c->I % 128 || c->I > 65536) return false;
  if (c->I_shared < 0 || (c->I_shared && (c->I_shared < 128 || c->I_shared % 128 ||
                                          c->I_shared > 65536)))
    return false;
  if (c->n_groups < 1 || c->n_groups > 32 || c->E % c->n_groups) return false;
  if (c->topk_groups < 1 || c->topk_groups > c->n_groups) return false;
  if ((long)c->k > (long)c->topk_groups * (c->E / c->n_groups)) return false;
  if (c->gate != MOE_GATE_SOFTMAX && c->gate != MOE_GATE_SIGMOID) return false;
  if (c->normalize != 0 && c->normalize != 1) return false;
  if (!std::isfinite(c->route_scale)) return false;
  if ((long long)c->T * c->k > (1LL << 30)) return false;
  return true;
}

bool valid_exec(const moe_exec* ex, const moe_config* c) {
  if (!ex) return false;
  if (ex->overlap != 0 && ex->overlap != 1) return false;
  if (ex->out_fp32 != 0 && ex->out_fp32 != 1) return false;
  if (ex->fuse_gather < 0 || ex->fuse_gather > 2) return false;
  if (ex->fp8 < 0 || ex->fp8 > 2) return false;
  if (ex->fuse_combine != 0 && ex->fuse_combine != 1) return false;
  if (ex->unit_trace_cap < 0 || (ex->unit_trace && ex->unit_trace_cap == 0)) return false;
  if (ex->unit_trace_gemm < 0 || ex->unit_trace_gemm > 2) return false;
  if (ex->n_pipe_events < 0 || (ex->pipe_events && ex->n_pipe_events == 0)) return false;
  if (ex->overlap) {
    if (ex->chunk_axis == 0) {
      if (ex->chunk_tokens < 1) return false;
    } else if (ex->chunk_axis == 1) {
      if (ex->n_expert_chunks < 1 || ex->n_expert_chunks > c->E) return false;
    } else {
      return false;
    }
  }
  return true;
}

// ---------------------------------------------------------------- workspace layout

struct Carver {
  uint8_t* base;
  size_t off = 0;
  explicit Carver(void* b) : base((uint8_t*)b) {}
  template <class T>
  T* take(size_t count) {
    off = align_up(off, 256);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

struct Layout {
  int chunk_T = 0, n_chunks = 1, perm_chunks = 0;
  float* logits;
  int32_t* idx;
  float* w;
  int32_t* counts;   // [n_chunks][E]
  int32_t* offsets;  // [n_chunks][E+1]
  int32_t* rst;      // [T*k]
  int32_t* slot_row; // [T*k]
  int32_t* perm_counts;
  int32_t* perm_base;
  void* router_ws;   // router scratch (planes + partials), sized for one chunk
  bool fp8 = false;
  bool fp8_block = false;  // block scales (fp8 = 2) instead of row scales (fp8 = 1)
  uint8_t* x_q;      // [T, H] e4m3 (fp8 only)
  float* x_s;        // [T] row scales of x_q
  uint8_t* x_sf;     // [T][H/128] block exponents of x_q (block form)
  void* x_perm;      // [T*k, H] bf16, or e4m3 bytes (fp8)
  uint16_t* h;       // [T*k, I]
  uint8_t* hq;       // [T*k, I] e4m3 copy of h (fp8 only)
  float* hs;         // [T*k] its row scales
  uint8_t* hsf;      // [T*k][I/128] its block exponents (block form)
  float* y_perm;     // [T*k, H] fp32
  int32_t* sh_off;   // [2]
  uint16_t* sh_h;    // [T, I_s]
  uint8_t* sh_hq;    // [T, I_s] (fp8 only)
  float* sh_hs;      // [T]
  uint8_t* sh_hsf;   // [T][I_s/128] (block form)
  float* sh_y;       // [T, H] fp32 (unfused combine)
  // Combine fused into GEMM2: the gate weight of every packed row, and the fp32
  // [T, H] accumulator the GEMM2s reduce into (the caller's output when it is
  // fp32, else carved here and converted to bf16 at the end).
  bool fuse_combine = false;
  float* row_w;      // [T*k]
  float* acc;        // [T, H] or null (= the fp32 output)
  // The expert GEMMs' dynamic unit scheduler (two ints): zeroed at the start
  // of each forward; every launch leaves it at 0 (all of a forward's expert
  // GEMMs run in order on the caller's stream). Followed by the dispatch fused
  // into GEMM1 (pack_in_gemm): its chunk counter and per-expert packed-row
  // counts, zeroed with it and likewise left at 0 by each launch.
  int32_t* sched;
  bool pack_in_gemm = false;
  // Without token chunks, bf16 or row-scaled e4m3: x_perm and GEMM2's operand
  // (bf16 h, or e4m3 hq; and the shared expert's) in the tile-packed row
  // layout of the expert GEMMs' token tile (TiledRow), each with 16 padding
  // rows per expert; 0 = row-major
  int tile = 0;
  int32_t* pack_next;   // sched + 2
  int32_t* pack_ready;  // sched + 3, [E]
  size_t bytes = 0;
};

Layout carve(const moe_config& c, const moe_exec& ex, void* ws) {
  Layout L;
  const size_t T = c.T, E = c.E, k = c.k;
  L.chunk_T = c.T;
  if (ex.overlap && ex.chunk_axis == 0) L.chunk_T = c.T < ex.chunk_tokens ? c.T : ex.chunk_tokens;
  if (L.chunk_T < 1) L.chunk_T = 1;
  L.n_chunks = (ex.overlap && ex.chunk_axis == 0) ? (c.T + L.chunk_T - 1) / L.chunk_T : 1;
  if (L.n_chunks < 1) L.n_chunks = 1;
  moe_config cc = c;
  cc.T = L.chunk_T;
  L.perm_chunks = perm_num_chunks(L.chunk_T);
  Carver cv(ws);
  L.logits = cv.take<float>(T * E);
  L.idx = cv.take<int32_t>(T * k);
  L.w = cv.take<float>(T * k);
  L.counts = cv.take<int32_t>((size_t)L.n_chunks * E);
  L.offsets = cv.take<int32_t>((size_t)L.n_chunks * (E + 1));
  L.rst = cv.take<int32_t>(T * k);
  L.slot_row = cv.take<int32_t>(T * k);
  L.perm_counts = cv.take<int32_t>((size_t)(L.perm_chunks + 1) * E);
  L.perm_base = cv.take<int32_t>((size_t)(L.perm_chunks + 1) * E);
  const size_t rws = router_workspace_bytes(cc);
  L.router_ws = rws ? static_cast<void*>(cv.take<uint8_t>(rws)) : nullptr;
  // The fused dispatch (GEMM1 gathering rows with TMA gather4) pays one gather
  // instruction per four token rows per k-block: a win for decode-sized tiles,
  // measured 1.8x slower GEMM1 at ~128 rows per expert. It is used when a
  // chunk averages at most 24 rows per expert.
  const bool fuse = ex.fuse_gather && (long)L.chunk_T * c.k <= 24L * c.E;
  L.fp8 = ex.fp8 != 0;
  L.fp8_block = ex.fp8 == 2;
  const bool rows_fp8 = L.fp8 && !L.fp8_block;
  const size_t xb = L.fp8 ? 1 : 2;  // bytes per activation element
  L.tile = (!L.fp8_block && L.n_chunks == 1) ? ffn_tile_rows((long)T * k, c.E, L.fp8, false)
                                               : 0;
  const size_t pad = L.tile ? 16 * E : 0;  // padding rows of the tile-packed buffers
  L.x_q = L.fp8 ? cv.take<uint8_t>(T * c.H) : nullptr;
  L.x_s = rows_fp8 ? cv.take<float>(T) : nullptr;
  L.x_sf = L.fp8_block ? cv.take<uint8_t>((size_t)(c.H / 128) * T) : nullptr;
  L.x_perm = fuse ? nullptr : static_cast<void*>(cv.take<uint8_t>((T * k + pad) * c.H * xb));
  L.h = cv.take<uint16_t>((T * k + (L.fp8 ? 0 : pad)) * c.I);
  L.hq = L.fp8 ? cv.take<uint8_t>((T * k + pad) * c.I) : nullptr;
  L.hs = rows_fp8 ? cv.take<float>(T * k) : nullptr;
  L.hsf = L.fp8_block ? cv.take<uint8_t>((size_t)(c.I / 128) * T * k) : nullptr;
  L.fuse_combine = ex.fuse_combine != 0;
  L.row_w = L.fuse_combine ? cv.take<float>(T * k) : nullptr;
  L.y_perm = L.fuse_combine ? nullptr : cv.take<float>(T * k * c.H);
  L.acc = (L.fuse_combine && !ex.out_fp32) ? cv.take<float>(T * c.H) : nullptr;
  L.sh_off = cv.take<int32_t>(2);
  const size_t sh_pad = L.tile ? 16 : 0;
  L.sh_h = c.I_shared ? cv.take<uint16_t>((T + (L.fp8 ? 0 : sh_pad)) * c.I_shared) : nullptr;
  L.sh_hq = (c.I_shared && L.fp8) ? cv.take<uint8_t>((T + sh_pad) * c.I_shared) : nullptr;
  L.sh_hs = (c.I_shared && rows_fp8) ? cv.take<float>(T) : nullptr;
  L.sh_hsf = (c.I_shared && L.fp8_block) ? cv.take<uint8_t>((size_t)(c.I_shared / 128) * T)
                                         : nullptr;
  L.sh_y = (c.I_shared && !L.fuse_combine) ? cv.take<float>(T * c.H) : nullptr;
  L.sched = cv.take<int32_t>(3 + E);
  L.pack_next = L.sched ? L.sched + 2 : nullptr;
  L.pack_ready = L.sched ? L.sched + 3 : nullptr;
  L.pack_in_gemm = ex.fuse_gather == 2 && !ex.overlap && ex.fp8 != 2;
  L.bytes = align_up(cv.off, 256);
  return L;
}

cudaStream_t pack_stream(int d) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_streams[d].pack) {
    int lo = 0, hi = 0;
    cudaDeviceGetStreamPriorityRange(&lo, &hi);
    cudaStreamCreateWithPriority(&g_streams[d].pack, cudaStreamNonBlocking, hi);
  }
  return g_streams[d].pack;
}

bool events(int d, size_t n, std::vector<cudaEvent_t>* out) {
  std::lock_guard<std::mutex> lk(g_mu);
  auto& ev = g_streams[d].events;
  while (ev.size() < n) {
    cudaEvent_t e;
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return false;
    ev.push_back(e);
  }
  out->assign(ev.begin(), ev.begin() + n);
  return true;
}

#define MOE_TRY(expr)                 \
  do {                                \
    moe_status _st = (expr);          \
    if (_st != MOE_OK) return _st;    \
  } while (0)

#define MOE_CUDA(expr)                                  \
  do {                                                  \
    if ((expr) != cudaSuccess) return MOE_ERR_CUDA;     \
  } while (0)

// Testing: a simulated failure of a stage call, made on the host (no CUDA call
// fails and nothing runs on the GPU). -1 = off; n >= 0 = the stage calls of
// the forwards that follow pass until n of them have, then the next one
// returns MOE_ERR_CUDA and the injector switches itself off.
std::atomic<int> g_fail_countdown{-1};

moe_status injected_failure() {
  int v = g_fail_countdown.load(std::memory_order_relaxed);
  while (v >= 0) {
    if (g_fail_countdown.compare_exchange_weak(v, v - 1, std::memory_order_relaxed))
      return v == 0 ? MOE_ERR_CUDA : MOE_OK;
  }
  return MOE_OK;
}

// After the pipelined forward forks the pack stream off `stream`, every return
// -- an error part-way through included -- joins it back: `stream` then waits
// for all the work this call put on the pack stream, so none of it can still
// be writing the caller's workspace once the caller's stream moves on, and a
// forward captured into a CUDA graph always leaves the fork joined.
struct JoinOnExit {
  cudaStream_t stream, ps;
  cudaEvent_t ev;
  ~JoinOnExit() {
    if (cudaEventRecord(ev, ps) == cudaSuccess) cudaStreamWaitEvent(stream, ev, 0);
  }
};

// Router + gate + permutation (+ packing) of tokens [t0, t0+Tc) into chunk slot `ci`.
// Records stage event i of a traced forward (no-op without tracing).
moe_status mark(cudaEvent_t* ev, int i, cudaStream_t s) {
  if (ev && ev[i] && cudaEventRecord(ev[i], s) != cudaSuccess) return MOE_ERR_CUDA;
  return MOE_OK;
}

// FP8: rows [t0, t0+Tc) of x -> e4m3 rows of x_q and their scales (per row,
// or per 1 x 128 block: exponents x_sf[t * H/128 + kb]).
moe_status quantize_tokens(const moe_config& c, const Layout& L, const uint16_t* x, int t0, int Tc,
                           cudaStream_t s) {
  if (L.fp8_block)
    return launch_quantize_blocks(x + (size_t)t0 * c.H, Tc, c.H, L.x_q + (size_t)t0 * c.H,
                                  L.x_sf + (size_t)t0 * (c.H / 128), c.H / 128, s);
  return launch_quantize_rows(x + (size_t)t0 * c.H, Tc, c.H, L.x_q + (size_t)t0 * c.H, L.x_s + t0,
                              s);
}

// With quantize (FP8 only) the chunk's rows are quantized after the
// permutation, inside the dispatch stage; the pipelined modes quantize all
// rows up front instead (the shared expert reads them on the other stream).
moe_status pack_tokens(const moe_config& c, const Layout& L, const moe_weights& w,
                       const uint16_t* x, int t0, int Tc, int ci, bool pack_rows,
                       cudaStream_t s, cudaEvent_t* ev = nullptr, bool quantize = false) {
  MOE_TRY(injected_failure());
  moe_config cc = c;
  cc.T = Tc;
  const size_t tk = (size_t)t0 * c.k;
  MOE_TRY(launch_router_auto(cc, x + (size_t)t0 * c.H, w.Wr, L.logits + (size_t)t0 * c.E,
                             L.router_ws, s));
  MOE_TRY(mark(ev, MOE_EV_ROUTER, s));
  MOE_TRY(launch_gate(cc, L.logits + (size_t)t0 * c.E, w.bias, L.idx + tk, L.w + tk, s));
  MOE_TRY(mark(ev, MOE_EV_GATE, s));
  MOE_TRY(launch_permutation(cc, L.idx + tk, L.counts + (size_t)ci * c.E,
                             L.offsets + (size_t)ci * (c.E + 1), L.rst + tk, L.slot_row + tk,
                             L.perm_counts, L.perm_base, s, L.w + tk,
                             L.row_w ? L.row_w + tk : nullptr));
  MOE_TRY(mark(ev, MOE_EV_PERMUTE, s));
  if (L.fp8) {
    // quantize, then dispatch the e4m3 rows: a row of H bytes is copied as
    // H / 2 two-byte units by the same copy kernel
    if (quantize) MOE_TRY(quantize_tokens(c, L, x, t0, Tc, s));
    if (pack_rows && L.tile)  // tile-packed e4m3 rows (H bytes: H / 16 chunks)
      MOE_TRY(launch_dispatch_rows(Tc, c.H / 2, c.k,
                                   reinterpret_cast<const uint16_t*>(L.x_q + (size_t)t0 * c.H),
                                   L.slot_row + tk, static_cast<uint16_t*>(L.x_perm), s, L.tile,
                                   L.idx + tk, L.offsets));
    else if (pack_rows)
      MOE_TRY(launch_dispatch_rows(Tc, c.H / 2, c.k,
                                   reinterpret_cast<const uint16_t*>(L.x_q + (size_t)t0 * c.H),
                                   L.slot_row + tk,
                                   static_cast<uint16_t*>(L.x_perm) + tk * c.H / 2, s));
  } else if (pack_rows && L.tile) {  // tile-packed x_perm
    MOE_TRY(launch_dispatch_rows(Tc, c.H, c.k, x + (size_t)t0 * c.H, L.slot_row + tk,
                                 static_cast<uint16_t*>(L.x_perm), s, L.tile, L.idx + tk,
                                 L.offsets));
  } else if (pack_rows) {
    MOE_TRY(launch_dispatch_rows(Tc, c.H, c.k, x + (size_t)t0 * c.H, L.slot_row + tk,
                                 static_cast<uint16_t*>(L.x_perm) + tk * c.H, s));
  }
  MOE_TRY(mark(ev, MOE_EV_DISPATCH, s));
  return MOE_OK;
}

// Routed experts of chunk ci (tokens [t0, t0+Tc)), experts [e0, e1), then nothing else.
// The routed operand group of tokens [t0, t0+Tc): packed rows of chunk ci, read
// from x_perm or (fused dispatch) gathered from x by row_src_token.
FfnGroup routed_group(const moe_config& c, const Layout& L, const moe_weights& w,
                      const uint16_t* x, int t0, int Tc, int ci, int e0, int e1) {
  const size_t tk = (size_t)t0 * c.k;
  FfnGroup g{};
  g.rows = Tc * c.k;
  g.offsets = L.offsets + (size_t)ci * (c.E + 1);
  g.sched = L.sched;
  g.n_experts = c.E;
  g.e_begin = e0;
  g.e_end = e1;
  g.W13 = w.W13;
  g.W2 = w.W2;
  g.packed = w.packed != 0;
  g.h = L.h + tk * c.I;
  g.h_tiled = L.tile > 0 && !L.fp8;  // (tiled only without token chunks: tk = 0)
  g.hq_tiled = L.tile > 0 && L.fp8;
  g.x_tiled = L.tile > 0 && L.x_perm != nullptr;
  g.x_tile = L.tile;
  if (L.fuse_combine) {  // GEMM2 adds w * y into the token rows of the accumulator
    g.comb_out = L.acc + (size_t)t0 * c.H;
    g.comb_tok = L.rst + tk;
    g.comb_w = L.row_w + tk;
  } else {
    g.y = L.y_perm + tk * c.H;
  }
  const size_t xb = L.fp8 ? 1 : 2;
  if (L.x_perm) {
    g.x = static_cast<const uint8_t*>(L.x_perm) + tk * c.H * xb;
    if (L.pack_in_gemm) {  // GEMM1 writes x_perm itself
      g.pack_src = L.fp8 ? static_cast<const void*>(L.x_q + (size_t)t0 * c.H)
                         : static_cast<const void*>(x + (size_t)t0 * c.H);
      g.pack_rst = L.rst + tk;
      g.pack_src_rows = Tc;
      g.pack_next = L.pack_next;
      g.pack_ready = L.pack_ready + e0;
      g.pack_slot = L.slot_row + tk;  // token-major copy when the shared expert runs first
      g.pack_k = c.k;
    }
  } else {
    g.x = L.fp8 ? static_cast<const void*>(L.x_q + (size_t)t0 * c.H)
                : static_cast<const void*>(x + (size_t)t0 * c.H);
    g.gather = L.rst + tk;
    g.x_rows = Tc;
  }
  if (L.fp8) {
    g.fp8 = true;
    g.x_scale_idx = L.rst + tk;  // the scales are per token, reached through row_src_token
    g.hq = L.hq + tk * c.I;
    if (L.fp8_block) {
      g.fp8_block = true;
      g.x_sf = L.x_sf + (size_t)t0 * (c.H / 128);
      g.x_sf_ld = c.H / 128;
      g.W13_sf = static_cast<const uint8_t*>(w.W13_scale);
      g.W2_sf = static_cast<const uint8_t*>(w.W2_scale);
      g.hsf = L.hsf + tk * (c.I / 128);
      g.h_sf_ld = c.I / 128;
    } else {
      g.x_scale = L.x_s + t0;
      g.W13_scale = static_cast<const float*>(w.W13_scale);
      g.W2_scale = static_cast<const float*>(w.W2_scale);
      g.hs = L.hs + tk;
    }
  }
  return g;
}

// The shared expert as a one-expert group over all T tokens (offsets {0, T}).
FfnGroup dense_group(const moe_config& c, const Layout& L, const moe_weights& w,
                     const uint16_t* x) {
  FfnGroup g{};
  g.offsets = L.sh_off;
  g.sched = L.sched;
  g.rows = c.T;
  g.n_experts = 1;
  g.e_end = 1;
  g.W13 = w.Ws13;
  g.W2 = w.Ws2;
  g.h = L.sh_h;
  g.h_tiled = L.tile > 0 && !L.fp8;
  g.hq_tiled = L.tile > 0 && L.fp8;
  g.y = L.sh_y;
  g.comb_out = L.fuse_combine ? L.acc : nullptr;  // token rows, weight 1
  g.packed = w.packed != 0;
  g.x = x;
  if (L.fp8) {
    g.fp8 = true;
    g.x = L.x_q;
    g.hq = L.sh_hq;
    if (L.fp8_block) {
      g.fp8_block = true;
      g.x_sf = L.x_sf;
      g.x_sf_ld = c.H / 128;
      g.W13_sf = static_cast<const uint8_t*>(w.Ws13_scale);
      g.W2_sf = static_cast<const uint8_t*>(w.Ws2_scale);
      g.hsf = L.sh_hsf;
      g.h_sf_ld = c.I_shared / 128;
    } else {
      g.x_scale = L.x_s;
      g.W13_scale = static_cast<const float*>(w.Ws13_scale);
      g.W2_scale = static_cast<const float*>(w.Ws2_scale);
      g.hs = L.sh_hs;
    }
  }
  return g;
}

moe_status experts_tokens(const moe_config& c, const Layout& L, const moe_weights& w,
                          const uint16_t* x, int t0, int Tc, int ci, int e0, int e1,
                          cudaStream_t s, cudaEvent_t* ev = nullptr,
                          const moe_exec* ex = nullptr) {
  MOE_TRY(injected_failure());
  FfnGroup g = routed_group(c, L, w, x, t0, Tc, ci, e0, e1);
  if (ex && ex->unit_trace) {
    g.trace = ex->unit_trace;
    g.trace_cap = ex->unit_trace_cap;
    g.trace_gemm = ex->unit_trace_gemm == 2 ? 2 : 1;
  }
  const long hint = (long)g.rows * (e1 - e0) / c.E;
  MOE_TRY(launch_expert_ffn_groups(g, nullptr, c.H, c.I, (int)hint, s,
                                   ev ? ev[MOE_EV_GEMM1] : nullptr));
  return mark(ev, MOE_EV_GEMM2, s);
}

moe_status shared_expert(const moe_config& c, const Layout& L, const moe_weights& w,
                         const uint16_t* x, cudaStream_t s, cudaEvent_t* ev = nullptr) {
  if (!c.I_shared) {
    MOE_TRY(mark(ev, MOE_EV_SHARED_GEMM1, s));
    return mark(ev, MOE_EV_SHARED_GEMM2, s);
  }
  MOE_TRY(launch_fill_range(L.sh_off, c.T, s));
  const FfnGroup g = dense_group(c, L, w, x);
  MOE_TRY(launch_expert_ffn_groups(g, nullptr, c.H, c.I_shared, c.T, s,
                                   ev ? ev[MOE_EV_SHARED_GEMM1] : nullptr));
  return mark(ev, MOE_EV_SHARED_GEMM2, s);
}

// Routed experts and the shared expert in one pair of grouped-GEMM launches
// (the shared expert's units share the persistent grid with the routed ones).
// Requires I_shared == I; the stage events then mark the fused GEMMs.
moe_status experts_and_shared(const moe_config& c, const Layout& L, const moe_weights& w,
                              const uint16_t* x, cudaStream_t s, cudaEvent_t* ev,
                              const moe_exec* ex = nullptr) {
  MOE_TRY(launch_fill_range(L.sh_off, c.T, s));
  FfnGroup routed = routed_group(c, L, w, x, 0, c.T, 0, 0, c.E);
  if (ex && ex->unit_trace) {
    routed.trace = ex->unit_trace;
    routed.trace_cap = ex->unit_trace_cap;
    routed.trace_gemm = ex->unit_trace_gemm == 2 ? 2 : 1;
  }
  const FfnGroup dense = dense_group(c, L, w, x);
  MOE_TRY(launch_expert_ffn_groups(routed, &dense, c.H, c.I, routed.rows, s,
                                   ev ? ev[MOE_EV_GEMM1] : nullptr));
  MOE_TRY(mark(ev, MOE_EV_GEMM2, s));
  MOE_TRY(mark(ev, MOE_EV_SHARED_GEMM1, s));
  return mark(ev, MOE_EV_SHARED_GEMM2, s);
}

// Fused combine: the accumulator starts at zero before any GEMM2 adds into it.
moe_status clear_acc(const moe_config& c, const Layout& L, cudaStream_t s) {
  if (!L.fuse_combine) return MOE_OK;
  return cudaMemsetAsync(L.acc, 0, (size_t)c.T * c.H * sizeof(float), s) == cudaSuccess
             ? MOE_OK
             : MOE_ERR_CUDA;
}

// Fused combine, bf16 output: out = bf16(acc) (the combine kernel with no
// routed term and acc as its dense term); with an fp32 output acc is out.
moe_status finish_acc(const moe_config& c, const Layout& L, void* out, int out_fp32,
                      cudaStream_t s) {
  if (out_fp32) return MOE_OK;
  return launch_combine(c.T, c.H, 0, nullptr, nullptr, nullptr, L.acc, out, 0, s);
}

moe_status combine_tokens(const moe_config& c, const Layout& L, int t0, int Tc, void* out,
                          int out_fp32, cudaStream_t s) {
  const size_t tk = (size_t)t0 * c.k;
  const size_t ob = out_fp32 ? 4 : 2;
  return launch_combine(Tc, c.H, c.k, L.y_perm + tk * c.H, L.slot_row + tk, L.w + tk,
                        L.sh_y ? L.sh_y + (size_t)t0 * c.H : nullptr,
                        (uint8_t*)out + (size_t)t0 * c.H * ob, out_fp32, s);
}

}  // namespace
}  // namespace moe

using namespace moe;

extern "C" {

const char* moe_status_string(moe_status s) {
  switch (s) {
    case MOE_OK: return "MOE_OK";
    case MOE_ERR_INVALID_ARG: return "MOE_ERR_INVALID_ARG";
    case MOE_ERR_UNSUPPORTED: return "MOE_ERR_UNSUPPORTED";
    case MOE_ERR_WORKSPACE: return "MOE_ERR_WORKSPACE";
    case MOE_ERR_CUDA: return "MOE_ERR_CUDA";
    case MOE_ERR_TIMEOUT: return "MOE_ERR_TIMEOUT";
    case MOE_ERR_DEVICE_CHECK: return "MOE_ERR_DEVICE_CHECK";
  }
  return "MOE_ERR_UNKNOWN";
}

moe_status moe_validate_config(const moe_config* cfg) {
  return valid_config(cfg) ? MOE_OK : MOE_ERR_INVALID_ARG;
}

size_t moe_workspace_size(const moe_config* cfg, const moe_exec* ex) {
  if (!valid_config(cfg) || !valid_exec(ex, cfg)) return 0;
  return carve(*cfg, *ex, nullptr).bytes;
}

size_t moe_router_workspace_size(const moe_config* cfg) {
  if (!valid_config(cfg)) return 0;
  return router_workspace_bytes(*cfg);
}

size_t moe_dispatch_workspace_size(const moe_config* cfg) {
  if (!valid_config(cfg)) return 0;
  return 2 * align_up((size_t)(perm_num_chunks(cfg->T) + 1) * cfg->E * sizeof(int32_t), 256);
}

size_t moe_expert_ffn_workspace_size(int32_t rows, int32_t I) {
  if (rows < 0 || I < 0) return 0;
  return (size_t)rows * I * 2;
}

moe_status moe_router_logits(const moe_config* cfg, const uint16_t* x, const float* Wr,
                             float* logits, void* ws, size_t ws_bytes, void* stream) {
  if (!valid_config(cfg)) return MOE_ERR_INVALID_ARG;
  if (cfg->T == 0) return MOE_OK;
  if (!x || !Wr || !logits || !aligned16(x) || !aligned16(Wr) || !aligned4(logits))
    return MOE_ERR_INVALID_ARG;
  const size_t need = moe_router_workspace_size(cfg);
  if (ws && need && (ws_bytes < need || !aligned16(ws))) return MOE_ERR_WORKSPACE;
  return launch_router_auto(*cfg, x, Wr, logits, need ? ws : nullptr, (cudaStream_t)stream);
}

moe_status moe_gate_topk(const moe_config* cfg, const float* logits, const float* bias,
                         int32_t* topk_idx, float* topk_w, void* stream) {
  if (!valid_config(cfg)) return MOE_ERR_INVALID_ARG;
  if (cfg->T == 0) return MOE_OK;
  if (!logits || !topk_idx || !topk_w || !aligned4(logits) || !aligned4(topk_idx) ||
      !aligned4(topk_w) || (bias && !aligned4(bias)))
    return MOE_ERR_INVALID_ARG;
  return launch_gate(*cfg, logits, bias, topk_idx, topk_w, (cudaStream_t)stream);
}

moe_status moe_dispatch(const moe_config* cfg, const uint16_t* x, const int32_t* topk_idx,
                        int32_t* counts, int32_t* offsets, int32_t* row_src_token,
                        int32_t* slot_row, uint16_t* x_perm, void* ws, size_t ws_bytes,
                        void* stream) {
  if (!valid_config(cfg)) return MOE_ERR_INVALID_ARG;
  if (!counts || !offsets || !aligned4(counts) || !aligned4(offsets)) return MOE_ERR_INVALID_ARG;
  if (cfg->T > 0 && (!topk_idx || !row_src_token || !slot_row || !aligned4(topk_idx) ||
                     !aligned4(row_src_token) || !aligned4(slot_row)))
    return MOE_ERR_INVALID_ARG;
  if (x_perm && (!x || !aligned16(x) || !aligned16(x_perm))) return MOE_ERR_INVALID_ARG;
  const size_t need = moe_dispatch_workspace_size(cfg);
  if (!ws || ws_bytes < need || ((uintptr_t)ws & 255)) return MOE_ERR_WORKSPACE;
  int32_t* pc = (int32_t*)ws;
  int32_t* pb = (int32_t*)((uint8_t*)ws + need / 2);
  cudaStream_t s = (cudaStream_t)stream;
  MOE_TRY(launch_permutation(*cfg, topk_idx, counts, offsets, row_src_token, slot_row, pc, pb, s));
  if (x_perm) MOE_TRY(launch_dispatch_rows(cfg->T, cfg->H, cfg->k, x, slot_row, x_perm, s));
  return MOE_OK;
}

moe_status moe_pack_weights(int64_t rows, int32_t K, const uint16_t* W, uint16_t* W_packed,
                            void* stream) {
  if (rows < 0 || rows % 128 || K < 64 || K % 64 || K > 65536) return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!W || !W_packed || !aligned16(W) || !aligned16(W_packed)) return MOE_ERR_INVALID_ARG;
  const uint8_t *a = (const uint8_t*)W, *b = (const uint8_t*)W_packed;
  const size_t n = (size_t)rows * K * 2;
  if (a < b + n && b < a + n) return MOE_ERR_INVALID_ARG;  // must not overlap
  return launch_pack_weights(W, W_packed, (long)rows, K, (cudaStream_t)stream);
}

moe_status moe_expert_ffn(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                          const uint16_t* x_perm, const int32_t* offsets, const uint16_t* W13,
                          const uint16_t* W2, float* y_perm, void* ws, size_t ws_bytes,
                          int32_t weights_packed, void* stream) {
  if (weights_packed != 0 && weights_packed != 1) return MOE_ERR_INVALID_ARG;
  if (rows < 0 || H < 128 || H % 128 || H > 65536 || I < 128 || I % 128 || I > 65536 ||
      n_experts < 1 || n_experts > 1024)
    return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!x_perm || !offsets || !W13 || !W2 || !y_perm || !aligned16(x_perm) || !aligned16(W13) ||
      !aligned16(W2) || !aligned16(y_perm) || !aligned4(offsets))
    return MOE_ERR_INVALID_ARG;
  const size_t need = moe_expert_ffn_workspace_size(rows, I);
  if (!ws || ws_bytes < need || !aligned16(ws)) return MOE_ERR_WORKSPACE;
  return launch_expert_ffn(rows, H, I, n_experts, 0, n_experts, x_perm, offsets, W13, W2,
                           (uint16_t*)ws, y_perm, rows, (cudaStream_t)stream, nullptr,
                           weights_packed != 0);
}

size_t moe_expert_ffn_fp8_workspace_size(int32_t rows, int32_t I) {
  if (rows < 0 || I < 0) return 0;
  Carver cv(nullptr);
  cv.take<uint16_t>((size_t)rows * I);
  cv.take<uint8_t>((size_t)rows * I);
  cv.take<float>((size_t)rows);
  return align_up(cv.off, 256);
}

moe_status moe_quantize_fp8(int64_t rows, int32_t K, const uint16_t* in, uint8_t* out,
                            float* scale, void* stream) {
  if (rows < 0 || rows > (1LL << 31) || K < 16 || K % 16 || K > 65536) return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!in || !out || !scale || !aligned16(in) || !aligned16(out) || !aligned4(scale))
    return MOE_ERR_INVALID_ARG;
  const uint8_t *a = (const uint8_t*)in, *b = out;
  if (a < b + (size_t)rows * K && b < a + (size_t)rows * K * 2) return MOE_ERR_INVALID_ARG;
  return launch_quantize_rows(in, (long)rows, K, out, scale, (cudaStream_t)stream);
}

moe_status moe_expert_ffn_fp8(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                              const uint8_t* x_q, const float* x_scale,
                              const int32_t* x_scale_idx, const int32_t* offsets,
                              const uint8_t* W13_q, const float* W13_scale, const uint8_t* W2_q,
                              const float* W2_scale, float* y_perm, void* ws, size_t ws_bytes,
                              void* stream) {
  if (rows < 0 || H < 128 || H % 128 || H > 65536 || I < 128 || I % 128 || I > 65536 ||
      n_experts < 1 || n_experts > 1024)
    return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!x_q || !x_scale || !offsets || !W13_q || !W13_scale || !W2_q || !W2_scale || !y_perm ||
      !aligned16(x_q) || !aligned16(W13_q) || !aligned16(W2_q) || !aligned16(y_perm) ||
      !aligned4(offsets) || !aligned4(x_scale) || !aligned4(W13_scale) || !aligned4(W2_scale) ||
      (x_scale_idx && !aligned4(x_scale_idx)))
    return MOE_ERR_INVALID_ARG;
  if (!ws || ws_bytes < moe_expert_ffn_fp8_workspace_size(rows, I) || ((uintptr_t)ws & 255))
    return MOE_ERR_WORKSPACE;
  Carver cv(ws);
  FfnGroup g{};
  g.x = x_q;
  g.offsets = offsets;
  g.rows = rows;
  g.n_experts = n_experts;
  g.e_end = n_experts;
  g.W13 = W13_q;
  g.W2 = W2_q;
  g.h = cv.take<uint16_t>((size_t)rows * I);
  g.hq = cv.take<uint8_t>((size_t)rows * I);
  g.hs = cv.take<float>((size_t)rows);
  g.y = y_perm;
  g.fp8 = true;
  g.x_scale = x_scale;
  g.x_scale_idx = x_scale_idx;
  g.W13_scale = W13_scale;
  g.W2_scale = W2_scale;
  return launch_expert_ffn_groups(g, nullptr, H, I, rows, (cudaStream_t)stream);
}

size_t moe_expert_ffn_fp8_blocks_workspace_size(int32_t rows, int32_t I) {
  if (rows < 0 || I < 0) return 0;
  Carver cv(nullptr);
  cv.take<uint16_t>((size_t)rows * I);
  cv.take<uint8_t>((size_t)rows * I);
  cv.take<uint8_t>((size_t)(I / 128) * rows);
  return align_up(cv.off, 256);
}

moe_status moe_quantize_fp8_blocks(int64_t rows, int32_t K, const uint16_t* in, uint8_t* out,
                                   uint8_t* sf, int64_t sf_ld, void* stream) {
  if (rows < 0 || rows > (1LL << 31) || K < 128 || K % 128 || K > 65536 || sf_ld < K / 128)
    return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!in || !out || !sf || !aligned16(in) || !aligned16(out)) return MOE_ERR_INVALID_ARG;
  const uint8_t *a = (const uint8_t*)in, *b = out;
  if (a < b + (size_t)rows * K && b < a + (size_t)rows * K * 2) return MOE_ERR_INVALID_ARG;
  return launch_quantize_blocks(in, (long)rows, K, out, sf, (long)sf_ld, (cudaStream_t)stream);
}

moe_status moe_quantize_fp8_weight_blocks(int64_t rows, int32_t K, const uint16_t* in,
                                          uint8_t* out, uint8_t* sf, void* stream) {
  if (rows < 0 || rows % 128 || rows / 128 > 65535 || K < 128 || K % 128 || K > 65536)
    return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!in || !out || !sf || !aligned16(in) || !aligned16(out)) return MOE_ERR_INVALID_ARG;
  const uint8_t *a = (const uint8_t*)in, *b = out;
  if (a < b + (size_t)rows * K && b < a + (size_t)rows * K * 2) return MOE_ERR_INVALID_ARG;
  return launch_quantize_weight_blocks(in, (long)rows, K, out, sf, (cudaStream_t)stream);
}

moe_status moe_expert_ffn_fp8_blocks(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                                     const uint8_t* x_q, const uint8_t* x_sf, int64_t x_sf_ld,
                                     const int32_t* x_scale_idx, const int32_t* offsets,
                                     const uint8_t* W13_q, const uint8_t* W13_sf,
                                     const uint8_t* W2_q, const uint8_t* W2_sf, float* y_perm,
                                     void* ws, size_t ws_bytes, void* stream) {
  if (rows < 0 || H < 128 || H % 128 || H > 65536 || I < 128 || I % 128 || I > 65536 ||
      n_experts < 1 || n_experts > 1024 || x_sf_ld < H / 128)
    return MOE_ERR_INVALID_ARG;
  if (rows == 0) return MOE_OK;
  if (!x_q || !x_sf || !offsets || !W13_q || !W13_sf || !W2_q || !W2_sf || !y_perm ||
      !aligned16(x_q) || !aligned16(W13_q) || !aligned16(W2_q) || !aligned16(y_perm) ||
      !aligned4(offsets) || (x_scale_idx && !aligned4(x_scale_idx)))
    return MOE_ERR_INVALID_ARG;
  if (!ws || ws_bytes < moe_expert_ffn_fp8_blocks_workspace_size(rows, I) ||
      ((uintptr_t)ws & 255))
    return MOE_ERR_WORKSPACE;
  Carver cv(ws);
  FfnGroup g{};
  g.x = x_q;
  g.offsets = offsets;
  g.rows = rows;
  g.n_experts = n_experts;
  g.e_end = n_experts;
  g.W13 = W13_q;
  g.W2 = W2_q;
  g.h = cv.take<uint16_t>((size_t)rows * I);
  g.hq = cv.take<uint8_t>((size_t)rows * I);
  g.hsf = cv.take<uint8_t>((size_t)(I / 128) * rows);
  g.h_sf_ld = I / 128;
  g.y = y_perm;
  g.fp8 = true;
  g.fp8_block = true;
  g.x_sf = x_sf;
  g.x_sf_ld = (long)x_sf_ld;
  g.x_scale_idx = x_scale_idx;
  g.W13_sf = W13_sf;
  g.W2_sf = W2_sf;
  return launch_expert_ffn_groups(g, nullptr, H, I, rows, (cudaStream_t)stream);
}

moe_status moe_testing_expert_ffn_stall(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                                        const uint16_t* x_perm, const int32_t* offsets,
                                        const uint16_t* W13, const uint16_t* W2, float* y_perm,
                                        void* ws, size_t ws_bytes, int64_t stall_fill,
                                        int64_t wait_limit_ns, void* stream) {
  if (rows < 1 || H < 128 || H % 128 || H > 65536 || I < 128 || I % 128 || I > 65536 ||
      n_experts < 1 || n_experts > 1024 || stall_fill < 0 || wait_limit_ns < 1000000 ||
      wait_limit_ns > 2000000000LL)
    return MOE_ERR_INVALID_ARG;
  if (!x_perm || !offsets || !W13 || !W2 || !y_perm || !aligned16(x_perm) || !aligned16(W13) ||
      !aligned16(W2) || !aligned16(y_perm) || !aligned4(offsets))
    return MOE_ERR_INVALID_ARG;
  if (!ws || ws_bytes < moe_expert_ffn_workspace_size(rows, I) || !aligned16(ws))
    return MOE_ERR_WORKSPACE;
  return launch_expert_ffn_stalled(rows, H, I, n_experts, x_perm, offsets, W13, W2,
                                   (uint16_t*)ws, y_perm, (long)stall_fill,
                                   (uint64_t)wait_limit_ns, (cudaStream_t)stream);
}

moe_status moe_combine(const moe_config* cfg, const float* y_perm, const int32_t* slot_row,
                       const float* topk_w, const float* shared_out, void* out,
                       int32_t out_fp32, void* stream) {
  if (!valid_config(cfg) || (out_fp32 != 0 && out_fp32 != 1)) return MOE_ERR_INVALID_ARG;
  if (cfg->T == 0) return MOE_OK;
  if (!y_perm || !slot_row || !topk_w || !out || !aligned16(y_perm) || !aligned4(slot_row) ||
      !aligned4(topk_w) || !aligned16(out) || (shared_out && !aligned16(shared_out)))
    return MOE_ERR_INVALID_ARG;
  return launch_combine(cfg->T, cfg->H, cfg->k, y_perm, slot_row, topk_w, shared_out, out,
                        out_fp32, (cudaStream_t)stream);
}

moe_status moe_layer_forward(const moe_config* cfg, const moe_exec* ex, const moe_weights* w,
                             const uint16_t* x, void* out, const moe_aux* aux, void* ws,
                             size_t ws_bytes, void* stream, void* aux_stream) {
  if (!valid_config(cfg) || !valid_exec(ex, cfg) || !w) return MOE_ERR_INVALID_ARG;
  if (w->packed != 0 && w->packed != 1) return MOE_ERR_INVALID_ARG;
  const moe_config& c = *cfg;
  if (ex->fp8) {  // e4m3 expert weights with row or block scales; no packed form
    if (w->packed) return MOE_ERR_UNSUPPORTED;
    const bool al = ex->fp8 == 2;  // exponent bytes need no alignment
    if (!w->W13_scale || !w->W2_scale || !(al || aligned4(w->W13_scale)) ||
        !(al || aligned4(w->W2_scale)))
      return MOE_ERR_INVALID_ARG;
    if (c.I_shared && (!w->Ws13_scale || !w->Ws2_scale || !(al || aligned4(w->Ws13_scale)) ||
                       !(al || aligned4(w->Ws2_scale))))
      return MOE_ERR_INVALID_ARG;
  }
  if (!w->Wr || !w->W13 || !w->W2 || !aligned16(w->Wr) || !aligned16(w->W13) ||
      !aligned16(w->W2) || (w->bias && !aligned4(w->bias)))
    return MOE_ERR_INVALID_ARG;
  if (c.I_shared && (!w->Ws13 || !w->Ws2 || !aligned16(w->Ws13) || !aligned16(w->Ws2)))
    return MOE_ERR_INVALID_ARG;
  if (!c.I_shared && (w->Ws13 || w->Ws2)) return MOE_ERR_INVALID_ARG;
  if (c.T == 0) return MOE_OK;
  if (!x || !out || !aligned16(x) || !aligned16(out)) return MOE_ERR_INVALID_ARG;
  if (aux && ((aux->logits && !aligned4(aux->logits)) || (aux->topk_idx && !aligned4(aux->topk_idx)) ||
              (aux->topk_w && !aligned4(aux->topk_w)) || (aux->counts && !aligned4(aux->counts))))
    return MOE_ERR_INVALID_ARG;
  Layout L = carve(c, *ex, nullptr);
  if (!ws || ws_bytes < L.bytes || ((uintptr_t)ws & 255)) return MOE_ERR_WORKSPACE;
  L = carve(c, *ex, ws);
  if (L.fuse_combine && ex->out_fp32) L.acc = static_cast<float*>(out);
  if (aux && aux->logits) L.logits = aux->logits;
  if (aux && aux->topk_idx) L.idx = aux->topk_idx;
  if (aux && aux->topk_w) L.w = aux->topk_w;

  cudaStream_t s = (cudaStream_t)stream;
  const int dev = current_device();
  MOE_CUDA(cudaMemsetAsync(L.sched, 0, (3 + (size_t)c.E) * sizeof(int32_t), s));

  if (!ex->overlap) {
    cudaEvent_t* ev = reinterpret_cast<cudaEvent_t*>(ex->stage_events);
    MOE_TRY(mark(ev, MOE_EV_START, s));
    MOE_TRY(clear_acc(c, L, s));
    MOE_TRY(pack_tokens(c, L, *w, x, 0, c.T, 0, L.x_perm != nullptr && !L.pack_in_gemm, s, ev,
                        true));
    if (c.I_shared == c.I) {
      MOE_TRY(experts_and_shared(c, L, *w, x, s, ev, ex));
    } else {
      MOE_TRY(experts_tokens(c, L, *w, x, 0, c.T, 0, 0, c.E, s, ev, ex));
      MOE_TRY(shared_expert(c, L, *w, x, s, ev));
    }
    if (L.fuse_combine)
      MOE_TRY(finish_acc(c, L, out, ex->out_fp32, s));
    else
      MOE_TRY(combine_tokens(c, L, 0, c.T, out, ex->out_fp32, s));
    MOE_TRY(mark(ev, MOE_EV_COMBINE, s));
    if (aux && aux->counts)
      MOE_CUDA(cudaMemcpyAsync(aux->counts, L.counts, sizeof(int32_t) * c.E,
                               cudaMemcpyDeviceToDevice, s));
    return MOE_OK;
  }

  std::lock_guard<std::mutex> pipe_lock(g_pipe_mu[dev]);
  cudaStream_t ps = aux_stream ? (cudaStream_t)aux_stream : pack_stream(dev);
  if (!ps) return MOE_ERR_CUDA;
  const int n_stage = ex->chunk_axis == 0 ? L.n_chunks : ex->n_expert_chunks;
  // the caller's timeline events, recorded in the documented order
  int n_tl = 0;
  auto tl = [&](cudaStream_t st) -> moe_status {
    if (!ex->pipe_events || n_tl >= ex->n_pipe_events) return MOE_OK;
    cudaEvent_t e = static_cast<cudaEvent_t>(ex->pipe_events[n_tl++]);
    return cudaEventRecord(e, st) == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
  };
  std::vector<cudaEvent_t> ev;
  if (!events(dev, (size_t)n_stage + 2, &ev)) return MOE_ERR_CUDA;
  if (L.fp8) MOE_TRY(quantize_tokens(c, L, x, 0, c.T, s));  // before the fork: both streams read x_q
  MOE_TRY(clear_acc(c, L, s));
  // the pack stream starts after everything already queued on `stream`
  MOE_CUDA(cudaEventRecord(ev[n_stage], s));
  MOE_CUDA(cudaStreamWaitEvent(ps, ev[n_stage], 0));
  const JoinOnExit join{s, ps, ev[n_stage + 1]};

  if (ex->chunk_axis == 0) {
    // Token chunks: chunk i+1 is routed and packed on the pack stream while
    // chunk i's experts compute on `stream`.
    for (int ci = 0; ci < L.n_chunks; ++ci) {
      const int t0 = ci * L.chunk_T, Tc = c.T - t0 < L.chunk_T ? c.T - t0 : L.chunk_T;
      MOE_TRY(tl(ps));
      MOE_TRY(pack_tokens(c, L, *w, x, t0, Tc, ci, L.x_perm != nullptr, ps));
      MOE_TRY(tl(ps));
      MOE_CUDA(cudaEventRecord(ev[ci], ps));
    }
    MOE_TRY(tl(s));
    MOE_TRY(shared_expert(c, L, *w, x, s));  // overlaps the first chunk's packing
    MOE_TRY(tl(s));
    for (int ci = 0; ci < L.n_chunks; ++ci) {
      const int t0 = ci * L.chunk_T, Tc = c.T - t0 < L.chunk_T ? c.T - t0 : L.chunk_T;
      MOE_CUDA(cudaStreamWaitEvent(s, ev[ci], 0));
      MOE_TRY(tl(s));
      MOE_TRY(experts_tokens(c, L, *w, x, t0, Tc, ci, 0, c.E, s));
      MOE_TRY(tl(s));
      if (!L.fuse_combine) MOE_TRY(combine_tokens(c, L, t0, Tc, out, ex->out_fp32, s));
    }
    if (L.fuse_combine) MOE_TRY(finish_acc(c, L, out, ex->out_fp32, s));
    if (aux && aux->counts) MOE_TRY(launch_sum_counts(L.counts, L.n_chunks, c.E, aux->counts, s));
    return MOE_OK;
  }

  // Expert ranges: route and permute all tokens once, then pack the rows of
  // expert range i+1 while range i computes; weights are streamed once.
  MOE_TRY(tl(ps));
  MOE_TRY(pack_tokens(c, L, *w, x, 0, c.T, 0, false, ps));
  MOE_TRY(tl(ps));
  const int nr = ex->n_expert_chunks;
  for (int r = 0; r < nr; ++r) {
    const int e0 = (int)((long)c.E * r / nr), e1 = (int)((long)c.E * (r + 1) / nr);
    if (L.x_perm && L.fp8)  // e4m3 rows: H bytes = H / 2 two-byte units
      MOE_TRY(launch_gather_rows(c.H / 2, reinterpret_cast<const uint16_t*>(L.x_q), L.rst,
                                 L.offsets, e0, e1, static_cast<uint16_t*>(L.x_perm), c.T * c.k,
                                 ps, L.tile));
    else if (L.x_perm)  // with a fused dispatch GEMM1 gathers the rows itself
      MOE_TRY(launch_gather_rows(c.H, x, L.rst, L.offsets, e0, e1,
                                 static_cast<uint16_t*>(L.x_perm), c.T * c.k, ps, L.tile));
    MOE_TRY(tl(ps));
    MOE_CUDA(cudaEventRecord(ev[r], ps));
  }
  MOE_TRY(tl(s));
  MOE_TRY(shared_expert(c, L, *w, x, s));  // overlaps routing on the pack stream
  MOE_TRY(tl(s));
  for (int r = 0; r < nr; ++r) {
    const int e0 = (int)((long)c.E * r / nr), e1 = (int)((long)c.E * (r + 1) / nr);
    MOE_CUDA(cudaStreamWaitEvent(s, ev[r], 0));
    MOE_TRY(tl(s));
    MOE_TRY(experts_tokens(c, L, *w, x, 0, c.T, 0, e0, e1, s));
    MOE_TRY(tl(s));
  }
  if (L.fuse_combine)
    MOE_TRY(finish_acc(c, L, out, ex->out_fp32, s));
  else
    MOE_TRY(combine_tokens(c, L, 0, c.T, out, ex->out_fp32, s));
  if (aux && aux->counts)
    MOE_CUDA(cudaMemcpyAsync(aux->counts, L.counts, sizeof(int32_t) * c.E,
                             cudaMemcpyDeviceToDevice, s));
  return MOE_OK;
}

moe_status moe_check_errors(void* stream) {
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return MOE_ERR_CUDA;
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_moe_device_error, sizeof(int)) != cudaSuccess) return MOE_ERR_CUDA;
  if (v != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_moe_device_error, &zero, sizeof(int)) != cudaSuccess)
      return MOE_ERR_CUDA;
  }
  if (v == MOE_ERR_TIMEOUT) return MOE_ERR_TIMEOUT;
  if (v != 0) return MOE_ERR_DEVICE_CHECK;
  return MOE_OK;
}

uint64_t moe_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

moe_status moe_testing_tiled_chunk(int32_t r, int32_t e, int32_t off_e, int32_t cnt_e,
                                   int32_t tile, int32_t chunks_per_row, int32_t c,
                                   int64_t* out) {
  if (!out || e < 0 || off_e < 0 || cnt_e < 1 || r < off_e || r - off_e >= cnt_e || tile < 16 ||
      tile % 16 || chunks_per_row < 8 || chunks_per_row % 8 || c < 0 || c >= chunks_per_row)
    return MOE_ERR_INVALID_ARG;
  *out = (int64_t)tiled_row(r, e, off_e, cnt_e, tile, chunks_per_row).chunk16(c);
  return MOE_OK;
}

moe_status moe_testing_fail_stage(int32_t n) {
  if (n < -1) return MOE_ERR_INVALID_ARG;
  g_fail_countdown.store(n, std::memory_order_relaxed);
  return MOE_OK;
}

void moe_shutdown(void) {
  forget_noalloc_scratch();
  std::lock_guard<std::mutex> lk(g_mu);
  int prev = 0;
  cudaGetDevice(&prev);
  for (int d = 0; d < MAX_DEVICES; ++d) {
    if (!g_streams[d].pack && g_streams[d].events.empty()) continue;
    cudaSetDevice(d);
    if (g_streams[d].pack) cudaStreamDestroy(g_streams[d].pack);
    for (auto e : g_streams[d].events) cudaEventDestroy(e);
    g_streams[d] = DeviceStreams{};
  }
  cudaSetDevice(prev);
}

}  // extern "C"
