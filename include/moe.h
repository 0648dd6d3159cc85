/*
 * moe.h -- C ABI of the single-GPU DeepSeek-V3 MoE layer forward (sm_103a).
 *
 * The operation is the MoE layer of the CUCo paper's DeepSeek-V3 workload
 * (Appendix "Workload Details"; host pipeline listing in Appendix "Static
 * Analysis Example"): route tokens to experts, dispatch them into per-expert
 * contiguous buffers, run GEMM1 (gate/up, H -> 2I) + SwiGLU + GEMM2 (down,
 * I -> H) per expert, and combine the expert outputs back into token order
 * with the gate weights. On one GPU the two AlltoAll exchanges of the paper
 * become on-device permutations; the paper's variable-size per-peer transfers
 * become unpadded per-expert row segments, and its "dispatch on a
 * high-priority stream, hidden behind local compute" (Section 4.3) becomes a
 * two-stream chunked pipeline inside one device.
 *
 * Conventions shared by every entry point:
 *  - Tensor pointers are DEVICE pointers owned by the caller, row-major and
 *    contiguous. bf16 tensors are passed as uint16_t bit patterns and must be
 *    16-byte aligned (they are read by 16-byte vector loads and TMA); other
 *    tensors must be 4-byte aligned.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *    stream). Every call only enqueues work on its stream(s): it does not
 *    synchronise, does not allocate device memory and does not abort.
 *  - Arguments are validated on the host before anything is launched; a bad
 *    argument returns MOE_ERR_INVALID_ARG or MOE_ERR_UNSUPPORTED and enqueues
 *    nothing. A failed launch returns MOE_ERR_CUDA.
 *  - Kernels that wait on on-chip barriers give up after a bounded time and
 *    latch MOE_ERR_TIMEOUT in a device error word; moe_check_errors() reads it.
 *  - The library keeps no state between calls except lazily created internal
 *    streams/events and per-device symbol addresses, released by moe_shutdown().
 */
#ifndef MOE_H_
#define MOE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MOE_OK = 0,
  MOE_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad size or knob */
  MOE_ERR_UNSUPPORTED = 2,   /* valid but outside what the kernels implement */
  MOE_ERR_WORKSPACE = 3,     /* workspace missing or smaller than required */
  MOE_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed */
  MOE_ERR_TIMEOUT = 5,       /* a bounded on-device wait expired (latched) */
  MOE_ERR_DEVICE_CHECK = 6   /* an on-device consistency check failed (latched) */
} moe_status;

typedef enum { MOE_GATE_SOFTMAX = 0, MOE_GATE_SIGMOID = 1 } moe_gate;

/*
 * Layer shape and routing rule.
 *  T tokens; H hidden size (multiple of 128); E routed experts (1..1024);
 *  k experts per token (1..32, k <= E); I expert intermediate size (multiple
 *  of 128); I_shared shared-expert intermediate size (0 = none, else a
 *  multiple of 128); n_groups expert groups (1..32, divides E); topk_groups
 *  groups kept (1..n_groups, with k <= topk_groups * E / n_groups); gate a
 *  moe_gate; normalize 1 = renormalise the k weights to sum 1 before scaling;
 *  route_scale final weight multiplier.
 * Routing rule (DeepSeek-V3, the layer the paper's MoE workload reproduces):
 *  sigmoid: s = sigmoid(L), selection score s' = s + bias (fp32); group score =
 *  sum of the two largest s' of the group; keep the top topk_groups groups;
 *  pick the top-k s' among kept experts (ties: lower index); weights = s of
 *  the picked experts (normalised if `normalize`) * route_scale.
 *  softmax: s = softmax(L) over the E experts, otherwise identical.
 */
typedef struct {
  int32_t T, H, E, k, I, I_shared, n_groups, topk_groups, gate, normalize;
  float route_scale;
} moe_config;

/*
 * Execution knobs of moe_layer_forward.
 *  overlap 0 = one stream, stages in order; 1 = two-stream chunked pipeline:
 *    chunk i+1 is routed and dispatched on a high-priority pack stream while
 *    chunk i's experts compute (Section 4.3: dispatch hidden behind compute).
 *  chunk_tokens tokens per chunk when overlap = 1 and chunk_axis = 0.
 *  chunk_axis 0 = chunk by tokens (each chunk re-streams the expert weights);
 *    1 = chunk by expert range within one full-T pass (weights read once):
 *    the rows of expert range i+1 are packed while range i computes.
 *  n_expert_chunks number of expert ranges when chunk_axis = 1.
 *  out_fp32 0 = bf16 output, 1 = fp32 output.
 *  fuse_gather 1 = fuse the dispatch into GEMM1 when a (chunk of the) batch
 *    averages at most 24 rows per expert (decode): GEMM1's operand loads then
 *    gather each expert's token rows straight from x (TMA gather4) and the
 *    packed copy x_perm is never written; larger batches, and 0, pack x_perm
 *    with a dispatch kernel first (one gather instruction per four rows per
 *    k-block costs more than the copy once tiles hold ~128 rows).
 *    2 = the dispatch copy runs inside the GEMM1 launch, at every batch size
 *    (sequential forward, bf16 or row-scaled FP8; otherwise as 0): warps of
 *    GEMM1 write x_perm while the shared expert's units, which read x directly
 *    and come first, compute; each routed expert's token tiles are loaded once
 *    all its rows are written (a bounded wait; on expiry MOE_ERR_TIMEOUT is
 *    latched). With the shared expert in the same launch (I_shared == I) the
 *    copy is token-major, each token row read once for its k packed rows;
 *    otherwise it goes in expert order, so the first experts' tiles can start
 *    early. This is the single-kernel form of the paper's dispatch hidden
 *    behind the layer's own compute (Section 4.3).
 *  fp8 0 = bf16 expert GEMMs; 1 = FP8 (e4m3) expert GEMMs, the quantized
 *    pipeline of the paper's MoE workload (Section 4.3 lists an FP8 quantize
 *    stage before the dispatch): after the gate every token row x[t] is
 *    quantized (moe_quantize_fp8: e4m3 values and one fp32 scale per row), the
 *    dispatch moves the e4m3 rows (half the bytes), GEMM1 and the shared
 *    expert's GEMM1 multiply e4m3 x e4m3 into fp32 and apply both row scales
 *    in the epilogue, h (bf16, as in the bf16 form) is quantized per row the
 *    same way, and GEMM2 runs on e4m3 h and W2. The expert weights of
 *    moe_weights must then be e4m3 with their row scales (fp8 fields there).
 *    2 = FP8 with block scales (DeepSeek-V3's fine-grained form): x and h are
 *    quantized per 1 x 128 block (moe_quantize_fp8_blocks) and the weights
 *    per 128 x 128 block (moe_quantize_fp8_weight_blocks), every scale a
 *    power of two kept as a UE8M0 exponent byte, and the tensor cores apply
 *    the scales inside the MMAs (tcgen05 kind::mxf8f6f4 block_scale, one
 *    scale per 32 products; H, I and I_shared, multiples of 128 in every
 *    valid configuration, hold whole blocks).
 *  fuse_combine 0 = GEMM2 writes y_perm (fp32) and a combine kernel sums each
 *    token's k rows in slot order (deterministic); 1 = the gate-weighted
 *    combine is fused into GEMM2's epilogue: every GEMM2 (and the shared
 *    expert's) adds w * y straight into an fp32 [T,H] accumulator (the output
 *    itself when out_fp32 = 1) with fp32 atomic reductions, so y_perm is never
 *    written; the order of the k + 1 additions per element is not fixed, so
 *    results may differ in the last fp32 bits from run to run.
 */
typedef struct {
  int32_t overlap, chunk_tokens, chunk_axis, n_expert_chunks, out_fp32, fuse_gather;
  /* Optional tracing: an array of MOE_N_STAGE_EVENTS cudaEvent_t (created by
   * the caller) recorded on `stream` at the stage boundaries of a sequential
   * (overlap = 0) forward; NULL = no tracing. Ignored when overlap = 1. */
  void** stage_events;
  int32_t fp8, fuse_combine;
  /* Optional per-unit trace of one grouped GEMM launch (no counterpart in the
   * paper; a profiling aid): a device buffer of unit_trace_cap records of 5
   * uint64, written by a sequential forward for the work units
   * u < unit_trace_cap of GEMM1 (unit_trace_gemm 0 or 1) or GEMM2
   * (unit_trace_gemm 2); the shared expert's units first, then the routed
   * experts' in expert order. Record u: the time the unit was handed to its
   * CTA, the time its first operand stage was ready for the MMAs, the time its
   * accumulator was complete, the time its epilogue had stored it (all
   * %globaltimer nanoseconds), then SM id | token rows << 16 | (expert +
   * 1024 * (1 for the shared expert)) << 32 | feature block << 48 (GEMM1:
   * blocks of 128 features of h; GEMM2: of 256 output features, or 128 when
   * H is not a multiple of 256). Records of units that did not run are left
   * untouched. NULL = off. */
  unsigned long long* unit_trace;
  int32_t unit_trace_cap;
  /* Optional timeline of a pipelined forward (overlap = 1; a profiling aid):
   * n_pipe_events cudaEvent_t created by the caller with timing enabled,
   * recorded at the launch boundaries of both streams in this order (n =
   * number of token chunks or expert ranges): on the pack stream, before and
   * after each chunk's routing + packing (token chunks: 2 per chunk), or
   * before and after the routing, then after each range's gather (expert
   * ranges: 2 + n); then on `stream`, before and after the shared expert, and
   * before and after each chunk's or range's expert GEMMs (2 + 2 n). Events
   * past n_pipe_events are not recorded. NULL = off; ignored when overlap = 0. */
  void** pipe_events;
  int32_t n_pipe_events;
  /* Which GEMM unit_trace records: 0 or 1 = GEMM1, 2 = GEMM2; else
   * MOE_ERR_INVALID_ARG. */
  int32_t unit_trace_gemm;
} moe_exec;

/* Indices into moe_exec.stage_events: event i is recorded when stage i ends
 * (MOE_EV_START before the first kernel). When I_shared == I the shared
 * expert runs inside the routed GEMM launches: its work is then timed in the
 * GEMM1/GEMM2 stages and the SHARED_* stages are empty. */
enum {
  MOE_EV_START = 0,
  MOE_EV_ROUTER = 1,       /* router logits */
  MOE_EV_GATE = 2,         /* gate + group-limited top-k */
  MOE_EV_PERMUTE = 3,      /* histogram, scan, stable permutation */
  MOE_EV_DISPATCH = 4,     /* packing of token rows into expert segments */
  MOE_EV_GEMM1 = 5,        /* routed grouped GEMM1 + SwiGLU */
  MOE_EV_GEMM2 = 6,        /* routed grouped GEMM2 */
  MOE_EV_SHARED_GEMM1 = 7, /* shared expert GEMM1 + SwiGLU (empty when fused) */
  MOE_EV_SHARED_GEMM2 = 8, /* shared expert GEMM2 (empty when fused) */
  MOE_EV_COMBINE = 9,      /* weighted combine (+ shared term) */
  MOE_N_STAGE_EVENTS = 10
};

/* Layer weights (device pointers). Wr [E,H] fp32; bias [E] fp32 or NULL;
 * W13 [E,2I,H] bf16 (rows 0..I-1 gate, I..2I-1 up); W2 [E,H,I] bf16;
 * Ws13 [2*I_shared,H] bf16 and Ws2 [H,I_shared] bf16, NULL iff I_shared = 0.
 * packed 1 = W13, W2, Ws13 and Ws2 are in the tile-packed layout written by
 * moe_pack_weights (same values, same sizes); 0 = row-major as above.
 * With moe_exec.fp8 = 1 the four expert matrices hold e4m3 bytes instead
 * (same shapes, row-major, packed = 0), as written by moe_quantize_fp8 over
 * their rows, and the *_scale arrays hold the fp32 scale of every row:
 * W13_scale [E*2I], W2_scale [E*H], Ws13_scale [2*I_shared], Ws2_scale [H]
 * (the shared ones NULL iff I_shared = 0). With fp8 = 2 the matrices hold
 * e4m3 bytes as written by moe_quantize_fp8_weight_blocks and the *_scale
 * arrays hold uint8 UE8M0 exponents (scale 2^(byte - 127)) of their 128 x 128
 * blocks, row-major [rows / 128][cols / 128]: W13_scale [E*2I/128][H/128],
 * W2_scale [E*H/128][I/128], Ws13_scale [2*I_shared/128][H/128], Ws2_scale
 * [H/128][I_shared/128]. With fp8 = 0 the scales are unused. */
typedef struct {
  const float* Wr;
  const float* bias;
  const void* W13;
  const void* W2;
  const void* Ws13;
  const void* Ws2;
  int32_t packed;
  const void* W13_scale; /* fp8 = 1: const float*; fp8 = 2: const uint8_t* */
  const void* W2_scale;
  const void* Ws13_scale;
  const void* Ws2_scale;
} moe_weights;

/* Optional outputs of moe_layer_forward; NULL fields are skipped.
 * logits [T,E] fp32; topk_idx [T,k] int32; topk_w [T,k] fp32; counts [E] int32. */
typedef struct {
  float* logits;
  int32_t* topk_idx;
  float* topk_w;
  int32_t* counts;
} moe_aux;

/* Human-readable name of a status. Never NULL. */
const char* moe_status_string(moe_status s);

/* Host-only check of a configuration (no CUDA call). MOE_OK if every entry
 * point accepts it. */
moe_status moe_validate_config(const moe_config* cfg);

/* Workspace bytes needed by moe_layer_forward for (cfg, ex); 0 on an invalid
 * configuration. Host-only. */
size_t moe_workspace_size(const moe_config* cfg, const moe_exec* ex);

/* Workspace bytes of moe_router_logits' scratch (may be 0). Host-only. */
size_t moe_router_workspace_size(const moe_config* cfg);

/* Workspace bytes of moe_dispatch's per-chunk histograms. Host-only. */
size_t moe_dispatch_workspace_size(const moe_config* cfg);

/* Workspace bytes of moe_expert_ffn: the SwiGLU activations [rows, I] bf16. */
size_t moe_expert_ffn_workspace_size(int32_t rows, int32_t I);

/* Workspace bytes of moe_expert_ffn_fp8: h [rows, I] bf16, its e4m3 copy
 * [rows, I] and its row scales [rows] fp32, each 256-byte aligned. */
size_t moe_expert_ffn_fp8_workspace_size(int32_t rows, int32_t I);

/*
 * Router logits: logits[t,e] = sum_h x[t,h] * Wr[e,h], fp32-accurate.
 * x [T,H] bf16; Wr [E,H] fp32; logits [T,E] fp32 (written). ws/ws_bytes:
 * scratch of moe_router_workspace_size bytes, 16-byte aligned. With it and E
 * a multiple of 128 the product runs on the tensor cores: Wr is split exactly
 * into three bf16 planes (hi + mid + lo) whose products with the bf16 x are
 * exact and summed in fp32; K is split across CTAs and the partials are added
 * in a fixed order. Otherwise (or with ws NULL) an fp32 SIMT kernel runs. The
 * gating of every routed token starts here (the paper's workload routes each
 * token to its experts, Section 4).
 */
moe_status moe_router_logits(const moe_config* cfg, const uint16_t* x, const float* Wr,
                             float* logits, void* ws, size_t ws_bytes, void* stream);

/*
 * Gate + group-limited top-k (the routing rule of moe_config).
 * logits [T,E] fp32; bias [E] fp32 or NULL (selection only);
 * topk_idx [T,k] int32 (written, slot j in descending selection score);
 * topk_w [T,k] fp32 (written).
 */
moe_status moe_gate_topk(const moe_config* cfg, const float* logits, const float* bias,
                         int32_t* topk_idx, float* topk_w, void* stream);

/*
 * Dispatch: the single-GPU form of the paper's AlltoAll dispatch (host MoE
 * listing; "variable-size per-peer transfers that avoid padding",
 * Appendix "Workload Details"). Computes a stable expert-major permutation of
 * the T*k (token, slot) entries and optionally packs the token rows.
 * topk_idx [T,k] int32 (values in [0,E)); counts [E] (written); offsets [E+1]
 * (written, exclusive prefix sum of counts); row_src_token [T*k] (written:
 * token of each packed row); slot_row [T*k] (written: packed row of entry
 * t*k+j). Rows of one expert are ordered by (t, j). x [T,H] bf16 and x_perm
 * [T*k,H] bf16: x_perm[r] = x[row_src_token[r]]; x_perm NULL = permutation
 * only (x may then be NULL). ws: moe_dispatch_workspace_size bytes.
 */
moe_status moe_dispatch(const moe_config* cfg, const uint16_t* x, const int32_t* topk_idx,
                        int32_t* counts, int32_t* offsets, int32_t* row_src_token,
                        int32_t* slot_row, uint16_t* x_perm, void* ws, size_t ws_bytes,
                        void* stream);

/*
 * moe_dispatch for callers that cannot allocate device memory. (The paper has
 * no counterpart; this is a deployment variant.) Some callers can't call
 * cudaMalloc: plugins inside a host framework that owns all device memory,
 * serving loops whose memory was planned once and must not grow, and
 * latency-critical paths where an allocation may synchronise the device; they
 * may also have no workspace to pass. This call computes exactly what
 * moe_dispatch computes (same arguments, minus the workspace) but keeps the
 * per-chunk histogram scratch in a fixed-size array inside the library
 * (2 x MOE_DISPATCH_NOALLOC_MAX_ENTRIES int32 = 1 MiB per device, held until
 * the process exits). It allocates nothing.
 *  - Size limit: (ceil(T / 128) + 1) * E <= MOE_DISPATCH_NOALLOC_MAX_ENTRIES
 *    (e.g. T <= 65408 tokens at E = 256); larger inputs return
 *    MOE_ERR_UNSUPPORTED and enqueue nothing.
 *  - The first call on each device looks up the array's device address (with
 *    that device current) and caches it; make that first call before any
 *    stream capture.
 *  - All calls on a device share the array, which keeps the previous call's
 *    contents (nothing in it needs to start at zero). Calls whose GPU work
 *    overlaps -- different streams with no ordering between them -- race on it.
 */
#define MOE_DISPATCH_NOALLOC_MAX_ENTRIES 131072
moe_status moe_dispatch_noalloc(const moe_config* cfg, const uint16_t* x, const int32_t* topk_idx,
                                int32_t* counts, int32_t* offsets, int32_t* row_src_token,
                                int32_t* slot_row, uint16_t* x_perm, void* stream);

/*
 * Weight layout for the expert GEMMs (a load-time transform; no counterpart in
 * the paper). Copies W [rows, K] bf16 (row-major; rows a multiple of 128, K a
 * multiple of 64) to W_packed (same size, caller-allocated, not overlapping W)
 * so that every 128-row x 64-column tile the GEMMs load is one contiguous
 * 16 KiB block, already in the 128-byte-swizzled order of the tensor-core
 * operands: tile (r / 128, c / 64) is block (r / 128) * (K / 64) + c / 64, and
 * inside it the 16-byte chunk j = (c % 64) / 8 of row r sits at element
 *   (r % 128) * 64 + 8 * (j ^ (r % 8)) + c % 8.
 * Pack W13 as rows = E*2I, K = H; W2 as rows = E*H, K = I; the shared expert's
 * Ws13 / Ws2 likewise; then set moe_weights.packed (or weights_packed of
 * moe_expert_ffn). The GEMMs then fetch each tile with one bulk copy.
 */
moe_status moe_pack_weights(int64_t rows, int32_t K, const uint16_t* W, uint16_t* W_packed,
                            void* stream);

/*
 * Grouped expert FFN (GEMM1 + SwiGLU + GEMM2 of the paper's expert compute,
 * shapes 7168 x 4096 and 2048 x 7168 in Appendix "Workload Details").
 * For each expert e < n_experts and each row r in [offsets[e], offsets[e+1]):
 *   h[r] = bf16(silu(x_perm[r] . Wg_e^T) * (x_perm[r] . Wu_e^T)),
 *   y_perm[r] = h[r] . W2_e^T             (fp32 accumulation and fp32 y).
 * h is rounded to bf16 because it is GEMM2's tensor-core operand; y stays in
 * fp32 for the combine. rows: rows of x_perm / y_perm; H hidden (multiple of
 * 128); I intermediate (multiple of 128); offsets [n_experts+1] int32 on the
 * device, non-decreasing, offsets[n_experts] <= rows (a violation is clamped
 * and latched as MOE_ERR_DEVICE_CHECK); W13 [n_experts,2I,H] bf16;
 * W2 [n_experts,H,I] bf16; x_perm [rows,H] bf16; y_perm [rows,H] fp32
 * (written; rows outside every segment are left untouched). ws:
 * moe_expert_ffn_workspace_size(rows, I) bytes, 16-byte aligned (receives h).
 * weights_packed 1 = W13 and W2 are tile-packed (moe_pack_weights).
 * The shared expert is this call with n_experts = 1 and offsets = {0, T}.
 */
moe_status moe_expert_ffn(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                          const uint16_t* x_perm, const int32_t* offsets, const uint16_t* W13,
                          const uint16_t* W2, float* y_perm, void* ws, size_t ws_bytes,
                          int32_t weights_packed, void* stream);

/*
 * FP8 row quantization, the paper's "quantize" stage (Section 4.3's FP8
 * quantize before the dispatch; the dequantize is folded into the GEMM
 * epilogues). For each row r of in [rows, K] bf16:
 *   scale[r] = fp32(amax_r / 448)   (1 when the row is all zero),
 *   out[r][c] = e4m3(fp32(in[r][c] / scale[r])),
 * with e4m3 the OCP E4M3 format (bias 7, no infinities, largest finite 448),
 * rounded to nearest even and saturated at +-448. out [rows, K] e4m3 bytes;
 * scale [rows] fp32; both written, caller-allocated. K a multiple of 16 and at
 * most 65536; in and out 16-byte aligned; in and out must not overlap.
 * Used on token rows inside moe_layer_forward (fp8 = 1) and, once, on the
 * expert weights (W13 as rows = E*2I, K = H; W2 as rows = E*H, K = I).
 */
moe_status moe_quantize_fp8(int64_t rows, int32_t K, const uint16_t* in, uint8_t* out,
                            float* scale, void* stream);

/*
 * Grouped expert FFN in the FP8 form (moe_expert_ffn with e4m3 operands).
 * For each expert e < n_experts and row r in [offsets[e], offsets[e+1]):
 *   g|u = (x_q[r] . W13_q[e]^T) * sx(r) * W13_scale[e*2I + j]  (fp32 accumulate),
 *   h[r] = bf16(silu(g) * u),  (h_q, s_h) = moe_quantize_fp8 of h per row,
 *   y_perm[r] = (h_q[r] . W2_q[e]^T) * s_h[r] * W2_scale[e*H + c].
 * sx(r) = x_scale[x_scale_idx[r]] when x_scale_idx is given (x_q rows are
 * copies of token rows, scales kept per token), else x_scale[r].
 * x_q [rows,H] e4m3; W13_q [n_experts,2I,H] and W2_q [n_experts,H,I] e4m3
 * (row-major); offsets, shapes, y_perm and the segment rules as in
 * moe_expert_ffn. ws: moe_expert_ffn_fp8_workspace_size(rows, I) bytes,
 * 256-byte aligned.
 */
moe_status moe_expert_ffn_fp8(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                              const uint8_t* x_q, const float* x_scale,
                              const int32_t* x_scale_idx, const int32_t* offsets,
                              const uint8_t* W13_q, const float* W13_scale, const uint8_t* W2_q,
                              const float* W2_scale, float* y_perm, void* ws, size_t ws_bytes,
                              void* stream);

/*
 * FP8 quantization with block scales: the paper's "quantize" stage (Section
 * 4.3's FP8 quantize before the dispatch) at DeepSeek-V3's fine-grained
 * granularity, with power-of-two (UE8M0) scales the tensor cores apply
 * inside the MMA. For activation rows: each 1 x 128 block
 * of in [rows, K] bf16 gets the exponent k = the smallest integer with
 * amax <= 448 * 2^k (k = 0 for an all-zero block, clamped to [-127, 127]),
 * stored as the UE8M0 byte sf[r * sf_ld + c / 128] = k + 127, and its
 * values out[r][c] = e4m3(in[r][c] * 2^-k) (exact scaling, then round to
 * nearest even, saturating at +-448). K a multiple of 128, at most 65536;
 * sf_ld >= K / 128; in and out 16-byte aligned and not overlapping; all written
 * buffers caller-allocated. Used on token rows and on h inside
 * moe_layer_forward (fp8 = 2).
 */
moe_status moe_quantize_fp8_blocks(int64_t rows, int32_t K, const uint16_t* in, uint8_t* out,
                                   uint8_t* sf, int64_t sf_ld, void* stream);

/*
 * The same in 128 x 128 blocks, for weight matrices viewed as [rows, K]:
 * sf[(r / 128) * (K / 128) + c / 128] = k + 127 of block (r / 128, c / 128).
 * rows a multiple of 128 (at most 128 * 65535), K a multiple of 128 (at most
 * 65536). A load-time step (W13 as rows = E*2I, K = H; W2 as rows = E*H, K = I).
 */
moe_status moe_quantize_fp8_weight_blocks(int64_t rows, int32_t K, const uint16_t* in,
                                          uint8_t* out, uint8_t* sf, void* stream);

/* Workspace bytes of moe_expert_ffn_fp8_blocks: h [rows, I] bf16, its e4m3
 * copy [rows, I] and its block exponents [rows][I/128], each 256-byte aligned. */
size_t moe_expert_ffn_fp8_blocks_workspace_size(int32_t rows, int32_t I);

/*
 * Grouped expert FFN with block-scaled FP8 operands: the expert compute of
 * the paper's MoE workload (GEMM1 up/gate + SwiGLU + GEMM2 down, Appendix
 * "Workload Details") on e4m3 operands, with moe_expert_ffn's segments and
 * shapes. With 2^kx, 2^kw the scales of the blocks a product's terms fall in:
 *   g|u[r][j] = sum_c x_q[r][c] 2^kx(r, c/128) * W13_q[e][j][c] 2^kw13(e, j/128, c/128),
 *   h[r] = bf16(silu(g) * u), h quantized by moe_quantize_fp8_blocks,
 *   y_perm[r][c] = sum_i h_q[r][i] 2^kh(r, i/128) * W2_q[e][c][i] 2^kw2(e, c/128, i/128),
 * fp32 accumulation on the tensor cores. kx(r, b) is x_sf[t * x_sf_ld + b] with
 * t = x_scale_idx[r] when given (x_q rows are copies of token rows, whose
 * exponent rows x_sf holds), else r; x_sf_ld >= H / 128.
 * W13_sf [n_experts*2I/128][H/128], W2_sf [n_experts*H/128][I/128] as in
 * moe_weights (fp8 = 2). H and I multiples of 128. ws:
 * moe_expert_ffn_fp8_blocks_workspace_size(rows, I) bytes, 256-byte aligned.
 */
moe_status moe_expert_ffn_fp8_blocks(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                                     const uint8_t* x_q, const uint8_t* x_sf, int64_t x_sf_ld,
                                     const int32_t* x_scale_idx, const int32_t* offsets,
                                     const uint8_t* W13_q, const uint8_t* W13_sf,
                                     const uint8_t* W2_q, const uint8_t* W2_sf, float* y_perm,
                                     void* ws, size_t ws_bytes, void* stream);

/*
 * Combine: the single-GPU form of the paper's reverse AlltoAll combine.
 * out[t] = sum_j topk_w[t,j] * y_perm[slot_row[t*k+j]] (+ shared_out[t]),
 * fp32 accumulation in slot order j = 0..k-1, then the shared term.
 * y_perm [T*k,H] fp32; slot_row [T*k] (values in [0, T*k); others are
 * skipped and latched as MOE_ERR_DEVICE_CHECK); topk_w [T,k] fp32;
 * shared_out [T,H] fp32 or NULL; out [T,H] bf16 (out_fp32 = 0, round to
 * nearest even) or fp32 (out_fp32 = 1).
 */
moe_status moe_combine(const moe_config* cfg, const float* y_perm, const int32_t* slot_row,
                       const float* topk_w, const float* shared_out, void* out,
                       int32_t out_fp32, void* stream);

/*
 * The whole layer: router -> gate/top-k -> dispatch -> grouped expert FFN
 * (+ shared expert) -> combine, in the paper's stage order.
 * x [T,H] bf16; out [T,H] bf16 or fp32 per ex->out_fp32; aux optional;
 * ws: moe_workspace_size(cfg, ex) bytes. aux_stream: the pack stream of the
 * overlapped pipeline (NULL = an internal high-priority stream); unused when
 * ex->overlap = 0. Passing `stream` itself runs the pipelined stage order on
 * one stream; a caller on the legacy default stream (whose handle is NULL,
 * the same value as "internal") passes cudaStreamLegacy for that. All work is ordered after prior work on `stream`, and later
 * work on `stream` is ordered after the whole layer. Calls from several host
 * threads are safe; pipelined calls on one device share internal events and
 * enqueue one at a time. Concurrent calls must not share a workspace.
 */
moe_status moe_layer_forward(const moe_config* cfg, const moe_exec* ex, const moe_weights* w,
                             const uint16_t* x, void* out, const moe_aux* aux, void* ws,
                             size_t ws_bytes, void* stream, void* aux_stream);

/*
 * A stack of n_layers consecutive MoE layers (the paper's multi-layer study,
 * Section 4.3 "Multi-layer scaling", L = 1..16): layer 0 reads x, layer l + 1
 * reads layer l's output, layer n_layers - 1 writes out. layers[l] holds layer
 * l's weights (layers may share tensors). rms_norm 1: between layers every
 * token row h is replaced by bf16(h / sqrt(mean(h^2) + 1e-6)) (fp32), the
 * unit-gain RMSNorm a DeepSeek-V3 block applies before its MoE; 0: raw chain. x and out [T,H] bf16 (may not
 * overlap each other or ws); ex->out_fp32 must be 0 (the layers chain through
 * bf16 activations); ex->stage_events, if set, are recorded by every layer.
 * ws: moe_stack_workspace_size(cfg, ex) bytes, 256-byte aligned: one layer
 * workspace shared by all layers plus two [T,H] bf16 activation buffers.
 * Ordering on `stream` as for moe_layer_forward.
 */
size_t moe_stack_workspace_size(const moe_config* cfg, const moe_exec* ex);

/* The normalization between stacked layers on its own: for each row r of
 * x [rows, H] bf16, out[r] = bf16(x[r] * rsqrt(mean(x[r]^2) + 1e-6)), the sum
 * of squares in fp32. H a multiple of 8; out may equal x (in place), otherwise
 * the two must not overlap; both 16-byte aligned. */
moe_status moe_rms_norm(int64_t rows, int32_t H, const uint16_t* x, uint16_t* out, void* stream);
moe_status moe_stack_forward(const moe_config* cfg, const moe_exec* ex, const moe_weights* layers,
                             int32_t n_layers, int32_t rms_norm, const uint16_t* x, uint16_t* out,
                             void* ws, size_t ws_bytes, void* stream, void* aux_stream);

/*
 * CUDA-graph form of moe_stack_forward: runs the stack once eagerly (on a
 * private stream ordered after prior work on `stream`, then synchronised, so
 * x must be ready by then), then records it by stream capture into an
 * executable graph bound to these pointers and shapes (x, out, ws, every
 * layer's weights; ex->stage_events must be NULL). moe_graph_launch replays
 * all layers with one launch on `stream`: new inputs are written into x, the
 * result is read from out. The weights, ws, x and out must stay allocated
 * while the graph exists. The graph does not synchronise; errors latched by
 * the kernels are read with moe_check_errors as usual.
 * moe_graph_kernel_count: kernels of this library in one replay.
 */
typedef struct moe_graph_s* moe_graph;
moe_status moe_graph_create_stack(const moe_config* cfg, const moe_exec* ex,
                                  const moe_weights* layers, int32_t n_layers, int32_t rms_norm,
                                  const uint16_t* x, uint16_t* out, void* ws, size_t ws_bytes,
                                  void* stream, moe_graph* graph);
moe_status moe_graph_launch(moe_graph graph, void* stream);
uint64_t moe_graph_kernel_count(moe_graph graph);
void moe_graph_destroy(moe_graph graph);

/*
 * Testing hook for failure detection (no counterpart in the paper): exactly
 * moe_expert_ffn, except that CTA 0 of each grouped GEMM never issues its
 * producer fill number `stall_fill` (0-based), so the MMA's barrier wait on
 * that stage cannot complete, and every barrier wait is limited to
 * wait_limit_ns (1 ms .. 2 s). The kernel must then latch MOE_ERR_TIMEOUT,
 * let its issued copies and MMAs finish (bounded), free its tensor memory
 * and return; moe_check_errors() reports the timeout and the context stays
 * usable. y_perm and the workspace hold garbage afterwards. Faults, traps and
 * hangs are never used: the wait simply runs out.
 */
moe_status moe_testing_expert_ffn_stall(int32_t rows, int32_t H, int32_t I, int32_t n_experts,
                                        const uint16_t* x_perm, const int32_t* offsets,
                                        const uint16_t* W13, const uint16_t* W2, float* y_perm,
                                        void* ws, size_t ws_bytes, int64_t stall_fill,
                                        int64_t wait_limit_ns, void* stream);

/*
 * Testing (no counterpart in the paper): a failure injected on the host. With
 * n >= 0, the stage calls inside the moe_layer_forward calls that follow (the
 * routing-and-packing step of a chunk, the expert GEMMs of a chunk or expert
 * range) pass until n of them have; the next one returns MOE_ERR_CUDA without
 * launching anything, and the injector turns itself off. n = -1 turns it off.
 * Process-wide. Used to check that a pipelined forward failing after it forked
 * its pack stream still joins that stream back into the caller's stream before
 * returning. MOE_ERR_INVALID_ARG for n < -1.
 */
moe_status moe_testing_fail_stage(int32_t n);

/*
 * Testing (no counterpart in the paper): the tile-packed row layout in which
 * the layer keeps its bf16 and row-scaled e4m3 token operands (x_perm, and
 * GEMM2's h or hq). Writes to *out the index, in 16-byte units from the buffer's
 * start, of 16-byte chunk c of packed row r, which belongs to expert e whose
 * rows are [off_e, off_e + cnt_e). The rows of expert e are cut into tiles of
 * `tile` rows; tile t starts at padded row off_e + 16 e + t tile and stores
 * n_pad = its rows rounded up to 16; block kb (chunks 8 kb .. 8 kb + 7 of
 * every row) of the tile is contiguous, n_pad x 8 chunks, and row i's chunk
 * j sits at i * 8 + (j xor (i mod 8)) inside it. Host computation only (the
 * function the kernels use). MOE_ERR_INVALID_ARG unless 0 <= e, cnt_e >= 1,
 * off_e <= r < off_e + cnt_e, tile a positive multiple of 16,
 * chunks_per_row a positive multiple of 8 and 0 <= c < chunks_per_row.
 */
moe_status moe_testing_tiled_chunk(int32_t r, int32_t e, int32_t off_e, int32_t cnt_e,
                                   int32_t tile, int32_t chunks_per_row, int32_t c,
                                   int64_t* out);

/* Synchronises `stream`, then reads and clears the device error word of the
 * current device. MOE_OK, MOE_ERR_TIMEOUT or MOE_ERR_DEVICE_CHECK (or
 * MOE_ERR_CUDA if the synchronisation itself failed). */
moe_status moe_check_errors(void* stream);

/* Number of kernels this library has launched in this process (all devices). */
uint64_t moe_launch_count(void);

/* Releases internal streams and events, and forgets the cached device address
 * of moe_dispatch_noalloc's scratch array (the next such call looks it up
 * again). Call it after cudaDeviceReset and before the library's next call on
 * that device. Safe to call more than once. */
void moe_shutdown(void);

#ifdef __cplusplus
}
#endif

#endif /* MOE_H_ */
