// Internal helpers shared by the kernels of the MoE library (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "moe.h"

namespace moe {

// ----------------------------------------------------------------------------
// host-side bookkeeping
// ----------------------------------------------------------------------------

// Counts every kernel launch of the library (exported through moe_launch_count).
void note_launch(int n = 1);

// Device error word of the current device (a file-scope __device__ int).
int* device_error_word();

// Number of SMs of the current device (cached per device).
int num_sms();

// Forgets the cached device addresses of moe_dispatch_noalloc's scratch array
// (moe_shutdown; after a device reset the array lives at a new address).
void forget_noalloc_scratch();

// Status of the last launch on this thread.
inline moe_status launch_status() {
  return cudaPeekAtLastError() == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

// ----------------------------------------------------------------------------
// kernel launchers (defined in the kernel translation units)
// ----------------------------------------------------------------------------

moe_status launch_router(const moe_config& c, const uint16_t* x, const float* Wr, float* logits,
                         float* partials, int splits, cudaStream_t s);
int router_splits(const moe_config& c);
// The router as the library runs it: tensor cores when E % 128 == 0 and a
// workspace of router_workspace_bytes(c) is given, else the SIMT kernel.
size_t router_workspace_bytes(const moe_config& c);
moe_status launch_router_auto(const moe_config& c, const uint16_t* x, const float* Wr,
                              float* logits, void* ws, cudaStream_t s);

// Tensor-core router (E a multiple of 128): Wr split into three bf16 planes
// (hi, mid, lo) whose sum is the fp32 value; partial logits per K split.
moe_status launch_split_planes(const float* Wr, size_t n, uint16_t* planes, cudaStream_t s);
int router_tc_splits(int T, int H, int E);
moe_status launch_router_tc(int T, int H, int E, const uint16_t* x, const uint16_t* planes,
                            float* partials, int k_splits, cudaStream_t s);
moe_status launch_router_reduce(const float* partials, int splits, size_t n, float* logits,
                                cudaStream_t s);

moe_status launch_gate(const moe_config& c, const float* logits, const float* bias, int32_t* idx,
                       float* w, cudaStream_t s);

int perm_num_chunks(int T);
// row_w (optional, with topk_w [T*k]): row_w[slot_row[n]] = topk_w[n], the
// gate weight of every packed row, for a combine fused into GEMM2.
moe_status launch_permutation(const moe_config& c, const int32_t* idx, int32_t* counts,
                              int32_t* offsets, int32_t* row_src_token, int32_t* slot_row,
                              int32_t* chunk_counts, int32_t* chunk_base, cudaStream_t s,
                              const float* topk_w = nullptr, float* row_w = nullptr);
// Tile-packed token rows: the layout in which the layer keeps the bf16
// operands of its expert GEMMs (x_perm and h), so that a stage's token rows
// are one contiguous bulk copy instead of a tensor-map load of n 128-byte row
// segments (hot GEMM1 units measured 8 % faster with the packed form). The
// packed rows of expert e (its global index), [off[e], off[e+1]), are cut into
// tiles of `tile` rows, the expert GEMMs' token tile. Tile t of expert e
// starts at padded row P = off[e] + 16 e + t * tile and holds n_pad = the
// tile's rows rounded up to 16. Its columns come in blocks of 128 bytes:
// block kb of the tile (n_pad rows x 128 bytes) is contiguous at byte
// P * row_bytes + kb * n_pad * 128, its row i at i * 128, and the 16-byte
// chunk j of that row at chunk j ^ (i % 8) (the 128-byte swizzle of a K-major
// MMA operand). A buffer of `rows` packed rows holds rows + 16 E rows (each
// expert's last tile pads at most 15). TiledRow locates packed row r of
// expert e; chunk16 gives the 16-byte unit index of its chunk c.
struct TiledRow {
  size_t tile16;  // 16-byte index of the tile's first byte
  int i;          // row within the tile
  int n_pad;      // rows the tile stores
  __host__ __device__ size_t chunk16(int c) const {
    return tile16 + (size_t)(c >> 3) * n_pad * 8 + (size_t)i * 8 + ((c & 7) ^ (i & 7));
  }
};
__host__ __device__ inline TiledRow tiled_row(int r, int e, int off_e, int cnt_e, int tile,
                                              int chunks_per_row) {
  const int l = r - off_e, t = l / tile;
  const int m = cnt_e - t * tile < tile ? cnt_e - t * tile : tile;
  TiledRow w;
  w.i = l - t * tile;
  w.n_pad = (m + 15) & ~15;
  w.tile16 = (size_t)(off_e + 16 * e + t * tile) * chunks_per_row;
  return w;
}

// tile > 0: x_perm in the tile-packed layout, slot n's expert idx[n] and the
// packed-row offsets [E+1] placing its row.
moe_status launch_dispatch_rows(int T, int H, int k, const uint16_t* x, const int32_t* slot_row,
                                uint16_t* x_perm, cudaStream_t s, int tile = 0,
                                const int32_t* idx = nullptr, const int32_t* offsets = nullptr);
// x_perm[r] = x[row_src_token[r]] for the rows of experts [e_begin, e_end);
// tile > 0 writes them in the tile-packed layout above (offsets global).
moe_status launch_gather_rows(int H, const uint16_t* x, const int32_t* row_src_token,
                              const int32_t* offsets, int e_begin, int e_end, uint16_t* x_perm,
                              int max_rows, cudaStream_t s, int tile = 0);
moe_status launch_combine(int T, int H, int k, const float* y_perm, const int32_t* slot_row,
                          const float* w, const float* shared, void* out, int out_fp32,
                          cudaStream_t s);

moe_status launch_fill_range(int32_t* offsets, int n, cudaStream_t s);
moe_status launch_sum_counts(const int32_t* counts, int n_chunks, int E, int32_t* out,
                             cudaStream_t s);

// One operand group of the grouped expert GEMMs: experts [e_begin, e_end) of
// the packed activations x [rows, H] with device row offsets, or (offsets
// unused) a single dense segment [0, rows) with one weight matrix.
struct FfnGroup {
  const void* x;  // [rows or x_rows, H] bf16, or e4m3 bytes when fp8
  const int32_t* offsets;
  int rows, n_experts, e_begin, e_end;
  const void* W13;  // bf16, or e4m3 bytes when fp8
  const void* W2;
  uint16_t* h;  // [rows, I] bf16
  float* y;     // [rows, H] fp32
  // Fused dispatch: packed row r of the group is row gather[r] of x (x_rows
  // rows), read by GEMM1 directly; null = x is already packed.
  const int32_t* gather;
  int x_rows;
  bool packed;  // W13 / W2 in the tile-packed layout (moe_pack_weights)
  // bf16 token operands in the tile-packed row layout (TiledRow) with the
  // launch's token tile: x (GEMM1's, when it is not gathered) and h (GEMM1's
  // output, GEMM2's operand); both buffers then hold rows + 16 * n_experts rows.
  bool x_tiled;
  bool h_tiled;
  int x_tile;  // the token tile x and h are laid out for (0 = chosen by the launch)
  // FP8 (row scales): hq, GEMM2's e4m3 operand, in the tile-packed layout (h
  // itself stays row-major for the quantizer); hq then holds the padding rows
  bool hq_tiled;
  // FP8 (e4m3) form: per-row fp32 scales of x (indexed by token through
  // x_scale_idx when x holds packed copies, else by row), of W13 and W2 rows;
  // hq / hs receive GEMM2's quantized operand and its row scales.
  bool fp8;
  const float* x_scale;
  const int32_t* x_scale_idx;
  const float* W13_scale;
  const float* W2_scale;
  uint8_t* hq;
  float* hs;
  // Block-scaled FP8 (fp8 and fp8_block): UE8M0 exponents of x's 1 x 128
  // blocks (x_sf[token * x_sf_ld + kb], the token through x_scale_idx as
  // above) and of the 128 x 128 blocks of W13 and W2 ([rows / 128][K / 128]);
  // hsf receives those of h's 1 x 128 blocks (hsf[row * h_sf_ld + kb]).
  bool fp8_block;
  const uint8_t* x_sf;
  long x_sf_ld;
  const uint8_t* W13_sf;
  const uint8_t* W2_sf;
  uint8_t* hsf;
  long h_sf_ld;
  // Combine fused into GEMM2 (comb_out non-null): instead of y, GEMM2 adds
  // comb_w[r] * y[r] into comb_out[comb_tok[r]] with fp32 reductions (comb_tok
  // null = row r is token r; comb_w null = weight 1).
  float* comb_out;
  const int32_t* comb_tok;
  const float* comb_w;
  // Dynamic unit scheduling (two ints, 0 before the first launch that uses them;
  // launches sharing them must run one after another): null = static.
  int* sched;
  // Dispatch fused into GEMM1 (pack_src non-null, x = the packed rows it
  // writes): packed row r = pack_src row pack_rst[r] (pack_src_rows rows, the
  // activation row size); pack_next (one int) and pack_ready (one int per
  // expert of the group) are 0 before the first launch and left at 0.
  const void* pack_src;
  const int32_t* pack_rst;
  int pack_src_rows;
  int* pack_next;
  int* pack_ready;
  // Token-major copy (used when the launch also runs group 1, whose units come
  // first): pack_slot[t * pack_k + j] is the packed row of token t's slot j.
  // Each token row is then read once for its pack_k rows. Null: packed-row
  // order through pack_rst.
  const int32_t* pack_slot;
  int pack_k;
  // Per-unit trace of the GEMM1 (trace_gemm 1) or GEMM2 (2) launch
  // (moe_exec.unit_trace; null = off).
  unsigned long long* trace;
  int trace_cap;
  int trace_gemm;
};

// The expert GEMMs' token tile for rows_hint packed rows over n_exp experts:
// small tiles leave more of the stage ring to weights (decode ~4 rows per
// expert -> 32; balanced prefill ~128 +- 10 % -> 144; larger or skewed loads
// -> 256, or 224 with block-scaled FP8).
int ffn_tile_rows(long rows_hint, int n_exp, bool fp8, bool fp8_block);

// Routed group plus an optional dense group (the shared expert, same I) in one
// pair of launches.
moe_status launch_expert_ffn_groups(const FfnGroup& routed, const FfnGroup* dense, int H, int I,
                                    int rows_hint, cudaStream_t s,
                                    cudaEvent_t after_gemm1 = nullptr);

// Testing: moe_expert_ffn whose GEMM1 has one producer fill of CTA 0 never issued,
// with the given barrier-wait limit (exercises the timeout and abort path).
moe_status launch_expert_ffn_stalled(int rows, int H, int I, int n_experts, const uint16_t* x_perm,
                                     const int32_t* offsets, const uint16_t* W13,
                                     const uint16_t* W2, uint16_t* h, float* y_perm,
                                     long stall_fill, uint64_t wait_limit_ns, cudaStream_t s);

// Grouped expert GEMM on tcgen05. Experts [e_begin, e_end) of `offsets`.
moe_status launch_expert_ffn(int rows, int H, int I, int n_experts, int e_begin, int e_end,
                             const uint16_t* x_perm, const int32_t* offsets, const uint16_t* W13,
                             const uint16_t* W2, uint16_t* h, float* y_perm, int rows_hint,
                             cudaStream_t s, cudaEvent_t after_gemm1 = nullptr,
                             bool packed = false);

// e4m3 row quantization of a bf16 matrix [rows, K] (K % 8 == 0); tile > 0:
// only the packed rows of experts [e_begin, e_end) of `offsets`, the e4m3
// rows written in the tile-packed layout (TiledRow), K % 16 == 0.
moe_status launch_quantize_rows(const uint16_t* in, long rows, int K, uint8_t* out, float* scale,
                                cudaStream_t s, const int32_t* offsets = nullptr,
                                int e_begin = 0, int e_end = 0, int tile = 0);

// e4m3 quantization of a bf16 matrix [rows, K] in 1 x 128 blocks (K % 128 == 0):
// k = the smallest exponent with amax <= 448 * 2^k (0 for a zero block, within
// [-127, 127]); out[r][c] = e4m3(in[r][c] * 2^-k); sf[r * sf_ld + c / 128] = k + 127.
moe_status launch_quantize_blocks(const uint16_t* in, long rows, int K, uint8_t* out, uint8_t* sf,
                                  long sf_ld, cudaStream_t s);
// The same in 128 x 128 blocks (rows % 128 == 0): sf[(r / 128) * (K / 128) + c / 128].
moe_status launch_quantize_weight_blocks(const uint16_t* in, long rows, int K, uint8_t* out,
                                         uint8_t* sf, cudaStream_t s);

// Tile-packed copy of a bf16 weight matrix [rows, K] (rows % 128 == 0, K % 64 == 0).
moe_status launch_pack_weights(const uint16_t* W, uint16_t* Wp, long rows, int K, cudaStream_t s);

// ----------------------------------------------------------------------------
// device helpers
// ----------------------------------------------------------------------------

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

__device__ __forceinline__ uint16_t float_to_bf16_bits(float f) {
  __nv_bfloat16 h = __float2bfloat16_rn(f);
  return *reinterpret_cast<uint16_t*>(&h);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

}  // namespace moe
