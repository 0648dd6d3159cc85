// Grouped expert GEMMs on the 5th-generation tensor cores (tcgen05 + TMEM),
// operands staged by TMA: the expert compute of the paper's MoE workload
// (GEMM1 up/gate 7168 x 4096 + SwiGLU + GEMM2 down 2048 x 7168, Appendix
// "Workload Details"), one launch per GEMM over every expert.
//
// Orientation ("swap AB"): the MMA's M side is 128 rows of an expert's weight
// matrix, its N side is up to NMAX packed token rows of that expert. So an
// expert with only a few tokens (decode) wastes no tensor work, and the weight
// tile -- the bytes that bound the layer -- is streamed exactly once per
// (expert, 128-feature block, token tile).
//   D[f, n] = sum_k W[f, k] * X[n, k]      (both operands K-major, bf16)
// D lives in TMEM: lane = output feature, column = token.
//
// Work unit = (expert e, token tile nt, feature block fb): experts in order,
// inside an expert blocks of up to 8 token tiles, each block's feature blocks
// in turn (block_order below). The units of every expert are enumerated on the
// device from the row offsets, so a launch needs no host-side knowledge of the
// routing. A launch may carry a
// second operand group: one dense segment with its own weights and
// activations (the shared expert), whose units run in the same persistent
// grid as the routed ones. A persistent grid (one CTA per SM) runs the units:
// each CTA's producer takes the next unit index from a global counter as it
// becomes free (so the units in flight are consecutive ones, sharing token and
// weight tiles in L2, however unequal their sizes), or, without a counter,
// round-robin; it announces each unit to the CTA's other roles through a
// small ring in shared memory. Warp roles:
//   warp 0     TMA producer: weight tile(s) 128 x 64 and token rows 16 x 64
//              per stage into a STAGES-deep ring (128-byte swizzle); takes and
//              announces the units;
//   warp 1     MMA issuer (one thread): 4 x tcgen05.mma (K = 16 each) per stage,
//              tcgen05.commit frees the stage, a final commit hands the
//              accumulator to the epilogue; also owns the TMEM allocation;
//   warps 2-9  epilogue, two warps per 32-lane TMEM quarter taking turns on
//              16-column chunks: tcgen05.ld the accumulator; GEMM1 applies
//              SwiGLU and stores h in bf16 (the operand of GEMM2), GEMM2 stores
//              y in fp32 (summed by combine, or added into the output by the
//              fused combine);
//   warp 10    block-scaled FP8 only: the stage's UE8M0 exponents as scale
//              images in shared memory, which the MMA thread copies to TMEM
//              (tcgen05.cp) ahead of block_scale MMAs;
//   warps 10-13 GEMM1 with bf16 or row-scaled e4m3 operands: the dispatch
//              fused into the launch (GemmArgs::pack_dst). They copy the
//              token rows into the packed order, a chunk at a time taken from
//              a global counter: a few tokens, each row read once and written
//              to its k packed rows, when the launch also runs the shared
//              expert; else a few packed rows in row (= expert) order. They
//              count each expert's packed rows; the producer waits for an
//              expert's count before loading its token tiles. The shared
//              expert's units (which read x itself) come first in the unit
//              order, so the copy runs while they compute: the paper's
//              dispatch hidden behind the layer's own compute, inside one
//              kernel.
// For SwiGLU the gate and up tiles of the same 128 features are two MMAs into
// two TMEM column ranges, so one thread holds both g and u of its feature.
// When two accumulators fit in TMEM's 512 columns they alternate, so the
// epilogue of one unit overlaps the MMAs of the next.
//
// Every mbarrier wait is bounded (%globaltimer): on expiry the kernel latches
// MOE_ERR_TIMEOUT, tells the other roles to stop, waits (bounded) for its own
// copies and MMAs in flight, frees TMEM and returns.
#include <cudaTypedefs.h>

#include <type_traits>

#include "common.cuh"

#define MOE_STATUS_TRY(expr)          \
  do {                                \
    moe_status _st = (expr);          \
    if (_st != MOE_OK) return _st;    \
  } while (0)

namespace moe {
namespace {

constexpr int BM = 128;           // weight rows per tile (MMA M)
constexpr int BK = 64;            // bf16 per stage along K: one 128-byte swizzle row
constexpr int UMMA_K = 16;        // K of one tcgen05.mma kind::f16
constexpr int B_BOX = 16;         // token rows per TMA box (tile remainders)
constexpr int B_BIG = 64;         // token rows per TMA box (bulk of tiles of >= 64 rows)
// Warps: 0 producer, 1 MMA issuer, then the epilogue warps (epi_warps of the
// mode), then the block-scaled form's scale warp or GEMM1's pack warps.
constexpr int PACK_WARPS = 4;     // GEMM1 (bf16, row-scaled e4m3): warps copying token rows
constexpr int PACK_ROWS = 4;      // token rows per chunk a pack warp takes
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;  // default limit of every barrier wait



constexpr int pow2ceil(int v) {
  int p = 32;
  while (p < v) p <<= 1;
  return p;
}

// Kernel modes: what one work unit's weight tiles are and what its epilogue does.
constexpr int MODE_PLAIN = 0;   // one 128-feature weight tile; fp32 output
constexpr int MODE_SWIGLU = 1;  // gate and up tiles of the same 128 features; SwiGLU, bf16 out
constexpr int MODE_PLAIN2 = 2;  // two adjacent 128-feature tiles sharing one token tile; fp32 out
constexpr int MODE_SPLIT3 = 3;  // three bf16 planes of one fp32 weight tile, summed into one
                                // accumulator (an fp32 x bf16 product on bf16 tensor cores)

// Operand precision of a launch: bf16; e4m3 with fp32 row scales applied in
// the epilogue; e4m3 with UE8M0 block scales (1 x 128 per token row, 128 x 128
// per weight block) applied by the tensor core (kind::mxf8f6f4 block_scale).
constexpr int Q_BF16 = 0;
constexpr int Q_ROW = 1;
constexpr int Q_BLOCK = 2;

template <int MODE, int NMAX, bool MX = false>
struct Tile {
  static constexpr int NA = MODE == MODE_PLAIN ? 1 : MODE == MODE_SPLIT3 ? 3 : 2;  // A tiles
  static constexpr bool TWO_ACC = MODE == MODE_SWIGLU || MODE == MODE_PLAIN2;  // tile i -> acc i
  static constexpr int FEAT = MODE == MODE_PLAIN2 ? 2 * BM : BM;  // output features per unit
  static constexpr int A_BYTES = BM * BK * 2;  // 16 KiB
  static constexpr int B_BYTES = NMAX * BK * 2;
  // Block scales (MX): per stage one 512-byte scale image per A tile and per
  // 128 token rows, in the order tcgen05.cp 32x128b.warpx4 expects (entry x at
  // byte 16 * (x % 32) + 4 * (x / 32 % 4)), after the operand tiles.
  static constexpr int SF_CB = MX ? (NMAX + 127) / 128 : 0;  // token-scale images
  static constexpr int SF_OFF = NA * A_BYTES + B_BYTES;
  static constexpr int SF_BYTES = MX ? ((NA + SF_CB) * 512 + 1023) / 1024 * 1024 : 0;
  static constexpr int STAGE_BYTES = NA * A_BYTES + B_BYTES + SF_BYTES;
  // MX: the producer's staging copy of a unit's exponents for SF_KC k-blocks:
  // token j's at j * SF_STR (a stride that keeps the per-stage reads of 32
  // consecutive tokens on distinct banks), then the A tiles' at t * SF_KC.
  static constexpr int SF_KC = 32;
  static constexpr int SF_STR = SF_KC + 4;
  static constexpr int SF_STG_A = NMAX * SF_STR;
  static constexpr int SF_STG_BYTES = MX ? (SF_STG_A + NA * SF_KC + 15) / 16 * 16 : 0;
  // ~217 KiB of stages and staging: with the control block, the expert tables
  // (<= 8 KiB) and the 1 KiB alignment slack this stays under 227 KiB per CTA.
  static constexpr int STAGES_RAW = (217 * 1024 - SF_STG_BYTES) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_RAW > 12 ? 12 : STAGES_RAW;
  static constexpr int ACC_COLS = TWO_ACC ? 2 * NMAX : NMAX;  // one accumulator (gate | up)
  // MX: each stage's scales live in TMEM columns of their own (4 per image)
  // until the stage's MMAs complete
  static constexpr int SF_COLS = MX ? 4 * (NA + SF_CB) : 0;
  static constexpr int ACC_STAGES =
      2 * ACC_COLS + STAGES * SF_COLS <= 512 ? 2 : 1;  // double-buffer when it fits
  static constexpr int SF_COL0 = ACC_STAGES * ACC_COLS;
  static constexpr int TMEM_COLS = pow2ceil(SF_COL0 + STAGES * SF_COLS);
  static_assert(STAGES >= 2, "pipeline too shallow");
  static_assert(NMAX % 16 == 0 && NMAX >= 16 && NMAX <= 256, "MMA N range for M = 128");
  static_assert(TMEM_COLS <= 512, "TMEM holds 512 columns");
  static_assert(SF_OFF % 1024 == 0 && STAGE_BYTES % 1024 == 0, "stage alignment");
};

constexpr int UNIT_RING = 8;  // units announced ahead by the producer (a power of two)
constexpr int TRACE_FIELDS = 5;  // per-unit trace record (GemmArgs::trace)

struct Ctrl {
  uint64_t full[12];
  uint64_t empty[12];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  // The producer announces each unit this CTA runs (its index, or an index
  // past the last unit to stop) in unit_ring; the other roles read it there.
  uint64_t unit_full[UNIT_RING];
  uint64_t unit_empty[UNIT_RING];
  int unit_ring[UNIT_RING];
  uint32_t tmem_base;
  int abort_flag;
};

// ------------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `bar` with the given parity; false on abort or timeout.
__device__ __noinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* err, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > limit_ns) {
      *abort_flag = 1;
      atomicExch(err, (int)MOE_ERR_TIMEOUT);
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// One weight tile of the tile-packed layout: 16 KiB, contiguous and already in
// the 128-byte-swizzled order the MMA descriptors expect, so a plain bulk copy
// (no tensor map) lands it ready to use.
__device__ __forceinline__ void bulk_load_tile(uint32_t dst, const void* src, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(BM * BK * 2), "r"(bar)
      : "memory");
}

// `bytes` contiguous bytes (a multiple of 16, both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
      : "memory");
}

// Four rows (y0..y3) of a 2-D tensor whose map has a one-row box, landing as
// four consecutive 128-byte rows of a swizzled tile (tile::gather4).
__device__ __forceinline__ void tma_gather4(uint32_t dst, const CUtensorMap* map, int x, int y0,
                                            int y1, int y2, int y3, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y0), "r"(y1), "r"(y2), "r"(y3), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tma_prefetch_map(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row swizzle atoms 1024 bytes apart (stride byte offset), the
// leading byte offset unused, descriptor version 1, base offset 0 (atoms are
// 1024-byte aligned). Advancing K by 16 bf16 adds 32 bytes to the start.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) |
         (2ull << 61);
}

// Instruction descriptor, kind::f16: fp32 accumulator (bits 4-5 = 1), A and B
// bf16 (bits 7-9, 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at bit 17,
// M >> 4 at bit 24.
__device__ __forceinline__ uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(BM >> 4) << 24);
}

// Instruction descriptor, kind::f8f6f4 with e4m3 A and B (format code 0 in bits
// 7-9 and 10-12), fp32 accumulator, K-major, same N / M fields.
__device__ __forceinline__ uint32_t idesc_e4m3(int n) {
  return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

// One MMA of K = 32 e4m3 values (32 bytes, like K = 16 bf16).
__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Instruction descriptor, kind::mxf8f6f4 with e4m3 A and B: as above without
// the accumulator-format field (bits 4-5 select the byte of each B scale word
// instead, 0 here, like bits 29-30 for A) and with UE8M0 scales (bit 23).
__device__ __forceinline__ uint32_t idesc_mx(int n) {
  return ((uint32_t)(n >> 3) << 17) | (1u << 23) | ((uint32_t)(BM >> 4) << 24);
}

// One block-scaled MMA of K = 32 e4m3 values: each A row and each B row
// carries one UE8M0 scale 2^(s - 127) for these 32 products, read from TMEM:
// A row i at lane i, column sfa + i / 32; B row j at column sfb + j / 32, lane
// j % 32 of every 32-lane quarter (byte 0 of each 32-bit word).
__device__ __forceinline__ void mma_mx(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t sfa, uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%4], "
      "[%5], p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

// Shared-memory descriptor of a 512-byte scale image for tcgen05.cp: no
// swizzle, 8-row core matrices of 16-byte rows 128 bytes apart.
__device__ __forceinline__ uint64_t sdesc_sf(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(128 >> 4) << 32) | (1ull << 46);
}

// 32 rows x 16 bytes of shared memory -> 4 TMEM columns, row r to lane r of
// each of the four 32-lane quarters. Ordered before the MMAs this thread
// issues next.
__device__ __forceinline__ void sf_copy(uint32_t taddr, uint32_t saddr) {
  asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr),
               "l"(sdesc_sf(saddr))
               : "memory");
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate);

template <bool F8>
__device__ __forceinline__ void mma_op(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t acc) {
  if (F8) mma_e4m3(d, a, b, idesc, acc);
  else mma_bf16(d, a, b, idesc, acc);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

// SiLU(g) * u for the SwiGLU epilogue: g / (1 + e^-g) * u with e^-g = 2^(-g log2 e)
// on the hardware exp2 and the quotient through the hardware reciprocal, both
// flushing denormals (the forms without .ftz add fix-up instructions for
// denormal inputs and results that this epilogue never needs: e^-g is
// denormal only for g > 87, where 1 + e^-g = 1 either way). The result's error
// is a few fp32 ulp, far below the bf16 rounding of h that follows.
__device__ __forceinline__ float silu_mul(float g, float u) {
  constexpr float kLog2e = 1.4426950408889634f;  // log2(e)
  float e, r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(-g * kLog2e));
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(1.0f + e));
  return g * r * u;
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ------------------------------------------------------------------ schedule

// Launch arguments besides the tensor maps. Group 0: experts [e_begin,
// e_begin + n_exp) of a packed activation matrix with `rows0` rows, segments
// given by device offsets. Group 1 (rows1 > 0): one segment [0, rows1) of its
// own activation matrix with one weight matrix (the shared expert).
struct GemmArgs {
  const int32_t* offsets;
  const int32_t* gather0;  // group 0: activation row of packed row r (fused dispatch), or null
  int rows0, e_begin, n_exp;
  int rows1;
  int K, n_fb;
  int w_rows0;  // weight rows per expert in group 0
  int up_off;   // row offset between a unit's weight tiles (SwiGLU: the up projection)
  const uint16_t* a0_packed;  // group 0 weights in the tile-packed layout (else null: tensor maps)
  const uint16_t* a1_packed;  // group 1 likewise
  int k_splits; // group 1 only: the K range is split into this many units ...
  long split_stride;  // ... whose outputs go to out1 + split * split_stride (partials)
  void* out0;
  void* out1;
  int out_ld;
  int* err;
  // FP8 only: fp32 scale of every weight row (a_scale*, indexed by the absolute
  // weight row) and of every activation row (b_scale*, indexed by the B row, or
  // through b_scale_idx0 for group 0 when the rows are packed copies of tokens)
  const float* a_scale0;
  const float* a_scale1;
  const float* b_scale0;
  const float* b_scale1;
  const int32_t* b_scale_idx0;
  // Block-scaled FP8 only: UE8M0 exponents of the 128 x 128 weight blocks
  // ([weight rows / 128][K / 128], absolute weight rows) and of the 1 x 128
  // activation blocks (b_sf[row * b_sf_ld + kb], the row through b_scale_idx0
  // for group 0 when given)
  const uint8_t* a_sf0;
  const uint8_t* a_sf1;
  const uint8_t* b_sf0;
  const uint8_t* b_sf1;
  long b_sf_ld0, b_sf_ld1;
  // PLAIN / PLAIN2 only: the combine fused into the epilogue. Non-null comb_out*
  // replaces the y store of that group by comb_out[tok][f] += w * y (fp32
  // reductions), tok = comb_tok0[row] and w = comb_w0[row] for group 0 (null:
  // the row itself, weight 1), the row itself and weight 1 for group 1.
  float* comb_out0;
  float* comb_out1;
  const int32_t* comb_tok0;
  const float* comb_w0;
  // Dynamic unit scheduling: sched[0] hands out unit indices (atomicAdd) to the
  // CTAs' producers as they become free, so the units running at one time are
  // consecutive ones whatever their sizes; sched[1] counts exited CTAs, and the
  // last one to exit sets both back to 0 for the next launch. Both must be 0 at
  // the first launch; launches sharing them must not overlap in time. Null:
  // CTA b runs units b, b + grid, b + 2 grid, ...
  int* sched;
  // Dispatch fused into GEMM1 (pack_dst non-null; group 0 only): packed row r
  // of group 0 is pack_src row pack_rst[r] (pack_src_rows rows of K elements).
  // pack_next hands out chunks of PACK_ROWS rows; pack_ready[e] counts the
  // packed rows of expert e_begin + e. Both are 0 at the first launch; the last
  // CTA out sets them back to 0.
  const uint4* pack_src;
  uint4* pack_dst;
  const int32_t* pack_rst;
  int pack_src_rows;
  int* pack_next;
  int* pack_ready;
  // Token-major form (non-null): pack_next hands out chunks of tokens and
  // token t's slot j goes to packed row pack_slot[t * pack_k + j].
  const int32_t* pack_slot;
  int pack_k;
  // Token operands (bf16, or e4m3 rows) in the tile-packed row layout
  // (TiledRow, tile = NMAX): group g's token rows come from b_tiled_g by one
  // bulk copy per stage (null: through the tensor maps), and GEMM1 writes group
  // g's bf16 h to out_g in that layout when out_tiled_g. A tile's first padded
  // row: row0 + 16 * (its global expert; 0 for group 1). The buffers hold 16
  // padding rows per expert.
  const uint8_t* b_tiled0;
  const uint8_t* b_tiled1;
  int out_tiled0, out_tiled1;
  // Per-unit trace of this launch (null = off): record u < trace_cap of
  // TRACE_FIELDS uint64: the unit's announcement by the producer, its first
  // stage ready at the MMA thread, its accumulator complete and its epilogue
  // done (warp 2), all %globaltimer ns, then SM id | m << 16 |
  // (expert + 1024 * group) << 32 | feature block << 48.
  unsigned long long* trace;
  int trace_cap;
  uint64_t wait_limit_ns;  // limit of each barrier wait
  long stall_fill;         // testing: CTA 0 never issues this fill (-1 = none), so the
                           // MMA's wait on it runs out and the abort path is exercised
};

struct Unit {
  int grp;   // operand group
  int e;     // expert (group 0, relative to e_begin)
  int fb;    // 128-feature block
  int row0;  // first activation row of the token tile
  int m;     // valid token rows in the tile (1..NMAX)
  int kb0, kb1;  // k-blocks [kb0, kb1) of this unit
  int split;     // K split index (group 1)
};

// Unit i of an operand with nt_n token tiles and n_fb feature blocks: blocks
// of up to 8 token tiles; inside a block the feature blocks in turn, and the
// block's token tiles together within a feature block. With the dynamic
// scheduler the units in flight are consecutive ones, so a weight tile is
// read from DRAM once per block of token tiles (its users are adjacent) and a
// token tile comes back after at most 8 units, while it is still in L2. Skewed
// batch, GEMM1 DRAM bytes: token-tile-major 19.3 GB, this order 17.8 GB
// (algorithmic 16.5 GB); with round-robin units 22.8 GB.
__device__ __forceinline__ void block_order(int i, int nt_n, int n_fb, int& nt, int& fb) {
  constexpr int G = 8;
  const int blk = i / (G * n_fb);
  const int nt0 = blk * G;
  const int gsz = min(G, nt_n - nt0);
  const int rem = i - blk * G * n_fb;
  fb = rem / gsz;
  nt = nt0 + (rem - fb * gsz);
}

template <int NMAX>
__device__ __forceinline__ Unit decode_unit(int u, const int* tile_off, const int* row_off,
                                            const GemmArgs& a, int units1, int kblocks) {
  Unit U;
  if (u < units1) {  // group 1: one dense segment (the shared expert, or the router)
    const int nt1 = (a.rows1 + NMAX - 1) / NMAX;
    const int per_split = nt1 * a.n_fb;
    U.split = u / per_split;
    u -= U.split * per_split;
    U.grp = 1;
    U.e = 0;
    int nt;
    block_order(u, nt1, a.n_fb, nt, U.fb);
    U.row0 = nt * NMAX;
    U.m = min(NMAX, a.rows1 - U.row0);
    const int kps = (kblocks + a.k_splits - 1) / a.k_splits;
    U.kb0 = min(kblocks, U.split * kps);
    U.kb1 = min(kblocks, U.kb0 + kps);
    return U;
  }
  U.split = 0;
  U.kb0 = 0;
  U.kb1 = kblocks;
  u -= units1;
  int lo = 0, hi = a.n_exp - 1;
  while (lo < hi) {  // largest e with tile_off[e] * n_fb <= u: an expert with tiles
    const int mid = (lo + hi + 1) >> 1;
    if (tile_off[mid] * a.n_fb <= u) lo = mid;
    else hi = mid - 1;
  }
  U.grp = 0;
  U.e = lo;
  const int local = u - tile_off[lo] * a.n_fb;
  int nt;
  block_order(local, tile_off[lo + 1] - tile_off[lo], a.n_fb, nt, U.fb);
  const int cnt = row_off[lo + 1] - row_off[lo];
  U.row0 = row_off[lo] + nt * NMAX;
  U.m = min(NMAX, cnt - nt * NMAX);
  return U;
}

// ------------------------------------------------------------------ kernel

// GEMM1 launches of the bf16 and row-scaled e4m3 forms carry the pack warps
// (idle and gone at once when the dispatch is not fused).
__host__ __device__ constexpr bool has_pack(int mode, int q) { return mode == MODE_SWIGLU && q != Q_BLOCK; }
// Epilogue warps (a multiple of 4: each TMEM lane quarter gets the same
// number). Eight: sixteen for GEMM2's two-tile units measured the same (their
// epilogue is bound by the SM's store bandwidth for the 256 KB of fp32 y of a
// full unit, not by the warps issuing the stores).
__host__ __device__ constexpr int epi_warps(int, int) { return 8; }
__host__ __device__ constexpr int threads_of(int mode, int q) {
  return 32 * (2 + epi_warps(mode, q) + (q == Q_BLOCK ? 1 : 0) +
               (has_pack(mode, q) ? PACK_WARPS : 0));
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ uint32_t sm_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
  return r;
}

// Field f of unit u's trace record (GemmArgs::trace), if tracing and u < cap.
__device__ __forceinline__ void trace_put(const GemmArgs& a, int u, int f,
                                          unsigned long long v) {
  if (a.trace && u < a.trace_cap) a.trace[(size_t)u * TRACE_FIELDS + f] = v;
}

template <int MODE, int NMAX, int Q, bool PK>
__global__ void __launch_bounds__(threads_of(MODE, Q), 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                        const __grid_constant__ CUtensorMap tmB0,
                        const __grid_constant__ CUtensorMap tmA1,
                        const __grid_constant__ CUtensorMap tmB1,
                        const __grid_constant__ CUtensorMap tmB0big,
                        const __grid_constant__ CUtensorMap tmB1big, const GemmArgs a) {
  constexpr bool F8 = Q != Q_BF16;  // e4m3 operands
  constexpr bool MX = Q == Q_BLOCK;  // ... with block scales applied by the MMA
  using TL = Tile<MODE, NMAX, MX>;
  constexpr bool SWIGLU = MODE == MODE_SWIGLU;
  constexpr int EPI = epi_warps(MODE, Q);  // epilogue warps 2 .. EPI_END - 1
  constexpr int EPI_END = 2 + EPI;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sf_stg = smem + TL::STAGES * TL::STAGE_BYTES;  // MX staging (SF_STG_BYTES)
  Ctrl* ctrl = reinterpret_cast<Ctrl*>(sf_stg + TL::SF_STG_BYTES);
  int* tile_off = reinterpret_cast<int*>(ctrl + 1);
  int* row_off = tile_off + a.n_exp + 1;
  volatile int* abort_flag = &ctrl->abort_flag;
  int* err = a.err;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < TL::STAGES; ++s) {
      mbar_init(smem_u32(&ctrl->full[s]), MX ? 2 : 1);  // MX: the producer and the scale warp
      mbar_init(smem_u32(&ctrl->empty[s]), 1);
    }
    for (int s = 0; s < TL::ACC_STAGES; ++s) {
      mbar_init(smem_u32(&ctrl->acc_full[s]), 1);
      mbar_init(smem_u32(&ctrl->acc_empty[s]), EPI);  // one arrive per epilogue warp
    }
    mbar_init(smem_u32(&ctrl->drain), 1);
    // readers of each announced unit: the MMA thread, the epilogue warps and
    // (block-scaled FP8) the scale warp
    for (int r = 0; r < UNIT_RING; ++r) {
      mbar_init(smem_u32(&ctrl->unit_full[r]), 1);
      mbar_init(smem_u32(&ctrl->unit_empty[r]), 1 + EPI + (MX ? 1 : 0));
    }
    ctrl->abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&ctrl->tmem_base)),
                 "r"(TL::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (warp == 2) {
    // Per-expert token tiles of group 0 and their prefix, from the device row
    // offsets. Offsets are clamped into [0, rows0] and made non-decreasing, so no
    // tile can reach outside the caller's buffers; a clamp latches
    // MOE_ERR_DEVICE_CHECK.
    const int n_exp = a.n_exp;
    const int per = (n_exp + 31) / 32;
    const int lo = min(n_exp, lane * per), hi = min(n_exp, lo + per);
    auto clamped = [&](int i) {
      const int v = a.offsets[a.e_begin + i];
      const int c = min(max(v, 0), a.rows0);
      if (c != v) atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
      return c;
    };
    int s = 0;
    for (int i = lo; i < hi; ++i) {
      const int r0 = clamped(i), r1 = max(clamped(i + 1), r0);
      if (r1 != clamped(i + 1)) atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
      row_off[i] = r0;
      s += (r1 - r0 + NMAX - 1) / NMAX;
    }
    int incl = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    int run = incl - s;
    for (int i = lo; i < hi; ++i) {
      tile_off[i] = run;
      run += (max(clamped(i + 1), row_off[i]) - row_off[i] + NMAX - 1) / NMAX;
    }
    if (lane == 31) {
      tile_off[n_exp] = incl;
      row_off[n_exp] = n_exp > 0 ? clamped(n_exp) : 0;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = ctrl->tmem_base;
  constexpr int KE = F8 ? 2 * BK : BK;  // elements per k-block: one 128-byte row
  const int kblocks = a.K / KE;
  const int units1 = a.rows1 > 0 ? ((a.rows1 + NMAX - 1) / NMAX) * a.n_fb * a.k_splits : 0;
  const int total_units = units1 + tile_off[a.n_exp] * a.n_fb;
  // The j-th unit of this CTA as announced by the producer (one lane of a role
  // calls this): its index, or -1 when the wait gave up (abort / timeout).
  auto next_unit = [&](int j) -> int {
    const int r = j & (UNIT_RING - 1);
    if (!wait_bounded(smem_u32(&ctrl->unit_full[r]), (uint32_t)((j / UNIT_RING) & 1), abort_flag,
                      err, a.wait_limit_ns))
      return -1;
    const int u = reinterpret_cast<volatile int*>(ctrl->unit_ring)[r];
    mbar_arrive(smem_u32(&ctrl->unit_empty[r]));
    return u;
  };

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    // Lane 0 owns the stage barriers and loads the weight tiles. Token rows are
    // either one contiguous 16-row box at a time (packed activations), or -- when
    // the dispatch is fused (a.gather0) -- gathered straight from x four rows per
    // tile::gather4 load, every lane issuing the groups of four it holds the row
    // indices of (registers, loaded once per unit).
    if (lane == 0) {
      tma_prefetch_map(&tmA0);
      tma_prefetch_map(&tmB0);
      if (units1) {
        tma_prefetch_map(&tmA1);
        tma_prefetch_map(&tmB1);
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    long fills = 0;
    bool ok = true;
    // lane 0 takes the next unit one unit ahead, so the atomic's round trip
    // overlaps the current unit's loads
    int u_next = 0;
    if (lane == 0) u_next = a.sched ? atomicAdd(a.sched, 1) : (int)blockIdx.x;
    for (int j = 0; ok; ++j) {
      int u = u_next, pub = 1;
      if (lane == 0) {  // announce unit j (its slot is free once every reader took unit j - 8)
        const int r = j & (UNIT_RING - 1);
        pub = wait_bounded(smem_u32(&ctrl->unit_empty[r]), (uint32_t)(((j / UNIT_RING) & 1) ^ 1),
                           abort_flag, err, a.wait_limit_ns)
                  ? 1
                  : 0;
        if (pub) {
          reinterpret_cast<volatile int*>(ctrl->unit_ring)[r] = u;
          if (u < total_units) trace_put(a, u, 0, global_timer_ns());
          mbar_arrive(smem_u32(&ctrl->unit_full[r]));
          if (u < total_units) u_next = a.sched ? atomicAdd(a.sched, 1) : u + (int)gridDim.x;
        }
      }
      pub = __shfl_sync(0xffffffffu, pub, 0);
      u = __shfl_sync(0xffffffffu, u, 0);
      if (!pub) {
        ok = false;
        break;
      }
      if (u >= total_units) break;
      const Unit U = decode_unit<NMAX>(u, tile_off, row_off, a, units1, kblocks);
      if (has_pack(MODE, Q) && a.pack_dst && U.grp == 0) {
        // fused dispatch: the expert's token rows must all be packed before its
        // token tiles are loaded (bounded wait on the pack warps' count)
        int okp = 1;
        if (lane == 0) {
          const int need = row_off[U.e + 1] - row_off[U.e];
          const int* rp = a.pack_ready + U.e;
          if (ld_acquire(rp) < need) {
            const uint64_t t0 = global_timer_ns();
            while (ld_acquire(rp) < need) {
              if (*abort_flag) {
                okp = 0;
                break;
              }
              if (global_timer_ns() - t0 > a.wait_limit_ns) {
                *abort_flag = 1;
                atomicExch(err, (int)MOE_ERR_TIMEOUT);
                okp = 0;
                break;
              }
              __nanosleep(128);
            }
          }
          fence_proxy_async_global();  // the rows were written by generic stores; TMA reads them
        }
        okp = __shfl_sync(0xffffffffu, okp, 0);
        if (!okp) {
          ok = false;
          break;
        }
      }
      const CUtensorMap* mA = U.grp ? &tmA1 : &tmA0;
      const CUtensorMap* mB = U.grp ? &tmB1 : &tmB0;
      const CUtensorMap* mBbig = U.grp ? &tmB1big : &tmB0big;
      const int n_pad = (U.m + 15) & ~15;
      // 64-row boxes for the bulk of a packed token tile, 16-row boxes for the rest
      const int n_big = NMAX >= B_BIG ? n_pad / B_BIG : 0;
      const int wrow = U.grp ? U.fb * TL::FEAT : (a.e_begin + U.e) * a.w_rows0 + U.fb * TL::FEAT;
      const uint32_t bytes = TL::NA * TL::A_BYTES + n_pad * BK * 2;
      const bool gather = U.grp == 0 && a.gather0 != nullptr;
      // rows of gather groups g = lane and g = lane + 32 (four rows each); rows past
      // the tile's valid ones repeat its last row (their columns are never stored)
      int gr[2][4];
      const int n_groups = n_pad / 4;
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int r = (lane + 32 * h) * 4 + j;
          gr[h][j] = gather && r < n_pad ? a.gather0[U.row0 + min(r, U.m - 1)] : 0;
        }
      for (int kb = U.kb0; kb < U.kb1; ++kb) {
        const uint32_t full = smem_u32(&ctrl->full[stage]);
        const uint32_t sa = smem_u32(smem + stage * TL::STAGE_BYTES);
        const uint32_t sb = sa + TL::NA * TL::A_BYTES;
        auto issue = [&]() {  // lane 0: arm the stage barrier, load the tiles
          mbar_arrive_expect_tx(full, bytes);
#pragma unroll
          for (int t = 0; t < TL::NA; ++t) {
            const int r = wrow + t * a.up_off;
            const uint16_t* ap = U.grp ? a.a1_packed : a.a0_packed;
            if (PK)  // tile (r / 128, kb): 8192 bf16 per tile
              bulk_load_tile(sa + t * TL::A_BYTES,
                             ap + ((size_t)(r / BM) * kblocks + kb) * (BM * BK), full);
            else
              tma_load_2d(sa + t * TL::A_BYTES, mA, kb * KE, r, full);
          }
          const uint8_t* bt = U.grp ? a.b_tiled1 : a.b_tiled0;
          if (bt) {  // tile-packed rows: block kb of the tile, already swizzled
            const int eg = U.grp ? 0 : a.e_begin + U.e;
            bulk_load(sb,
                      bt + (size_t)(U.row0 + 16 * eg) * a.K * (F8 ? 1 : 2) +
                          (size_t)kb * n_pad * 128,
                      (uint32_t)n_pad * 128, full);
          } else if (!gather) {
            for (int i = 0; i < n_big; ++i)
              tma_load_2d(sb + i * (B_BIG * BK * 2), mBbig, kb * KE, U.row0 + i * B_BIG, full);
            for (int i = n_big * (B_BIG / B_BOX); i < n_pad / B_BOX; ++i)
              tma_load_2d(sb + i * (B_BOX * BK * 2), mB, kb * KE, U.row0 + i * B_BOX, full);
          }
        };
        int got = 1;
        if (lane == 0) {
          got = wait_bounded(smem_u32(&ctrl->empty[stage]), phase ^ 1, abort_flag, err,
                             a.wait_limit_ns)
                    ? 1
                    : 0;
          if (got && blockIdx.x == 0 && fills == a.stall_fill) got = 2;  // skip this fill
          if (got == 1) issue();
        }
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) {
          ok = false;
          break;
        }
        if (gather && got == 1) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int g = lane + 32 * h;
            if (g < n_groups)
              tma_gather4(sb + g * (4 * BK * 2), mB, kb * KE, gr[h][0], gr[h][1], gr[h][2],
                          gr[h][3], full);
          }
        }
        ++fills;
        if (++stage == TL::STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
    }
    if (!ok && lane == 0) {
      // let the copies already issued land before the CTA can exit
      for (int s = 0; s < TL::STAGES; ++s) {
        if (fills <= s) continue;
        const long f = s + ((fills - 1 - s) / TL::STAGES) * TL::STAGES;  // last fill of stage s
        if (blockIdx.x == 0 && f == a.stall_fill) continue;  // never issued
        const uint32_t par = (uint32_t)((f / TL::STAGES) & 1);
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(smem_u32(&ctrl->full[s]), par) &&
               global_timer_ns() - t0 < a.wait_limit_ns) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true, issued = false;
      for (int j = 0; ok; ++j) {  // j: units of this CTA so far (accumulator j % ACC_STAGES)
        const int u = next_unit(j);
        if (u < 0) {
          ok = false;
          break;
        }
        if (u >= total_units) break;
        const Unit U = decode_unit<NMAX>(u, tile_off, row_off, a, units1, kblocks);
        const int n_pad = (U.m + 15) & ~15;
        const uint32_t idesc = MX ? idesc_mx(n_pad) : F8 ? idesc_e4m3(n_pad) : idesc_bf16(n_pad);
        const int as = j % TL::ACC_STAGES;
        const uint32_t acc_par = (uint32_t)((j / TL::ACC_STAGES) & 1);
        if (!wait_bounded(smem_u32(&ctrl->acc_empty[as]), acc_par ^ 1, abort_flag, err,
                          a.wait_limit_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(as * TL::ACC_COLS);
        for (int kb = U.kb0; kb < U.kb1; ++kb) {
          if (!wait_bounded(smem_u32(&ctrl->full[stage]), phase, abort_flag, err,
                            a.wait_limit_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (kb == U.kb0) trace_put(a, u, 1, global_timer_ns());
          const uint32_t sa = smem_u32(smem + stage * TL::STAGE_BYTES);
          const uint32_t sb = sa + TL::NA * TL::A_BYTES;
          if constexpr (MX) {
            // the stage's scale images -> its TMEM scale columns: A tile t at
            // sfc + 4 t, token rows 128 c .. at sfc + 4 (NA + c); the copies run
            // before the MMAs below (same issuing thread), and the stage's commit
            // covers them before the producer rewrites the images
            const uint32_t sfs = sa + TL::SF_OFF;
            const uint32_t sfc = tmem_base + (uint32_t)(TL::SF_COL0 + stage * TL::SF_COLS);
#pragma unroll
            for (int t = 0; t < TL::NA; ++t) sf_copy(sfc + 4 * t, sfs + t * 512);
            for (int c = 0; c < (n_pad + 127) / 128; ++c)
              sf_copy(sfc + 4 * (TL::NA + c), sfs + (TL::NA + c) * 512);
            const uint32_t sfb = sfc + 4 * TL::NA;
#pragma unroll
            for (int k = 0; k < BK / UMMA_K; ++k) {
              const uint32_t acc = (kb > U.kb0 || k > 0) ? 1u : 0u;
              const uint64_t bdesc = sdesc(sb + k * UMMA_K * 2);
              mma_mx(d, sdesc(sa + k * UMMA_K * 2), bdesc, idesc, sfc, sfb, acc);
              if (TL::TWO_ACC)
                mma_mx(d + NMAX, sdesc(sa + TL::A_BYTES + k * UMMA_K * 2), bdesc, idesc, sfc + 4,
                       sfb, acc);
            }
          } else {
#pragma unroll
            for (int k = 0; k < BK / UMMA_K; ++k) {
              const uint32_t acc = (kb > U.kb0 || k > 0) ? 1u : 0u;
              const uint64_t bdesc = sdesc(sb + k * UMMA_K * 2);
              mma_op<F8>(d, sdesc(sa + k * UMMA_K * 2), bdesc, idesc, acc);
              if (TL::TWO_ACC)
                mma_op<F8>(d + NMAX, sdesc(sa + TL::A_BYTES + k * UMMA_K * 2), bdesc, idesc, acc);
              if (MODE == MODE_SPLIT3) {  // the lower planes add into the same accumulator
                mma_op<F8>(d, sdesc(sa + TL::A_BYTES + k * UMMA_K * 2), bdesc, idesc, 1u);
                mma_op<F8>(d, sdesc(sa + 2 * TL::A_BYTES + k * UMMA_K * 2), bdesc, idesc, 1u);
              }
            }
          }
          issued = true;
          mma_commit(smem_u32(&ctrl->empty[stage]));
          if (++stage == TL::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(smem_u32(&ctrl->acc_full[as]));
      }
      if (!ok && issued) {
        // wait (bounded) for the MMAs already issued before TMEM is freed
        mma_commit(smem_u32(&ctrl->drain));
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(smem_u32(&ctrl->drain), 0) &&
               global_timer_ns() - t0 < a.wait_limit_ns) {
        }
      }
    }
  } else if (MX && warp == EPI_END) {
    // ------------------------------------------------------------------ scale warp
    // Block-scaled FP8 only. Per stage, once the slot is free: the UE8M0
    // exponents of the stage's A tiles and token rows, written as the 512-byte
    // images tcgen05.cp expects (every byte of a word holds the exponent) and
    // made visible to the tensor core's reads, then one arrive on the stage's
    // full barrier (its second arrival besides the producer's). Every SF_KC
    // k-blocks of a unit the warp first stages the next SF_KC exponents of each
    // token row and A tile in shared memory, every lane issuing all the 8-byte
    // loads of its token rows before its first store (one round trip), so the
    // per-stage values come from shared memory. Lane l holds token columns
    // j = 32 g + l of the tile (activation row sf_row[g]; -1 past the valid rows).
    constexpr int NG = MX ? (NMAX + 31) / 32 : 1;
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int j = 0; ok; ++j) {
      int u = 0;
      if (lane == 0) u = next_unit(j);
      u = __shfl_sync(0xffffffffu, u, 0);
      if (u < 0 || u >= total_units) break;
      const Unit U = decode_unit<NMAX>(u, tile_off, row_off, a, units1, kblocks);
      const int wrow = U.grp ? U.fb * TL::FEAT : (a.e_begin + U.e) * a.w_rows0 + U.fb * TL::FEAT;
      int sf_row[NG];
      {
        const int32_t* bidx = U.grp ? nullptr : a.b_scale_idx0;
#pragma unroll
        for (int g = 0; g < NG; ++g) {
          const int j = 32 * g + lane;
          sf_row[g] = j < U.m ? (bidx ? bidx[U.row0 + j] : U.row0 + j) : -1;
        }
      }
      for (int kb = U.kb0; kb < U.kb1; ++kb) {
        uint32_t sfa[TL::NA], sfb[NG];
        const int kbl = (kb - U.kb0) % TL::SF_KC;
        if (kbl == 0) {
          const int kc = min(TL::SF_KC, U.kb1 - kb);
          const uint8_t* asf = U.grp ? a.a_sf1 : a.a_sf0;
          const uint8_t* bsf = U.grp ? a.b_sf1 : a.b_sf0;
          const long ld = U.grp ? a.b_sf_ld1 : a.b_sf_ld0;
          uint32_t av[TL::NA];
#pragma unroll
          for (int t = 0; t < TL::NA; ++t)
            av[t] = lane < kc ? asf[(size_t)((wrow + t * a.up_off) / BM) * kblocks + kb + lane]
                              : 0u;
          if ((ld & 7) == 0 && ((uintptr_t)bsf & 7) == 0 && (kb & 7) == 0) {
            // rows of 8-byte multiples: bytes [kb, kb + 8 ceil(kc / 8)) of a row
            // stay inside it (kb + kc <= K / 128 <= ld)
            uint2 v[NG][TL::SF_KC / 8];
#pragma unroll
            for (int g = 0; g < NG; ++g)
#pragma unroll
              for (int i = 0; i < TL::SF_KC / 8; ++i)
                v[g][i] = sf_row[g] >= 0 && 8 * i < kc
                              ? *reinterpret_cast<const uint2*>(bsf + (size_t)sf_row[g] * ld +
                                                                kb + 8 * i)
                              : make_uint2(0u, 0u);
#pragma unroll
            for (int g = 0; g < NG; ++g) {
              uint32_t* d = reinterpret_cast<uint32_t*>(sf_stg + (32 * g + lane) * TL::SF_STR);
#pragma unroll
              for (int i = 0; i < TL::SF_KC / 8; ++i)
                if (sf_row[g] >= 0 && 8 * i < kc) {
                  d[2 * i] = v[g][i].x;
                  d[2 * i + 1] = v[g][i].y;
                }
            }
          } else {  // any other stride: byte loads
#pragma unroll
            for (int g = 0; g < NG; ++g)
              if (sf_row[g] >= 0)
                for (int i = 0; i < kc; ++i)
                  sf_stg[(32 * g + lane) * TL::SF_STR + i] = bsf[(size_t)sf_row[g] * ld + kb + i];
          }
          if (lane < kc) {
#pragma unroll
            for (int t = 0; t < TL::NA; ++t) sf_stg[TL::SF_STG_A + t * TL::SF_KC + lane] = av[t];
          }
          __syncwarp();
        }
#pragma unroll
        for (int t = 0; t < TL::NA; ++t) sfa[t] = sf_stg[TL::SF_STG_A + t * TL::SF_KC + kbl];
#pragma unroll
        for (int g = 0; g < NG; ++g)
          sfb[g] = sf_row[g] >= 0 ? sf_stg[(32 * g + lane) * TL::SF_STR + kbl] : 127u;
        int got = 1;
        if (lane == 0)
          got = wait_bounded(smem_u32(&ctrl->empty[stage]), phase ^ 1, abort_flag, err,
                             a.wait_limit_ns)
                    ? 1
                    : 0;
        got = __shfl_sync(0xffffffffu, got, 0);
        if (!got) {
          ok = false;
          break;
        }
        uint8_t* sf = smem + stage * TL::STAGE_BYTES + TL::SF_OFF;
#pragma unroll
        for (int t = 0; t < TL::NA; ++t) {
          const uint32_t v = sfa[t] * 0x01010101u;
          *reinterpret_cast<uint4*>(sf + t * 512 + lane * 16) = make_uint4(v, v, v, v);
        }
#pragma unroll
        for (int c = 0; c < TL::SF_CB; ++c) {
          uint32_t w[4];
#pragma unroll
          for (int q = 0; q < 4; ++q)
            w[q] = (4 * c + q < NG ? sfb[min(4 * c + q, NG - 1)] : 127u) * 0x01010101u;
          *reinterpret_cast<uint4*>(sf + (TL::NA + c) * 512 + lane * 16) =
              make_uint4(w[0], w[1], w[2], w[3]);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&ctrl->full[stage]));
        if (++stage == TL::STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
    }
  } else if (has_pack(MODE, Q) && warp >= EPI_END) {
    // ------------------------------------------------------------------ pack warps
    // Fused dispatch: packed row r of group 0 = source row pack_rst[r]. A warp
    // takes PACK_ROWS consecutive packed rows from the global counter, copies
    // them with 16-byte vectors (each lane two columns of every row in flight
    // at once), then adds the rows to their experts' counts with release
    // semantics. Rows with a source index outside the source matrix are left
    // unwritten and latched as MOE_ERR_DEVICE_CHECK; they are still counted.
    //
    // Token-major form (pack_slot non-null; the shared expert's units run first,
    // so the routed units' waits for whole experts fall behind them): a warp
    // takes TPC consecutive tokens, loads each token row once and stores it to
    // the packed rows of all its pack_k slots, lane s holding slot s's
    // destination; x is read once instead of once per slot. A slot row outside
    // this launch's rows is skipped and latched as MOE_ERR_DEVICE_CHECK (its
    // expert's count then stays short and the producer's bounded wait expires).
    if (a.pack_dst && a.pack_slot) {
      const int r_begin = row_off[0], r_end = row_off[a.n_exp];
      const int vpr = a.K * (F8 ? 1 : 2) / 16;  // 16-byte vectors per row
      const int kk = a.pack_k;                  // 1..32 (checked on the host)
      const int tpc = min(PACK_ROWS, 32 / kk);  // tokens per chunk: tpc * kk <= 32
      const int n_tok = a.pack_src_rows;
      const int n_chunks = (n_tok + tpc - 1) / tpc;
      const bool tiled = a.b_tiled0 != nullptr;
      while (!*abort_flag) {
        int c = 0;
        if (lane == 0) c = atomicAdd(a.pack_next, 1);
        c = __shfl_sync(0xffffffffu, c, 0);
        if (c >= n_chunks) break;
        const int t0 = c * tpc, nt = min(tpc, n_tok - t0), ns = nt * kk;
        // lane s < ns: slot s (token t0 + s / kk, slot s % kk) -> its expert
        // (binary search over the clamped offsets) and destination: the tile's
        // first 16-byte unit and (row in tile | padded rows << 16), or the row's
        // first unit (row-major); ipk < 0 marks no slot
        int e_s = -1, ipk = -1;
        unsigned long long d0 = 0;
        if (lane < ns) {
          const int r = a.pack_slot[(size_t)t0 * kk + lane];
          if (r >= r_begin && r < r_end) {
            int lo = 0, hi = a.n_exp - 1;
            while (lo < hi) {
              const int mid = (lo + hi + 1) >> 1;
              if (row_off[mid] <= r) lo = mid;
              else hi = mid - 1;
            }
            e_s = lo;
            if (tiled) {
              const TiledRow w = tiled_row(r, a.e_begin + lo, row_off[lo],
                                           row_off[lo + 1] - row_off[lo], NMAX, vpr);
              d0 = w.tile16;
              ipk = w.i | (w.n_pad << 16);
            } else {
              d0 = (unsigned long long)r * vpr;
              ipk = 0;
            }
          } else {
            atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
          }
        }
        // the trip count is the same for every lane (the slot destinations are
        // shuffled inside the loop); lanes past the row's end only skip their
        // loads and stores
        for (int vb = 0; vb < vpr; vb += 64) {
          const int v0 = vb + lane;
          uint4 val[PACK_ROWS][2];
#pragma unroll
          for (int q = 0; q < PACK_ROWS; ++q)
#pragma unroll
            for (int h = 0; h < 2; ++h)
              if (q < nt && v0 + 32 * h < vpr)
                val[q][h] = a.pack_src[(size_t)(t0 + q) * vpr + v0 + 32 * h];
#pragma unroll
          for (int q = 0; q < PACK_ROWS; ++q) {
            if (q >= nt) break;
            for (int j = 0; j < kk; ++j) {
              const int sl = q * kk + j;
              const unsigned long long ds = __shfl_sync(0xffffffffu, d0, sl);
              const int ip = __shfl_sync(0xffffffffu, ipk, sl);
              if (ip < 0) continue;
              TiledRow w;
              w.tile16 = ds;
              w.i = ip & 0xffff;
              w.n_pad = ip >> 16;
#pragma unroll
              for (int h = 0; h < 2; ++h)
                if (v0 + 32 * h < vpr)
                  a.pack_dst[tiled ? w.chunk16(v0 + 32 * h) : ds + v0 + 32 * h] = val[q][h];
            }
          }
        }
        __threadfence();
        fence_proxy_async_global();
        __syncwarp();
        if (e_s >= 0)
          asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(a.pack_ready + e_s), "r"(1)
                       : "memory");
      }
    } else if (a.pack_dst) {
      const int r_begin = row_off[0], r_end = row_off[a.n_exp];
      const int vpr = a.K * (F8 ? 1 : 2) / 16;  // 16-byte vectors per row
      const int n_chunks = (r_end - r_begin + PACK_ROWS - 1) / PACK_ROWS;
      while (!*abort_flag) {
        int c = 0;
        if (lane == 0) c = atomicAdd(a.pack_next, 1);
        c = __shfl_sync(0xffffffffu, c, 0);
        if (c >= n_chunks) break;
        const int r0 = r_begin + c * PACK_ROWS, nr = min(PACK_ROWS, r_end - r0);
        int src = -1;
        if (lane < nr) {
          const int t = a.pack_rst[r0 + lane];
          if (t >= 0 && t < a.pack_src_rows) src = t;
          else atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
        }
        int tq[PACK_ROWS];
#pragma unroll
        for (int q = 0; q < PACK_ROWS; ++q) tq[q] = __shfl_sync(0xffffffffu, src, q);
        // tile-packed destination: lane q < nr places row r0 + q (its expert by
        // binary search over the clamped offsets), every lane gets the result
        TiledRow dq[PACK_ROWS];
        if (a.b_tiled0) {
          unsigned long long tb = 0;
          int ti = 0, tn = 0;
          if (lane < nr) {
            const int r = r0 + lane;
            int lo = 0, hi = a.n_exp - 1;
            while (lo < hi) {
              const int mid = (lo + hi + 1) >> 1;
              if (row_off[mid] <= r) lo = mid;
              else hi = mid - 1;
            }
            const TiledRow w =
                tiled_row(r, a.e_begin + lo, row_off[lo], row_off[lo + 1] - row_off[lo], NMAX, vpr);
            tb = w.tile16;
            ti = w.i;
            tn = w.n_pad;
          }
#pragma unroll
          for (int q = 0; q < PACK_ROWS; ++q) {
            dq[q].tile16 = __shfl_sync(0xffffffffu, tb, q);
            dq[q].i = __shfl_sync(0xffffffffu, ti, q);
            dq[q].n_pad = __shfl_sync(0xffffffffu, tn, q);
          }
        }
        for (int v0 = lane; v0 < vpr; v0 += 64) {
          uint4 val[PACK_ROWS][2];
#pragma unroll
          for (int q = 0; q < PACK_ROWS; ++q)
#pragma unroll
            for (int h = 0; h < 2; ++h)
              if (tq[q] >= 0 && v0 + 32 * h < vpr)
                val[q][h] = a.pack_src[(size_t)tq[q] * vpr + v0 + 32 * h];
#pragma unroll
          for (int q = 0; q < PACK_ROWS; ++q)
#pragma unroll
            for (int h = 0; h < 2; ++h)
              if (tq[q] >= 0 && v0 + 32 * h < vpr)
                a.pack_dst[a.b_tiled0 ? dq[q].chunk16(v0 + 32 * h)
                                      : (size_t)(r0 + q) * vpr + v0 + 32 * h] = val[q][h];
        }
        __threadfence();
        fence_proxy_async_global();
        __syncwarp();
        if (lane == 0) {
          int lo = 0, hi = a.n_exp - 1;  // the expert of row r0: last e with row_off[e] <= r0
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (row_off[mid] <= r0) lo = mid;
            else hi = mid - 1;
          }
          for (int e = lo, r = r0; r < r0 + nr; ++e) {
            const int end = min(row_off[e + 1], r0 + nr);
            if (end > r) {
              asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(a.pack_ready + e),
                           "r"(end - r)
                           : "memory");
              r = end;
            }
          }
        }
      }
    }
  } else if (warp < EPI_END) {
    // ------------------------------------------------------------------ epilogue
    // EPI / 4 warps per TMEM lane quarter: warp w reads lanes 32 * (w % 4) ..
    // + 31 and the 16-column chunks c0 = 16 * half, 16 * half + 16 * EPI / 4,
    // ... of a unit.
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int half = (warp - 2) >> 2;  // this warp's turn among its quarter's EPI / 4
    for (int j = 0;; ++j) {
      int u = 0;
      if (lane == 0) u = next_unit(j);
      u = __shfl_sync(0xffffffffu, u, 0);
      if (u < 0 || u >= total_units) break;
      const Unit U = decode_unit<NMAX>(u, tile_off, row_off, a, units1, kblocks);
      const int as = j % TL::ACC_STAGES;
      const uint32_t acc_par = (uint32_t)((j / TL::ACC_STAGES) & 1);
      const int f = U.fb * TL::FEAT + q * 32 + lane;
      const size_t o = (size_t)U.row0 * a.out_ld + f;
      // FP8: the scales of this thread's weight row(s); the token columns' scales
      // are fetched with the other per-column data below
      float sa0 = 1.f, sa1 = 1.f;
      const float* bsc = nullptr;
      const int32_t* bidx = nullptr;
      constexpr bool RS = F8 && !MX;  // row scales applied here
      if (RS) {
        const float* asc = U.grp ? a.a_scale1 : a.a_scale0;
        const int wr = (U.grp ? 0 : (a.e_begin + U.e) * a.w_rows0) + f;
        sa0 = asc[wr];
        if (TL::NA == 2) sa1 = asc[wr + a.up_off];
        bsc = U.grp ? a.b_scale1 : a.b_scale0;
        bidx = U.grp ? nullptr : a.b_scale_idx0;
      }
      void* out = U.grp ? static_cast<void*>(static_cast<float*>(a.out1) + U.split * a.split_stride)
                        : a.out0;
      // SwiGLU with tile-packed h: this thread's element of block f / 64 of the
      // unit's tile (the tile of n_pad rows at padded row row0 + 16 * expert)
      const bool h_tiled = SWIGLU && (U.grp ? a.out_tiled1 : a.out_tiled0);
      const int h_pad = (U.m + 15) & ~15;
      const size_t h_blk = (size_t)(U.row0 + 16 * (U.grp ? 0 : a.e_begin + U.e)) * a.out_ld +
                           (size_t)(f >> 6) * h_pad * 64 + (f & 7);
      const int h_chk = (f & 63) >> 3;
      float* comb = U.grp ? a.comb_out1 : a.comb_out0;
      const int32_t* ctok = U.grp ? nullptr : a.comb_tok0;
      const float* cw = U.grp ? nullptr : a.comb_w0;
      // What each column of the unit needs from global memory (the token's FP8
      // scale; with the fused combine its token row and gate weight), loaded
      // for all of this warp's 16-column chunks at once and before the
      // accumulator is complete, so the loads overlap the unit's MMAs: lane
      // l < 16 holds column 16 * half + 16 * (EPI / 4) * i + l of chunk i.
      constexpr bool CBP = MODE == MODE_PLAIN || MODE == MODE_PLAIN2;  // combine possible
      constexpr int CSTEP = 16 * (EPI / 4);
      constexpr int NCH = (NMAX + CSTEP - 1) / CSTEP;  // chunks per warp, at most
      float sbv[NCH], wvv[NCH];
      int tvv[NCH];
      const bool cbx = CBP && comb != nullptr;
#pragma unroll
      for (int i = 0; i < NCH; ++i) {
        const int mc = 16 * half + CSTEP * i + (lane & 15);
        const bool cv = mc < U.m;
        const int br = U.row0 + (cv ? mc : 0);
        sbv[i] = (RS && cv) ? bsc[bidx ? bidx[br] : br] : 1.f;
        wvv[i] = (cbx && cv && cw) ? cw[br] : 1.f;
        tvv[i] = (cbx && cv && ctok) ? ctok[br] : br;
      }
      if (!wait_bounded(smem_u32(&ctrl->acc_full[as]), acc_par, abort_flag, err, a.wait_limit_ns))
        break;
      if (warp == 2 && lane == 0) trace_put(a, u, 2, global_timer_ns());
      tc_fence_after();
      const uint32_t tq = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(as * TL::ACC_COLS);
      // The unit's columns; CB (the fused combine) is a compile-time copy of the
      // loop so the plain stores keep their unrolled form. The other lanes read
      // a chunk's per-column values from lanes 0-15 with a shuffle.
      auto columns = [&](auto cb_tag) {
        constexpr bool CB = decltype(cb_tag)::value;
#pragma unroll
        for (int ci = 0; ci < NCH; ++ci) {
          const int c0 = 16 * half + CSTEP * ci;
          if (c0 >= U.m) break;
          const float sb_l = sbv[ci], w_l = wvv[ci];
          const int t_l = tvv[ci];
          uint32_t g[16];
          tmem_ld16(tq + c0, g);
          if constexpr (SWIGLU) {
            uint32_t v[16];
            tmem_ld16(tq + NMAX + c0, v);
            tmem_wait_ld();
            // the chunk's 16 SwiGLU values first, in straight-line code (16
            // independent chains the scheduler can interleave), then the stores
            // of the valid columns
            uint32_t hb[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float sb = RS ? __shfl_sync(0xffffffffu, sb_l, i) : 1.f;
              const float gv = __uint_as_float(g[i]) * (sa0 * sb);
              const float uv = __uint_as_float(v[i]) * (sa1 * sb);
              hb[i] = float_to_bf16_bits(silu_mul(gv, uv));
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              if (c0 + i < U.m) {
                // tile-packed h: token column c = c0 + i is row c of the tile;
                // this thread's feature f is element f % 8 of 16-byte chunk
                // (f % 64) / 8 of block f / 64
                const int c = c0 + i;
                const size_t idx = h_tiled ? h_blk + (size_t)c * 64 + ((h_chk ^ (c & 7)) << 3)
                                           : o + (size_t)c * a.out_ld;
                static_cast<uint16_t*>(out)[idx] = (uint16_t)hb[i];
              }
            }
          } else if constexpr (MODE == MODE_PLAIN2) {
            uint32_t v[16];
            tmem_ld16(tq + NMAX + c0, v);  // the second tile: features f + 128
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float sb = RS ? __shfl_sync(0xffffffffu, sb_l, i) : 1.f;
              const float wv = CB ? __shfl_sync(0xffffffffu, w_l, i) : 1.f;
              const int tv = CB ? __shfl_sync(0xffffffffu, t_l, i) : 0;
              if (c0 + i < U.m) {
                const float y0 = __uint_as_float(g[i]) * (sa0 * sb);
                const float y1 = __uint_as_float(v[i]) * (sa1 * sb);
                if constexpr (CB) {
                  float* d = comb + (size_t)tv * a.out_ld + f;
                  atomicAdd(d, wv * y0);
                  atomicAdd(d + BM, wv * y1);
                } else {
                  float* y = static_cast<float*>(out) + o + (size_t)(c0 + i) * a.out_ld;
                  y[0] = y0;
                  y[BM] = y1;
                }
              }
            }
          } else {
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float sb = RS ? __shfl_sync(0xffffffffu, sb_l, i) : 1.f;
              const float wv = CB ? __shfl_sync(0xffffffffu, w_l, i) : 1.f;
              const int tv = CB ? __shfl_sync(0xffffffffu, t_l, i) : 0;
              if (c0 + i < U.m) {
                const float y0 = __uint_as_float(g[i]) * (sa0 * sb);
                if constexpr (CB) {
                  atomicAdd(comb + (size_t)tv * a.out_ld + f, wv * y0);
                } else {
                  static_cast<float*>(out)[o + (size_t)(c0 + i) * a.out_ld] = y0;
                }
              }
            }
          }
        }
      };
      if constexpr (MODE == MODE_PLAIN || MODE == MODE_PLAIN2) {
        if (comb) {
          columns(std::true_type{});
        } else {
          columns(std::false_type{});
        }
      } else {
        columns(std::false_type{});
      }
      tc_fence_before();
      __syncwarp();
      if (warp == 2 && lane == 0) {
        trace_put(a, u, 3, global_timer_ns());
        trace_put(a, u, 4,
                  (unsigned long long)sm_id() | ((unsigned long long)U.m << 16) |
                      ((unsigned long long)(U.e + 1024 * U.grp) << 32) |
                      ((unsigned long long)U.fb << 48));
      }
      if (lane == 0) mbar_arrive(smem_u32(&ctrl->acc_empty[as]));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TL::TMEM_COLS)
                 : "memory");
  }
  if (a.sched && threadIdx.x == 0) {
    // every unit index this CTA will ever take has been taken: the last CTA
    // out resets the scheduler for the next launch
    __threadfence();
    if (atomicAdd(a.sched + 1, 1) == (int)gridDim.x - 1) {
      atomicExch(a.sched, 0);
      atomicExch(a.sched + 1, 0);
      if (a.pack_dst) {  // and the fused dispatch's counters
        atomicExch(a.pack_next, 0);
        for (int e = 0; e < a.n_exp; ++e) atomicExch(a.pack_ready + e, 0);
      }
    }
  }
}

// ------------------------------------------------------------------ host side

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 row-major tensor [outer, inner] with a (box_inner x box_outer) box, 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint32_t box_inner,
              uint32_t box_outer) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Barrier-wait limit and injected stall of the expert-FFN launches: WAIT_LIMIT_NS
// and none, except inside moe_testing_expert_ffn_stall (one host thread).
uint64_t g_wait_limit_ns = WAIT_LIMIT_NS;
long g_stall_fill = -1;

template <int MODE, int NMAX, bool MX>
size_t gemm_smem_bytes(int n_exp) {
  using TL = Tile<MODE, NMAX, MX>;
  return 1024 + (size_t)TL::STAGES * TL::STAGE_BYTES + TL::SF_STG_BYTES + sizeof(Ctrl) +
         2 * sizeof(int) * (n_exp + 1);
}

template <int MODE, int NMAX, int Q, bool PK>
moe_status launch_gemm(const CUtensorMap& A0, const CUtensorMap& B0, const CUtensorMap& A1,
                       const CUtensorMap& B1, const CUtensorMap& B0big, const CUtensorMap& B1big,
                       const GemmArgs& args, cudaStream_t s) {
  const size_t smem = gemm_smem_bytes<MODE, NMAX, Q == Q_BLOCK>(args.n_exp);
  if (smem > 227 * 1024) return MOE_ERR_UNSUPPORTED;
  if (cudaFuncSetAttribute(grouped_gemm_kernel<MODE, NMAX, Q, PK>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return MOE_ERR_CUDA;
  grouped_gemm_kernel<MODE, NMAX, Q, PK><<<num_sms(), threads_of(MODE, Q), smem, s>>>(A0, B0, A1, B1,
                                                                              B0big, B1big, args);
  note_launch();
  return launch_status();
}

// Row-major [rows, cols] operand map with (one 128-byte row segment) x box_rows
// boxes: bf16 elements, or e4m3 bytes for the FP8 form.
template <bool F8>
bool make_rows_map(CUtensorMap* m, const void* ptr, uint64_t cols, uint64_t rows,
                   uint32_t box_rows) {
  if (!F8) return make_map(m, ptr, cols, rows, BK, box_rows);
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols};
  cuuint32_t box[2] = {2 * BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// PK: weights in the tile-packed layout, fetched by bulk copies (a separate
// instantiation: a runtime choice between the two weight paths in the
// producer's loop measured 12 % slower decode GEMM2 even when never taken).
template <int NMAX, int Q, bool PK>
moe_status run_ffn(const FfnGroup& g0, const FfnGroup* g1, int H, int I, cudaStream_t s,
                   cudaEvent_t after_gemm1) {
  constexpr bool F8 = Q != Q_BF16;
  constexpr bool MX = Q == Q_BLOCK;
  CUtensorMap a1, b1, a2, b2, sa1, sb1, sa2, sb2, b1big, b2big, sb1big, sb2big;
  // with a fused dispatch GEMM1 reads token rows of x by index: a one-row box
  const bool gather = g0.gather != nullptr;
  const bool pk = PK;
  if (g0.packed != PK || (F8 && PK)) return MOE_ERR_UNSUPPORTED;  // packed tiles are bf16 only
  const uint64_t xr = gather ? g0.x_rows : g0.rows;
  // tile-packed token rows: bf16 (x, h) or row-scaled e4m3 (x, hq), x written
  // for this launch's tile
  if (g0.x_tiled || g0.h_tiled || g0.hq_tiled ||
      (g1 && (g1->x_tiled || g1->h_tiled || g1->hq_tiled))) {
    if (MX || (F8 && (g0.h_tiled || (g1 && g1->h_tiled))) ||
        (!F8 && (g0.hq_tiled || (g1 && g1->hq_tiled))) ||
        (g0.x_tiled && (gather || g0.x_tile != NMAX)) ||
        (g1 && g1->x_tiled && g1->x_tile != NMAX))
      return MOE_ERR_UNSUPPORTED;
  }
  // GEMM2's token operand: h (bf16), or its e4m3 copy hq in the FP8 form
  const void* h0 = F8 ? static_cast<const void*>(g0.hq) : static_cast<const void*>(g0.h);
  if (!make_rows_map<F8>(&a1, g0.W13, H, (uint64_t)g0.n_experts * 2 * I, BM) ||
      !make_rows_map<F8>(&b1, g0.x, H, xr, gather ? 1 : B_BOX) ||
      !make_rows_map<F8>(&a2, g0.W2, I, (uint64_t)g0.n_experts * H, BM) ||
      !make_rows_map<F8>(&b2, h0, I, g0.rows, B_BOX) ||
      !make_rows_map<F8>(&b1big, g0.x, H, xr, gather ? 1 : B_BIG) ||
      !make_rows_map<F8>(&b2big, h0, I, g0.rows, B_BIG))
    return MOE_ERR_CUDA;
  if (g1) {
    if (g1->packed != g0.packed || g1->fp8 != g0.fp8 || g1->fp8_block != g0.fp8_block)
      return MOE_ERR_INVALID_ARG;
    const void* h1 = F8 ? static_cast<const void*>(g1->hq) : static_cast<const void*>(g1->h);
    if (!make_rows_map<F8>(&sa1, g1->W13, H, (uint64_t)2 * I, BM) ||
        !make_rows_map<F8>(&sb1, g1->x, H, g1->rows, B_BOX) ||
        !make_rows_map<F8>(&sa2, g1->W2, I, (uint64_t)H, BM) ||
        !make_rows_map<F8>(&sb2, h1, I, g1->rows, B_BOX) ||
        !make_rows_map<F8>(&sb1big, g1->x, H, g1->rows, B_BIG) ||
        !make_rows_map<F8>(&sb2big, h1, I, g1->rows, B_BIG))
      return MOE_ERR_CUDA;
  } else {
    sa1 = a1;  // unused: group 1 is empty
    sb1 = b1;
    sa2 = a2;
    sb2 = b2;
    sb1big = b1big;
    sb2big = b2big;
  }
  GemmArgs args{};
  args.k_splits = 1;
  args.a0_packed = pk ? static_cast<const uint16_t*>(g0.W13) : nullptr;
  args.a1_packed = (pk && g1) ? static_cast<const uint16_t*>(g1->W13) : nullptr;
  args.wait_limit_ns = g_wait_limit_ns;
  args.stall_fill = g_stall_fill;
  args.sched = g0.sched;  // GEMM1 and GEMM2 run one after the other on `s`
  args.offsets = g0.offsets;
  args.rows0 = g0.rows;
  args.e_begin = g0.e_begin;
  args.n_exp = g0.e_end - g0.e_begin;
  args.rows1 = g1 ? g1->rows : 0;
  args.err = device_error_word();
  // GEMM1 + SwiGLU: h = silu(x Wg^T) * (x Wu^T)
  args.gather0 = g0.gather;
  args.K = H;
  args.n_fb = I / BM;
  args.w_rows0 = 2 * I;
  args.up_off = I;
  args.out0 = g0.h;
  args.out1 = g1 ? g1->h : nullptr;
  args.out_ld = I;
  if (F8 && !MX) {
    args.a_scale0 = g0.W13_scale;
    args.a_scale1 = g1 ? g1->W13_scale : nullptr;
    args.b_scale0 = g0.x_scale;
    args.b_scale1 = g1 ? g1->x_scale : nullptr;
    args.b_scale_idx0 = g0.x_scale_idx;
  }
  if (MX) {
    args.a_sf0 = g0.W13_sf;
    args.a_sf1 = g1 ? g1->W13_sf : nullptr;
    args.b_sf0 = g0.x_sf;
    args.b_sf_ld0 = g0.x_sf_ld;
    args.b_sf1 = g1 ? g1->x_sf : nullptr;
    args.b_sf_ld1 = g1 ? g1->x_sf_ld : 0;
    args.b_scale_idx0 = g0.x_scale_idx;
  }
  if (g0.pack_src) {  // the dispatch copy inside GEMM1 (needs the dynamic scheduler's reset)
    if (gather || MX || !g0.sched || !g0.pack_rst || !g0.pack_next || !g0.pack_ready)
      return MOE_ERR_UNSUPPORTED;
    args.pack_src = static_cast<const uint4*>(g0.pack_src);
    args.pack_dst = static_cast<uint4*>(const_cast<void*>(g0.x));
    args.pack_rst = g0.pack_rst;
    args.pack_src_rows = g0.pack_src_rows;
    args.pack_next = g0.pack_next;
    args.pack_ready = g0.pack_ready;
    // token-major only behind the shared expert's units: without them the
    // routed units would wait for the whole copy instead of expert by expert
    if (g1 && g0.pack_slot && g0.pack_k >= 1 && g0.pack_k <= 32) {
      args.pack_slot = g0.pack_slot;
      args.pack_k = g0.pack_k;
    }
  }
  const bool trace2 = g0.trace && g0.trace_gemm == 2;  // the trace is GEMM2's
  args.trace = trace2 ? nullptr : g0.trace;
  args.trace_cap = args.trace ? g0.trace_cap : 0;
  args.b_tiled0 = g0.x_tiled ? static_cast<const uint8_t*>(g0.x) : nullptr;
  args.b_tiled1 = (g1 && g1->x_tiled) ? static_cast<const uint8_t*>(g1->x) : nullptr;
  args.out_tiled0 = g0.h_tiled;
  args.out_tiled1 = g1 && g1->h_tiled;
  moe_status st =
      launch_gemm<MODE_SWIGLU, NMAX, Q, PK>(a1, b1, sa1, sb1, b1big, sb1big, args, s);
  if (st != MOE_OK) return st;
  if (MX) {  // h of every packed row -> e4m3 in 1 x 128 blocks: GEMM2's operand
    MOE_STATUS_TRY(launch_quantize_blocks(g0.h, g0.rows, I, g0.hq, g0.hsf, g0.h_sf_ld, s));
    if (g1)
      MOE_STATUS_TRY(launch_quantize_blocks(g1->h, g1->rows, I, g1->hq, g1->hsf, g1->h_sf_ld, s));
  } else if (F8) {  // h of every packed row -> e4m3 and its row scale: GEMM2's operand
    if (g0.hq_tiled)  // the rows of this launch's experts, tile-packed
      MOE_STATUS_TRY(launch_quantize_rows(g0.h, g0.rows, I, g0.hq, g0.hs, s, g0.offsets,
                                          g0.e_begin, g0.e_end, NMAX));
    else
      MOE_STATUS_TRY(launch_quantize_rows(g0.h, g0.rows, I, g0.hq, g0.hs, s));
    if (g1 && g1->hq_tiled)
      MOE_STATUS_TRY(launch_quantize_rows(g1->h, g1->rows, I, g1->hq, g1->hs, s, g1->offsets, 0,
                                          1, NMAX));
    else if (g1)
      MOE_STATUS_TRY(launch_quantize_rows(g1->h, g1->rows, I, g1->hq, g1->hs, s));
  }
  if (after_gemm1 && cudaEventRecord(after_gemm1, s) != cudaSuccess) return MOE_ERR_CUDA;
  args.gather0 = nullptr;  // GEMM2 reads h, already in packed row order
  args.b_tiled0 = g0.h_tiled    ? reinterpret_cast<const uint8_t*>(g0.h)
                  : g0.hq_tiled ? static_cast<const uint8_t*>(g0.hq)
                                : nullptr;
  args.b_tiled1 = !g1              ? nullptr
                  : g1->h_tiled  ? reinterpret_cast<const uint8_t*>(g1->h)
                  : g1->hq_tiled ? static_cast<const uint8_t*>(g1->hq)
                                 : nullptr;
  args.out_tiled0 = 0;
  args.out_tiled1 = 0;
  args.pack_src = nullptr;
  args.pack_dst = nullptr;
  args.trace = trace2 ? g0.trace : nullptr;
  args.trace_cap = trace2 ? g0.trace_cap : 0;
  args.a0_packed = pk ? static_cast<const uint16_t*>(g0.W2) : nullptr;
  args.a1_packed = (pk && g1) ? static_cast<const uint16_t*>(g1->W2) : nullptr;
  if (F8 && !MX) {
    args.a_scale0 = g0.W2_scale;
    args.a_scale1 = g1 ? g1->W2_scale : nullptr;
    args.b_scale0 = g0.hs;
    args.b_scale1 = g1 ? g1->hs : nullptr;
    args.b_scale_idx0 = nullptr;
  }
  if (MX) {
    args.a_sf0 = g0.W2_sf;
    args.a_sf1 = g1 ? g1->W2_sf : nullptr;
    args.b_sf0 = g0.hsf;
    args.b_sf_ld0 = g0.h_sf_ld;
    args.b_sf1 = g1 ? g1->hsf : nullptr;
    args.b_sf_ld1 = g1 ? g1->h_sf_ld : 0;
    args.b_scale_idx0 = nullptr;
  }
  args.comb_out0 = g0.comb_out;
  args.comb_tok0 = g0.comb_tok;
  args.comb_w0 = g0.comb_w;
  args.comb_out1 = g1 ? g1->comb_out : nullptr;
  if (g1 && (g1->comb_tok || g1->comb_w)) return MOE_ERR_INVALID_ARG;  // group 1 is dense
  // GEMM2: y = h W2^T (fp32). Two 128-feature weight tiles per unit share one
  // token tile (twice the weight bytes per stage and half the units): measured
  // faster at every tile size since the epilogue's column loads were moved out
  // of the column loop (decode GEMM2 1.14 -> 1.10 ms).
  args.K = I;
  args.w_rows0 = H;
  args.out0 = g0.y;
  args.out1 = g1 ? g1->y : nullptr;
  args.out_ld = H;
  if (H % (2 * BM) == 0) {
    args.n_fb = H / (2 * BM);
    args.up_off = BM;
    return launch_gemm<MODE_PLAIN2, NMAX, Q, PK>(a2, b2, sa2, sb2, b2big, sb2big, args, s);
  }
  args.n_fb = H / BM;
  args.up_off = 0;
  return launch_gemm<MODE_PLAIN, NMAX, Q, PK>(a2, b2, sa2, sb2, b2big, sb2big, args, s);
}

}  // namespace

int ffn_tile_rows(long rows_hint, int n_exp, bool fp8, bool fp8_block) {
  const long per = rows_hint / (n_exp > 0 ? n_exp : 1);
  if (per <= 24) return 32;
  if (per <= 132) return 144;
  return fp8 && fp8_block ? 224 : 256;
}

moe_status launch_expert_ffn_groups(const FfnGroup& routed, const FfnGroup* dense, int H, int I,
                                    int rows_hint, cudaStream_t s, cudaEvent_t after_gemm1) {
  if ((routed.rows == 0 || routed.e_end <= routed.e_begin) && (!dense || dense->rows == 0))
    return MOE_OK;
  const int n_exp = routed.e_end - routed.e_begin;
  const FfnGroup* g1 = (dense && dense->rows > 0) ? dense : nullptr;
  // the token tile (ffn_tile_rows); block-scaled FP8's largest is 224 rows:
  // two 224-column accumulators and the stages' scale columns share TMEM's
  // 512 columns
  // (the tile its rows were written with, for a tile-packed routed group)
  const int tile = routed.x_tile > 0 ? routed.x_tile
                                     : ffn_tile_rows(rows_hint, n_exp, routed.fp8, routed.fp8_block);
  if (routed.fp8 && routed.fp8_block) {
    if (tile == 32) return run_ffn<32, Q_BLOCK, false>(routed, g1, H, I, s, after_gemm1);
    if (tile == 144) return run_ffn<144, Q_BLOCK, false>(routed, g1, H, I, s, after_gemm1);
    return run_ffn<224, Q_BLOCK, false>(routed, g1, H, I, s, after_gemm1);
  }
  if (routed.fp8) {
    if (tile == 32) return run_ffn<32, Q_ROW, false>(routed, g1, H, I, s, after_gemm1);
    if (tile == 144) return run_ffn<144, Q_ROW, false>(routed, g1, H, I, s, after_gemm1);
    return run_ffn<256, Q_ROW, false>(routed, g1, H, I, s, after_gemm1);
  }
  if (routed.packed) {
    if (tile == 32) return run_ffn<32, Q_BF16, true>(routed, g1, H, I, s, after_gemm1);
    if (tile == 144) return run_ffn<144, Q_BF16, true>(routed, g1, H, I, s, after_gemm1);
    return run_ffn<256, Q_BF16, true>(routed, g1, H, I, s, after_gemm1);
  }
  if (tile == 32) return run_ffn<32, Q_BF16, false>(routed, g1, H, I, s, after_gemm1);
  if (tile == 144) return run_ffn<144, Q_BF16, false>(routed, g1, H, I, s, after_gemm1);
  return run_ffn<256, Q_BF16, false>(routed, g1, H, I, s, after_gemm1);
}

int router_tc_splits(int T, int H, int E) {
  const int tiles = ((T + 127) / 128) * (E / BM);
  const int kblocks = H / BK;
  int ks = (2 * 152 + tiles - 1) / tiles;  // about two units per SM
  if (ks > kblocks / 2) ks = kblocks / 2;  // at least two k-blocks per unit
  return ks < 1 ? 1 : ks;
}

moe_status launch_router_tc(int T, int H, int E, const uint16_t* x, const uint16_t* planes,
                            float* partials, int k_splits, cudaStream_t s) {
  if (T == 0) return MOE_OK;
  CUtensorMap A, B, Bbig;
  if (!make_map(&A, planes, H, (uint64_t)3 * E, BK, BM) || !make_map(&B, x, H, T, BK, B_BOX) ||
      !make_map(&Bbig, x, H, T, BK, B_BIG))
    return MOE_ERR_CUDA;
  GemmArgs args{};
  args.wait_limit_ns = WAIT_LIMIT_NS;
  args.stall_fill = -1;
  args.rows1 = T;  // group 1: all tokens; group 0 is empty
  args.K = H;
  args.n_fb = E / BM;
  args.up_off = E;  // plane p of expert row r sits at row p * E + r
  args.k_splits = k_splits;
  args.split_stride = (long)T * E;
  args.out1 = partials;
  args.out_ld = E;
  args.err = device_error_word();
  return launch_gemm<MODE_SPLIT3, 128, Q_BF16, false>(A, B, A, B, Bbig, Bbig, args, s);
}

moe_status launch_expert_ffn_stalled(int rows, int H, int I, int n_experts, const uint16_t* x_perm,
                                     const int32_t* offsets, const uint16_t* W13,
                                     const uint16_t* W2, uint16_t* h, float* y_perm,
                                     long stall_fill, uint64_t wait_limit_ns, cudaStream_t s) {
  g_wait_limit_ns = wait_limit_ns;
  g_stall_fill = stall_fill;
  FfnGroup g{};
  g.x = x_perm;
  g.offsets = offsets;
  g.rows = rows;
  g.n_experts = n_experts;
  g.e_end = n_experts;
  g.W13 = W13;
  g.W2 = W2;
  g.h = h;
  g.y = y_perm;
  const moe_status st = launch_expert_ffn_groups(g, nullptr, H, I, rows, s);
  g_wait_limit_ns = WAIT_LIMIT_NS;
  g_stall_fill = -1;
  return st;
}

moe_status launch_expert_ffn(int rows, int H, int I, int n_experts, int e_begin, int e_end,
                             const uint16_t* x_perm, const int32_t* offsets, const uint16_t* W13,
                             const uint16_t* W2, uint16_t* h, float* y_perm, int rows_hint,
                             cudaStream_t s, cudaEvent_t after_gemm1, bool packed) {
  if (rows == 0 || e_end <= e_begin) return MOE_OK;
  FfnGroup g{};
  g.x = x_perm;
  g.offsets = offsets;
  g.rows = rows;
  g.n_experts = n_experts;
  g.e_begin = e_begin;
  g.e_end = e_end;
  g.W13 = W13;
  g.W2 = W2;
  g.h = h;
  g.y = y_perm;
  g.packed = packed;
  return launch_expert_ffn_groups(g, nullptr, H, I, rows_hint, s, after_gemm1);
}

}  // namespace moe
