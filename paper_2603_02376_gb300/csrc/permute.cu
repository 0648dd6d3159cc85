// Dispatch and combine: the single-GPU form of the paper's two AlltoAll
// exchanges (host MoE listing, Appendix "Static Analysis Example"; unpadded
// variable-size per-peer transfers, Appendix "Workload Details").
//
// Permutation (stable, deterministic, no global atomics deciding order):
//   1. perm_hist:    each CTA takes PERM_TOK consecutive tokens (all k slots)
//                    and counts its entries per expert -> chunk_counts[c][e];
//   2. perm_scan:    one CTA: per expert, exclusive prefix of chunk counts over
//                    chunks -> chunk_base[c][e] and counts[e]; then offsets =
//                    exclusive prefix of counts over experts;
//   3. perm_scatter: each CTA re-walks its entries in (t, j) order; each warp
//                    ranks its 32-entry steps with __match_any_sync, so every
//                    expert's rows come out ordered by (t, j).
// Row copies move 16-byte vectors: dispatch scatters each token row once to
// its k packed rows (x read once); combine gathers the k fp32 expert rows of a
// token and reduces them in fp32 in slot order.
#include "common.cuh"

namespace moe {
namespace {

constexpr int PERM_WARPS = 8;
constexpr int PERM_TOK = 128;  // tokens per permutation chunk

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Per-warp histogram of the warp's share of a chunk. hist: [PERM_WARPS][E] in smem.
// Expert id of entry n, or -1 (and a latched error) if it lies outside [0, E).
__device__ __forceinline__ int entry_expert(const int32_t* __restrict__ idx, long n, long n1, int E,
                                            int* err) {
  if (n >= n1) return -1;
  const int e = idx[n];
  if (e < 0 || e >= E) {
    atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
    return -1;
  }
  return e;
}

__device__ void warp_histogram(const int32_t* __restrict__ idx, long n0, long n1, int E,
                               int* hist_w, int* err) {
  const int lane = threadIdx.x % 32;
  for (long base = n0; base < n1; base += 32) {
    const long n = base + lane;
    const int e = entry_expert(idx, n, n1, E, err);
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    const int leader = __ffs(peers) - 1;
    if (e >= 0 && lane == leader) hist_w[e] += __popc(peers);
    __syncwarp();
  }
}

// Entry range [n0, n1) of warp w within chunk c.
__device__ __forceinline__ void warp_range(int c, int w, int T, int k, long* n0, long* n1) {
  const long cb = (long)c * PERM_TOK * k;
  const long ce = min((long)T * k, cb + (long)PERM_TOK * k);
  const long per = ((long)PERM_TOK * k + PERM_WARPS - 1) / PERM_WARPS;
  *n0 = min(ce, cb + w * per);
  *n1 = min(ce, cb + (w + 1) * per);
}

__global__ void __launch_bounds__(PERM_WARPS * 32) perm_hist_kernel(
    const int32_t* __restrict__ idx, int T, int k, int E, int32_t* __restrict__ chunk_counts,
    int* __restrict__ err) {
  extern __shared__ int perm_smem[];  // [PERM_WARPS][E]
  for (int i = threadIdx.x; i < PERM_WARPS * E; i += blockDim.x) perm_smem[i] = 0;
  __syncthreads();
  const int w = threadIdx.x / 32;
  long n0, n1;
  warp_range(blockIdx.x, w, T, k, &n0, &n1);
  warp_histogram(idx, n0, n1, E, perm_smem + w * E, err);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int s = 0;
    for (int q = 0; q < PERM_WARPS; ++q) s += perm_smem[q * E + e];
    chunk_counts[(size_t)blockIdx.x * E + e] = s;
  }
}

// One CTA of 1024 threads; thread e owns expert e (E <= 1024). It walks the
// chunks in order and writes each chunk's base, the exclusive prefix of its
// count over the earlier chunks: threads of consecutive experts touch adjacent
// words, so every chunk row is one coalesced pass, and the loads of eight
// chunks are issued before their sums are needed. The CTA then scans the E
// totals into the expert offsets.
__global__ void __launch_bounds__(1024) perm_scan_kernel(const int32_t* __restrict__ chunk_counts,
                                                         int n_chunks, int E,
                                                         int32_t* __restrict__ chunk_base,
                                                         int32_t* __restrict__ counts,
                                                         int32_t* __restrict__ offsets) {
  __shared__ int wsum[32];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int e = threadIdx.x;
  int total = 0;
  if (e < E) {
    int c = 0;
    for (; c + 8 <= n_chunks; c += 8) {
      int v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) v[q] = chunk_counts[(size_t)(c + q) * E + e];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        chunk_base[(size_t)(c + q) * E + e] = total;
        total += v[q];
      }
    }
    for (; c < n_chunks; ++c) {
      const int v = chunk_counts[(size_t)c * E + e];
      chunk_base[(size_t)c * E + e] = total;
      total += v;
    }
    counts[e] = total;
  }
  // exclusive scan of the E totals with 1024 threads (E <= 1024)
  const int i = threadIdx.x;
  const int v = i < E ? total : 0;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int s = wsum[lane];
    int inc = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += u;
    }
    wsum[lane] = inc - s;
  }
  __syncthreads();
  const int excl = incl - v + wsum[warp];
  if (i < E) offsets[i] = excl;
  if (i == E - 1) offsets[E] = excl + v;
}

__global__ void __launch_bounds__(PERM_WARPS * 32) perm_scatter_kernel(
    const int32_t* __restrict__ idx, int T, int k, int E, const int32_t* __restrict__ offsets,
    const int32_t* __restrict__ chunk_base, int32_t* __restrict__ row_src_token,
    int32_t* __restrict__ slot_row, const float* __restrict__ topk_w, float* __restrict__ row_w,
    int* __restrict__ err) {
  extern __shared__ int perm_smem[];  // [PERM_WARPS][E]: histogram, then cursors
  for (int i = threadIdx.x; i < PERM_WARPS * E; i += blockDim.x) perm_smem[i] = 0;
  __syncthreads();
  const int w = threadIdx.x / 32, lane = threadIdx.x % 32;
  long n0, n1;
  warp_range(blockIdx.x, w, T, k, &n0, &n1);
  int* hist_w = perm_smem + w * E;
  warp_histogram(idx, n0, n1, E, hist_w, err);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int run = offsets[e] + chunk_base[(size_t)blockIdx.x * E + e];
    for (int q = 0; q < PERM_WARPS; ++q) {
      const int v = perm_smem[q * E + e];
      perm_smem[q * E + e] = run;
      run += v;
    }
  }
  __syncthreads();
  const unsigned lt = lanemask_lt();
  for (long base = n0; base < n1; base += 32) {
    const long n = base + lane;
    const int e = entry_expert(idx, n, n1, E, err);
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    int row = 0;
    if (e >= 0) row = hist_w[e] + __popc(peers & lt);
    __syncwarp();
    if (e >= 0 && lane == __ffs(peers) - 1) hist_w[e] += __popc(peers);
    __syncwarp();
    if (e >= 0) {
      row_src_token[row] = (int32_t)(n / k);
      slot_row[n] = row;
      if (row_w) row_w[row] = topk_w[n];  // the gate weight in packed-row order
    }
  }
}

// Tile-packed weights: the 128 x 64 tile (r / 128, c / 64) of W [rows, K] is one
// contiguous 16 KiB block, tiles in (row block, column block) order; inside a
// tile, row r % 128 occupies 128 bytes and its 16-byte chunk j = (c % 64) / 8 sits
// at chunk j ^ (r % 8) -- the 128-byte swizzle the MMA operand descriptors use,
// so the GEMM copies tiles to shared memory unchanged. 16-byte vectors.
__global__ void pack_weights_kernel(const uint4* __restrict__ W, uint4* __restrict__ Wp, long rows,
                                    int K) {
  const long vpr = K / 8;  // 16-byte vectors per row
  const long total = rows * vpr;
  const long kbs = K / 64;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < total;
       i += (long)gridDim.x * blockDim.x) {
    const long r = i / vpr, v = i % vpr;
    const long tile = (r / 128) * kbs + v / 8;
    const long chunk = (v % 8) ^ (r % 8);
    Wp[tile * 1024 + (r % 128) * 8 + chunk] = W[i];
  }
}

// The whole permutation in one CTA when the batch is a single chunk (decode):
// the histogram, the scan over experts and the stable scatter of perm_hist /
// perm_scan / perm_scatter, without two launches and the chunk tables.
__global__ void __launch_bounds__(PERM_WARPS * 32) perm_single_kernel(
    const int32_t* __restrict__ idx, int T, int k, int E, int32_t* __restrict__ counts,
    int32_t* __restrict__ offsets, int32_t* __restrict__ row_src_token,
    int32_t* __restrict__ slot_row, const float* __restrict__ topk_w, float* __restrict__ row_w,
    int* __restrict__ err) {
  extern __shared__ int perm_smem[];  // [PERM_WARPS][E] histograms, then [E] totals
  int* tot = perm_smem + PERM_WARPS * E;
  for (int i = threadIdx.x; i < PERM_WARPS * E; i += blockDim.x) perm_smem[i] = 0;
  __syncthreads();
  const int w = threadIdx.x / 32, lane = threadIdx.x % 32;
  long n0, n1;
  warp_range(0, w, T, k, &n0, &n1);
  int* hist_w = perm_smem + w * E;
  warp_histogram(idx, n0, n1, E, hist_w, err);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int s = 0;
    for (int q = 0; q < PERM_WARPS; ++q) s += perm_smem[q * E + e];
    tot[e] = s;
    counts[e] = s;
  }
  __syncthreads();
  if (w == 0) {  // exclusive scan of the E totals by one warp, 32 experts per step
    int base = 0;
    for (int e0 = 0; e0 < E; e0 += 32) {
      const int e = e0 + lane;
      const int v = e < E ? tot[e] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
      }
      if (e < E) {
        offsets[e] = base + incl - v;
        tot[e] = base + incl - v;
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) offsets[E] = base;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int run = tot[e];
    for (int q = 0; q < PERM_WARPS; ++q) {
      const int v = perm_smem[q * E + e];
      perm_smem[q * E + e] = run;
      run += v;
    }
  }
  __syncthreads();
  const unsigned lt = lanemask_lt();
  for (long base = n0; base < n1; base += 32) {
    const long n = base + lane;
    const int e = entry_expert(idx, n, n1, E, err);
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    int row = 0;
    if (e >= 0) row = hist_w[e] + __popc(peers & lt);
    __syncwarp();
    if (e >= 0 && lane == __ffs(peers) - 1) hist_w[e] += __popc(peers);
    __syncwarp();
    if (e >= 0) {
      row_src_token[row] = (int32_t)(n / k);
      slot_row[n] = row;
      if (row_w) row_w[row] = topk_w[n];  // the gate weight in packed-row order
    }
  }
}

// x_perm[slot_row[t*k + j]] = x[t] for every token t and slot j (16-byte vectors).
// The slot rows of a token are read eight at a time before their stores, so a
// thread has its row reads in flight together rather than one after another.
__global__ void dispatch_rows_kernel(const uint4* __restrict__ x, int T, int vpr, int k,
                                     const int32_t* __restrict__ slot_row,
                                     uint4* __restrict__ x_perm) {
  constexpr int KB = 8;
  const size_t total = (size_t)T * vpr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t t = i / vpr, v = i % vpr;
    const uint4 val = x[i];
    for (int j0 = 0; j0 < k; j0 += KB) {
      int r[KB];
#pragma unroll
      for (int q = 0; q < KB; ++q) r[q] = j0 + q < k ? slot_row[t * k + j0 + q] : -1;
#pragma unroll
      for (int q = 0; q < KB; ++q)
        if (j0 + q < k) x_perm[(size_t)r[q] * vpr + v] = val;
    }
  }
}

// The same into the tile-packed layout (TiledRow): slot n = t*k + j of token t
// goes to packed row slot_row[n] of expert idx[n] (the gate's choice); the
// slot rows, experts and expert offsets of eight slots are read (loads the
// lanes of a warp share, one token's chunks being consecutive threads) before
// the eight stores.
__global__ void dispatch_rows_tiled_kernel(const uint4* __restrict__ x, int T, int vpr, int k,
                                           const int32_t* __restrict__ slot_row,
                                           const int32_t* __restrict__ idx,
                                           const int32_t* __restrict__ offsets, int tile,
                                           uint4* __restrict__ x_perm) {
  constexpr int KB = 8;
  const size_t total = (size_t)T * vpr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t t = i / vpr;
    const int v = (int)(i % vpr);
    const uint4 val = x[i];
    for (int j0 = 0; j0 < k; j0 += KB) {
      int r[KB], e[KB];
#pragma unroll
      for (int q = 0; q < KB; ++q) {
        const bool ok = j0 + q < k;
        r[q] = ok ? slot_row[t * k + j0 + q] : 0;
        e[q] = ok ? idx[t * k + j0 + q] : 0;
      }
      int oe[KB], ne[KB];
#pragma unroll
      for (int q = 0; q < KB; ++q) {
        oe[q] = offsets[e[q]];
        ne[q] = offsets[e[q] + 1];
      }
#pragma unroll
      for (int q = 0; q < KB; ++q)
        if (j0 + q < k)
          x_perm[tiled_row(r[q], e[q], oe[q], ne[q] - oe[q], tile, vpr).chunk16(v)] = val;
    }
  }
}

// x_perm[r] = x[row_src_token[r]] for rows of experts [e_begin, e_end).
__global__ void gather_rows_kernel(const uint4* __restrict__ x, int vpr,
                                   const int32_t* __restrict__ row_src_token,
                                   const int32_t* __restrict__ offsets, int e_begin, int e_end,
                                   uint4* __restrict__ x_perm) {
  const int r0 = offsets[e_begin], r1 = offsets[e_end];
  const size_t total = (size_t)(r1 - r0) * vpr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t r = r0 + i / vpr, v = i % vpr;
    x_perm[r * vpr + v] = x[(size_t)row_src_token[r] * vpr + v];
  }
}

// The same in the tile-packed layout (TiledRow): one warp per packed row, the
// row's expert found by binary search over the range's offsets (the last e
// with offsets[e] <= r, so empty experts are passed over), four 16-byte loads
// of a lane in flight before its stores.
__global__ void gather_rows_tiled_kernel(const uint4* __restrict__ x, int vpr,
                                         const int32_t* __restrict__ row_src_token,
                                         const int32_t* __restrict__ offsets, int e_begin,
                                         int e_end, int tile, uint4* __restrict__ x_perm) {
  constexpr int U = 4;
  const int r0 = offsets[e_begin], r1 = offsets[e_end];
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  const int n_warps = gridDim.x * wpb;
  for (int r = r0 + blockIdx.x * wpb + (threadIdx.x >> 5); r < r1; r += n_warps) {
    int lo = e_begin, hi = e_end - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (offsets[mid] <= r) lo = mid;
      else hi = mid - 1;
    }
    const int oe = offsets[lo];
    const TiledRow w = tiled_row(r, lo, oe, offsets[lo + 1] - oe, tile, vpr);
    const uint4* src = x + (size_t)row_src_token[r] * vpr;
    for (int v0 = lane; v0 < vpr; v0 += 32 * U) {
      uint4 val[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (v0 + 32 * u < vpr) val[u] = src[v0 + 32 * u];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (v0 + 32 * u < vpr) x_perm[w.chunk16(v0 + 32 * u)] = val[u];
    }
  }
}

// out[t] = sum_j w[t,j] * y_perm[slot_row[t*k+j]] (+ shared[t]); 8 elements per thread-step.
// The slots are taken eight at a time: their rows and weights first, then all
// sixteen 16-byte row loads, then the fused multiply-adds in slot order (the
// same order, and so the same rounding, as one slot after another).
__global__ void combine_kernel(const float4* __restrict__ y_perm, int T, int vpr, int k,
                               const int32_t* __restrict__ slot_row, const float* __restrict__ w,
                               const float4* __restrict__ shared, void* __restrict__ out,
                               int out_fp32, int* __restrict__ err) {
  constexpr int KB = 8;
  const int nrows = T * k;
  const size_t total = (size_t)T * vpr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t t = i / vpr, v = i % vpr;
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    for (int j0 = 0; j0 < k; j0 += KB) {
      int r[KB];
      float wj[KB];
#pragma unroll
      for (int q = 0; q < KB; ++q) {
        const int j = j0 + q;
        r[q] = -1;
        wj[q] = 0.f;
        if (j < k) {
          const int rr = slot_row[t * k + j];
          if (rr < 0 || rr >= nrows) {  // not a packed row: skip it and report
            atomicExch(err, (int)MOE_ERR_DEVICE_CHECK);
          } else {
            r[q] = rr;
            wj[q] = w[t * k + j];
          }
        }
      }
      float4 y[KB][2];
#pragma unroll
      for (int q = 0; q < KB; ++q) {
        if (r[q] >= 0) {
          y[q][0] = y_perm[((size_t)r[q] * vpr + v) * 2];
          y[q][1] = y_perm[((size_t)r[q] * vpr + v) * 2 + 1];
        } else {
          y[q][0] = y[q][1] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
#pragma unroll
      for (int q = 0; q < KB; ++q) {
        if (r[q] < 0) continue;
        const float yv[8] = {y[q][0].x, y[q][0].y, y[q][0].z, y[q][0].w,
                             y[q][1].x, y[q][1].y, y[q][1].z, y[q][1].w};
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(wj[q], yv[e], acc[e]);
      }
    }
    if (shared) {
      const float4 s0 = shared[i * 2], s1 = shared[i * 2 + 1];
      const float sv[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] += sv[q];
    }
    if (out_fp32) {
      float4* o = reinterpret_cast<float4*>(out) + i * 2;
      o[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
      o[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    } else {
      uint4 ov;
      uint16_t* oh = reinterpret_cast<uint16_t*>(&ov);
#pragma unroll
      for (int q = 0; q < 8; ++q) oh[q] = float_to_bf16_bits(acc[q]);
      reinterpret_cast<uint4*>(out)[i] = ov;
    }
  }
}

// offsets = {0, n}: the one-segment layout of the shared expert.
__global__ void fill_range_kernel(int32_t* __restrict__ offsets, int n) {
  if (threadIdx.x == 0) {
    offsets[0] = 0;
    offsets[1] = n;
  }
}

// out[e] = sum_c counts[c][e] over the chunks of a token-chunked layer.
__global__ void sum_counts_kernel(const int32_t* __restrict__ counts, int n_chunks, int E,
                                  int32_t* __restrict__ out) {
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < E; e += gridDim.x * blockDim.x) {
    int s = 0;
    for (int c = 0; c < n_chunks; ++c) s += counts[(size_t)c * E + e];
    out[e] = s;
  }
}

int copy_grid(size_t work) {
  const size_t per = 256;
  size_t b = (work + per - 1) / per;
  const size_t cap = (size_t)num_sms() * 8;
  if (b > cap) b = cap;
  if (b < 1) b = 1;
  return (int)b;
}

}  // namespace

int perm_num_chunks(int T) { return (T + PERM_TOK - 1) / PERM_TOK; }

moe_status launch_permutation(const moe_config& c, const int32_t* idx, int32_t* counts,
                              int32_t* offsets, int32_t* row_src_token, int32_t* slot_row,
                              int32_t* chunk_counts, int32_t* chunk_base, cudaStream_t s,
                              const float* topk_w, float* row_w) {
  const int nch = perm_num_chunks(c.T);
  if (nch == 1) {
    const size_t smem1 = (size_t)(PERM_WARPS + 1) * c.E * sizeof(int);
    if (smem1 > 48 * 1024)
      cudaFuncSetAttribute(perm_single_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem1);
    perm_single_kernel<<<1, PERM_WARPS * 32, smem1, s>>>(idx, c.T, c.k, c.E, counts, offsets,
                                                         row_src_token, slot_row, topk_w,
                                                         row_w, device_error_word());
    note_launch();
    return launch_status();
  }
  const size_t smem = (size_t)PERM_WARPS * c.E * sizeof(int);
  if (smem > 48 * 1024) {
    cudaFuncSetAttribute(perm_hist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaFuncSetAttribute(perm_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
  }
  if (nch > 0) {
    perm_hist_kernel<<<nch, PERM_WARPS * 32, smem, s>>>(idx, c.T, c.k, c.E, chunk_counts,
                                                        device_error_word());
    note_launch();
  }
  perm_scan_kernel<<<1, 1024, 0, s>>>(chunk_counts, nch, c.E, chunk_base, counts, offsets);
  note_launch();
  if (nch > 0) {
    perm_scatter_kernel<<<nch, PERM_WARPS * 32, smem, s>>>(idx, c.T, c.k, c.E, offsets, chunk_base,
                                                           row_src_token, slot_row, topk_w,
                                                           row_w, device_error_word());
    note_launch();
  }
  return launch_status();
}

moe_status launch_dispatch_rows(int T, int H, int k, const uint16_t* x, const int32_t* slot_row,
                                uint16_t* x_perm, cudaStream_t s, int tile, const int32_t* idx,
                                const int32_t* offsets) {
  if (T == 0) return MOE_OK;
  const int vpr = H / 8;
  if (tile > 0) {
    dispatch_rows_tiled_kernel<<<copy_grid((size_t)T * vpr), 256, 0, s>>>(
        reinterpret_cast<const uint4*>(x), T, vpr, k, slot_row, idx, offsets, tile,
        reinterpret_cast<uint4*>(x_perm));
    note_launch();
    return launch_status();
  }
  dispatch_rows_kernel<<<copy_grid((size_t)T * vpr), 256, 0, s>>>(
      reinterpret_cast<const uint4*>(x), T, vpr, k, slot_row, reinterpret_cast<uint4*>(x_perm));
  note_launch();
  return launch_status();
}

moe_status launch_gather_rows(int H, const uint16_t* x, const int32_t* row_src_token,
                              const int32_t* offsets, int e_begin, int e_end, uint16_t* x_perm,
                              int max_rows, cudaStream_t s, int tile) {
  if (max_rows == 0 || e_end <= e_begin) return MOE_OK;
  const int vpr = H / 8;
  if (tile > 0) {
    const int per_block = 8;  // warps of a 256-thread block, one packed row each
    long blocks = ((long)max_rows + per_block - 1) / per_block;
    const long cap = (long)num_sms() * 16;
    gather_rows_tiled_kernel<<<(int)(blocks < cap ? blocks : cap), 32 * per_block, 0, s>>>(
        reinterpret_cast<const uint4*>(x), vpr, row_src_token, offsets, e_begin, e_end, tile,
        reinterpret_cast<uint4*>(x_perm));
    note_launch();
    return launch_status();
  }
  gather_rows_kernel<<<copy_grid((size_t)max_rows * vpr), 256, 0, s>>>(
      reinterpret_cast<const uint4*>(x), vpr, row_src_token, offsets, e_begin, e_end,
      reinterpret_cast<uint4*>(x_perm));
  note_launch();
  return launch_status();
}

moe_status launch_combine(int T, int H, int k, const float* y_perm, const int32_t* slot_row,
                          const float* w, const float* shared, void* out, int out_fp32,
                          cudaStream_t s) {
  if (T == 0) return MOE_OK;
  const int vpr = H / 8;
  combine_kernel<<<copy_grid((size_t)T * vpr), 256, 0, s>>>(
      reinterpret_cast<const float4*>(y_perm), T, vpr, k, slot_row, w,
      reinterpret_cast<const float4*>(shared), out, out_fp32, device_error_word());
  note_launch();
  return launch_status();
}

moe_status launch_fill_range(int32_t* offsets, int n, cudaStream_t s) {
  fill_range_kernel<<<1, 32, 0, s>>>(offsets, n);
  note_launch();
  return launch_status();
}

moe_status launch_sum_counts(const int32_t* counts, int n_chunks, int E, int32_t* out,
                             cudaStream_t s) {
  sum_counts_kernel<<<(E + 255) / 256, 256, 0, s>>>(counts, n_chunks, E, out);
  note_launch();
  return launch_status();
}

moe_status launch_pack_weights(const uint16_t* W, uint16_t* Wp, long rows, int K, cudaStream_t s) {
  if (rows == 0) return MOE_OK;
  pack_weights_kernel<<<copy_grid((size_t)rows * (K / 8)), 256, 0, s>>>(
      reinterpret_cast<const uint4*>(W), reinterpret_cast<uint4*>(Wp), rows, K);
  note_launch();
  return launch_status();
}

}  // namespace moe
