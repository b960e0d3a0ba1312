// ShiftQuant quantizer kernels for sm_103a and their C entry points.
//
//   range pass  (Sec. 3.1)   per-column max|x| with 128-bit loads and an atomic max on the
//                            bit pattern of the non-negative float; per-row max for the
//                            per-in-channel weight role
//   grouping    (Eq. 3)      tau_0 = max_c r_c, e_c = the largest e <= N_G-1 with
//                            r_c 2^e <= tau_0, i.e. floor(log2(tau_0 / r_c)) clipped
//   quantize    (App. D/B)   q = round(x 2^e_c Q / tau_0) with round-to-nearest-even or
//                            stochastic rounding on a counter-based SplitMix64 draw;
//                            optional shift of weight codes by 2^(N_G-1-e) (ShiftMM)
//
// All three are HBM-bound streaming passes.  The quantizer writes the codes directly in
// the operand format of the tensor-core GEMM (E4M3 or BF16, exact integers) and, in the
// same pass, the transposed copy the weight-gradient GEMM reads, staged through shared
// memory so both writes stay coalesced.
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>

#include "sq_device.cuh"
#include "sq_host.h"
#include "sq_quant_dev.cuh"

namespace sq {

static thread_local char g_last_error[512];

int fail(int status, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
  va_end(ap);
  return status;
}

static void clear_error() { g_last_error[0] = 0; }

// the group order a shiftquant_quantize_ordered call hands to the quantizer launch it makes
// (per host thread; null outside such a call)
static thread_local const int* g_order_cols = nullptr;
static thread_local const int* g_order_rows = nullptr;

// ===================================================================== range pass
constexpr int kColTx = 32;  // threads along columns, 4 columns each: 128 columns per block
constexpr int kColTy = 8;   // threads along rows

__device__ __forceinline__ uint32_t abs_bits(float v) { return __float_as_uint(v) & 0x7FFFFFFFu; }

// range_bits[c] = max over this block's rows of |x[r, c]| as an ordered bit pattern
// (for non-negative floats, larger value <=> larger unsigned pattern; NaN sorts above Inf).
// zero the range accumulators a[na] and b[nb] (b may be null); the range pass that follows
// may launch at once: it reads x first and these only after its wait
__global__ void __launch_bounds__(256)
    calib_init_kernel(unsigned* __restrict__ a, int64_t na, unsigned* __restrict__ b, int64_t nb) {
  griddep_launch_dependents();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < na; i += stride)
    a[i] = 0u;
  if (b != nullptr)
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nb; i += stride)
      b[i] = 0u;
}

// Grouping (Eq. 3) by one block of THREADS threads from the per-channel range bits:
// tau_0 = the largest range, then every channel's exponent; tau0_out receives tau_0 and
// the status word the non-finite flag.  Thread t holds channels t, t + THREADS, ... (up to
// kGroupPerThread of them in registers, so all its loads are in flight together; wider
// tensors read the rest twice).  Small blocks start faster, large ones take wide tensors
// in one round of loads.  Launched behind the range pass with programmatic stream
// serialization, it waits for the range pass before reading anything.
constexpr int kGroupPerThread = 16;
constexpr int kGroupSmallThreads = 256;
constexpr int kGroupLargeThreads = 1024;

template <int THREADS>
__global__ void __launch_bounds__(THREADS)
    group_kernel(const unsigned* __restrict__ range_bits, int64_t C, int G,
                 float* __restrict__ tau0_out, uint8_t* __restrict__ exp_out,
                 int* __restrict__ status) {
  __shared__ unsigned wmax[THREADS / 32];
  __shared__ unsigned tau_bits;
  griddep_wait();
  griddep_launch_dependents();
  const int tid = threadIdx.x;
  unsigned v[kGroupPerThread];
  unsigned m = 0;
#pragma unroll
  for (int k = 0; k < kGroupPerThread; ++k) {
    const int64_t c = tid + static_cast<int64_t>(k) * THREADS;
    v[k] = c < C ? __ldcg(range_bits + c) : 0u;
    m = max(m, v[k]);
  }
  constexpr int64_t kHeld = static_cast<int64_t>(THREADS) * kGroupPerThread;
  for (int64_t c = kHeld + tid; c < C; c += THREADS) m = max(m, __ldcg(range_bits + c));
  m = __reduce_max_sync(0xFFFFFFFFu, m);
  if ((tid & 31) == 0) wmax[tid >> 5] = m;
  __syncthreads();
  if (tid < 32) {
    const unsigned w = __reduce_max_sync(0xFFFFFFFFu, tid < THREADS / 32 ? wmax[tid] : 0u);
    if (tid == 0) tau_bits = w;
  }
  __syncthreads();
  const unsigned tb = tau_bits;
  const float tau = __uint_as_float(tb);
  const bool nonfinite = tb >= 0x7F800000u;
#pragma unroll
  for (int k = 0; k < kGroupPerThread; ++k) {
    const int64_t c = tid + static_cast<int64_t>(k) * THREADS;
    if (c < C) exp_out[c] = static_cast<uint8_t>(nonfinite ? 0 : group_exponent(__uint_as_float(v[k]), tau, G));
  }
  for (int64_t c = kHeld + tid; c < C; c += THREADS)
    exp_out[c] = static_cast<uint8_t>(nonfinite ? 0 : group_exponent(__uint_as_float(__ldcg(range_bits + c)), tau, G));
  if (tid == 0) {
    *tau0_out = tau;
    if (nonfinite) atomicOr(status, kDevNonFinite);
  }
}

// Range pass: block (x, y) reads tile (y, x) of TC = 4 << lg columns (the column count
// rounded up to a power of two, 4 to 128) by 8 passes of 1024 / TC rows -- thread t owns
// the four-column quad t mod (TC / 4) and the rows t / (TC / 4) + k 1024 / TC, with all
// eight 16-byte loads in flight -- and takes its per-column maxima as ordered bit patterns
// of the non-negative floats (NaN sorts above Inf), sent to range_bits with one atomic max
// per column.  Same-address atomics from hundreds of tiles of a narrow tensor serialise in
// L2, so narrow tensors (CL = kRangeCluster) run in clusters of CL blocks along the rows:
// each block merges its maxima into the first block of its cluster with atomic maxima on
// that block's shared memory, and only that block sends them on.  Wide tensors (CL = 1)
// spread their atomics over many addresses and run without clusters, which schedule more
// slowly.  Grids taller than the 65535-block limit
// walk the extra tiles in steps of gridDim.y.
// ROWS: the range pass of a weight for both of its roles -- also every row's max|x| over
// all columns (the per-in-channel ranges), each warp's eight rows of a tile reduced across
// its lanes and sent to row_bits with one atomic max per row and column block.
constexpr int kRangeCluster = 8;
constexpr int64_t kRangeClusterMaxCols = 512;   // clusters for tensors of at most 512 columns

template <int CL, bool ROWS>
__global__ void __launch_bounds__(kColTx* kColTy)
    colmax_kernel(const float* __restrict__ x, int64_t R, int64_t C, int64_t ld, int vec, int lg,
                  unsigned* __restrict__ range_bits, unsigned* __restrict__ row_bits,
                  int* __restrict__ status) {
  __shared__ unsigned red[kColTy * kColTx * 4];
  __shared__ unsigned cmax[CL > 1 ? kColTx * 4 : 1];   // the cluster's maxima (first block)
  const int tid = threadIdx.y * kColTx + threadIdx.x;
  // the tile: tc = 4 << lg columns (one four-column quad per thread) by 8 passes of rpp rows
  const int tc = 4 << lg, rpp = (kColTx * kColTy) >> lg;
  const int qc = tid & ((1 << lg) - 1), ro = tid >> lg;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * tc + 4 * qc;
  const int64_t tile_rows = 8 * static_cast<int64_t>(rpp);
  const int64_t tiles = (R + tile_rows - 1) / tile_rows;
  if (CL > 1) {
    if (tid < kColTx * 4) cmax[tid] = 0u;
    cluster_arrive_release();   // the zeroed cmax is visible to the cluster after the wait
  }
  unsigned m0 = 0, m1 = 0, m2 = 0, m3 = 0;
  bool row_bad = false;
#pragma unroll 1
  for (int64_t t = blockIdx.y; t < tiles; t += gridDim.y) {
    const int64_t r0 = t * tile_rows + ro;   // this thread's rows: r0 + u rpp
    unsigned rm[8];   // ROWS: this thread's four columns of each of its rows
    if (vec && c0 + 3 < C) {
      // rows past the end re-read the last row, which leaves a maximum unchanged
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = ld_stream_v4(x + min(r0 + u * rpp, R - 1) * ld + c0);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const unsigned a0 = abs_bits(v[u].x), a1 = abs_bits(v[u].y);
        const unsigned a2 = abs_bits(v[u].z), a3 = abs_bits(v[u].w);
        m0 = max(m0, a0);
        m1 = max(m1, a1);
        m2 = max(m2, a2);
        m3 = max(m3, a3);
        if (ROWS) rm[u] = max(max(a0, a1), max(a2, a3));
      }
    } else {
#pragma unroll
      for (int u = 0; u < 8; ++u) rm[u] = 0u;
#pragma unroll 1
      for (int u = 0; u < 8; ++u) {
        const int64_t r = r0 + u * rpp;
        if (r >= R) break;
        const float* row = x + r * ld;
        unsigned a[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (c0 + k < C) a[k] = abs_bits(__ldg(row + c0 + k));
        m0 = max(m0, a[0]);
        m1 = max(m1, a[1]);
        m2 = max(m2, a[2]);
        m3 = max(m3, a[3]);
        if (ROWS) {
#pragma unroll
          for (int k = 0; k < 8; ++k)  // rm stays in registers: no run-time index
            if (k == u) rm[k] = max(max(a[0], a[1]), max(a[2], a[3]));
        }
      }
    }
    if (ROWS) {
      // (lg = 5: a warp's 32 quads are one row of the tile, a warp row per pass)
      // the row accumulators are zeroed by the preceding kernel, which must have completed
      griddep_wait();
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const unsigned m = __reduce_max_sync(0xFFFFFFFFu, rm[u]);
        const int64_t r = r0 + u * rpp;
        if (threadIdx.x == 0 && r < R && m != 0u) {
          atomicMax(row_bits + r, m);
          row_bad |= m >= 0x7F800000u;
        }
      }
    }
  }
  if (ROWS && row_bad) atomicOr(status, kDevNonFinite);
  // x has been read: the next kernel (the grouping) may start launching
  griddep_launch_dependents();
  red[ro * tc + 4 * qc + 0] = m0;
  red[ro * tc + 4 * qc + 1] = m1;
  red[ro * tc + 4 * qc + 2] = m2;
  red[ro * tc + 4 * qc + 3] = m3;
  __syncthreads();
  // thread t < tc: column t of the tile
  unsigned m = 0;
  if (tid < tc)
    for (int y = 0; y < rpp; ++y) m = max(m, red[y * tc + tid]);
  if (CL > 1) {
    cluster_wait_acquire();
    if (tid < tc && m != 0) red_max_cluster_u32(mapa_shared(smem_u32(cmax), 0) + tid * 4, m);
    cluster_arrive_release();
    cluster_wait_acquire();   // every block's maxima are in the first block's cmax
    if (cluster_ctarank() != 0) return;
    if (tid < tc) m = cmax[tid];
  }
  if (tid >= tc) return;
  // the accumulators are zeroed by the preceding kernel, which must have completed
  griddep_wait();
  const int64_t c = static_cast<int64_t>(blockIdx.x) * tc + tid;
  if (c < C && m != 0) {
    atomicMax(range_bits + c, m);
    if (m >= 0x7F800000u) atomicOr(status, kDevNonFinite);
  }
}

// The range pass of a wide weight (more than 512 columns) for both roles: per-column and
// per-row max|x|.  A block takes one tile of 64 rows (8 passes of 8) and walks kWeightRun
// consecutive 128-column blocks of it, one after another: each column block's maxima leave
// by atomics as in colmax_kernel, but every row's maximum leaves the block once per run.
// A block per column block would send each row cblocks atomics, and the blocks of one row
// tile send them together: on [4096, 11008] those 86 same-address atomics per row queued
// in L2 and took the pass from 33 us (columns alone) to 55 us; with runs of 4 it takes
// 36.5 us (measured, a scratch probe; prefetching the next column block into registers was
// slower).
constexpr int kWeightRun = 4;

__global__ void __launch_bounds__(kColTx* kColTy)
    weight_range_kernel(const float* __restrict__ x, int64_t R, int64_t C, int64_t ld, int vec,
                        unsigned* __restrict__ col_bits, unsigned* __restrict__ row_bits,
                        int* __restrict__ status) {
  __shared__ unsigned red[kColTy * kColTx * 4];
  const int tx = threadIdx.x, ty = threadIdx.y, tid = ty * kColTx + tx;
  const int64_t cblocks = (C + 4 * kColTx - 1) / (4 * kColTx);
  const int64_t tiles = (R + 8 * kColTy - 1) / (8 * kColTy);
  const int64_t j0 = static_cast<int64_t>(blockIdx.x) * kWeightRun;
  bool bad = false;
  bool waited = false;
#pragma unroll 1
  for (int64_t t = blockIdx.y; t < tiles; t += gridDim.y) {
    const int64_t r0 = t * 8 * kColTy + ty;   // this thread's rows: r0 + u kColTy
    unsigned rm[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) rm[u] = 0u;
#pragma unroll 1
    for (int64_t j = j0; j < j0 + kWeightRun && j < cblocks; ++j) {
      const int64_t c0 = j * 4 * kColTx + 4 * tx;
      unsigned m0 = 0, m1 = 0, m2 = 0, m3 = 0;
      if (vec && c0 + 3 < C) {
        // rows past the end re-read the last row, which leaves a maximum unchanged
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = ld_stream_v4(x + min(r0 + u * kColTy, R - 1) * ld + c0);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const unsigned a0 = abs_bits(v[u].x), a1 = abs_bits(v[u].y);
          const unsigned a2 = abs_bits(v[u].z), a3 = abs_bits(v[u].w);
          m0 = max(m0, a0);
          m1 = max(m1, a1);
          m2 = max(m2, a2);
          m3 = max(m3, a3);
          rm[u] = max(rm[u], max(max(a0, a1), max(a2, a3)));
        }
      } else {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int64_t r = min(r0 + u * kColTy, R - 1);
          unsigned a[4] = {0u, 0u, 0u, 0u};
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (c0 + k < C) a[k] = abs_bits(__ldg(x + r * ld + c0 + k));
          m0 = max(m0, a[0]);
          m1 = max(m1, a[1]);
          m2 = max(m2, a[2]);
          m3 = max(m3, a[3]);
          rm[u] = max(rm[u], max(max(a[0], a[1]), max(a[2], a[3])));
        }
      }
      red[ty * 4 * kColTx + 4 * tx + 0] = m0;
      red[ty * 4 * kColTx + 4 * tx + 1] = m1;
      red[ty * 4 * kColTx + 4 * tx + 2] = m2;
      red[ty * 4 * kColTx + 4 * tx + 3] = m3;
      __syncthreads();
      if (!waited) {   // the accumulators are zeroed by the preceding kernel
        griddep_wait();
        waited = true;
      }
      if (tid < 4 * kColTx) {
        unsigned m = 0;
        for (int y = 0; y < kColTy; ++y) m = max(m, red[y * 4 * kColTx + tid]);
        const int64_t c = j * 4 * kColTx + tid;
        if (c < C && m != 0u) {
          atomicMax(col_bits + c, m);
          bad |= m >= 0x7F800000u;
        }
      }
      __syncthreads();   // red is rewritten by the next column block
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const unsigned m = __reduce_max_sync(0xFFFFFFFFu, rm[u]);
      const int64_t r = r0 + u * kColTy;
      if (tx == 0 && r < R && m != 0u) {
        atomicMax(row_bits + r, m);
        bad |= m >= 0x7F800000u;
      }
    }
  }
  // x has been read: the next kernel may start launching
  griddep_launch_dependents();
  if (bad) atomicOr(status, kDevNonFinite);
}

// one warp per row: range[r] = max_c |x[r, c]|
__global__ void __launch_bounds__(256)
    rowmax_kernel(const float* __restrict__ x, int64_t R, int64_t C, int64_t ld, int vec,
                  float* __restrict__ range, int* __restrict__ status) {
  const int lane = threadIdx.x & 31;
  const int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + (threadIdx.x >> 5);
  if (r >= R) return;
  const float* row = x + r * ld;
  unsigned m = 0;
  int64_t c = 0;
  if (vec) {
    const int64_t c4 = C & ~int64_t(3);
#pragma unroll 4
    for (int64_t cc = lane * 4; cc < c4; cc += 128) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(row + cc));
      m = max(max(m, abs_bits(v.x)), max(abs_bits(v.y), max(abs_bits(v.z), abs_bits(v.w))));
    }
    c = c4;
  }
  for (int64_t cc = c + lane; cc < C; cc += 32) m = max(m, abs_bits(__ldg(row + cc)));
  m = __reduce_max_sync(0xFFFFFFFFu, m);
  if (lane == 0) {
    range[r] = __uint_as_float(m);
    if (m >= 0x7F800000u) atomicOr(status, kDevNonFinite);
  }
}

// ======================================================================= quantize
struct QuantArgs {
  const float* x;
  int64_t R, C, ld;
  int gran, Q, G, mode;
  uint64_t seed;
  int64_t row0;           // the tensor's first row within the logical tensor (SR index)
  const float* rt;        // &tau_0 (SHIFT) or range[] (PER_COL / PER_ROW)
  const uint8_t* exp;     // SHIFT: e_c
  const uint8_t* fold;    // optional: exponents of the other GEMM operand
  void* codes;
  int64_t ldc;
  void* codes_t;
  int64_t ldt;
  float* scale_out;
  int vec_in, vec_out, vec_t;
  // group order of the GEMM inner index (or null): codes column c goes to pos_cols[c]
  // (ShiftQuant and per-row grans), codes_t column r to pos_rows[r] (per-column gran)
  const int* pos_cols;
  const int* pos_rows;
};


template <typename CodeT>
__device__ __forceinline__ CodeT encode_code(float v);

template <>
__device__ __forceinline__ uint16_t encode_code<uint16_t>(float v) {
  // v is an integer with at most 8 significant bits: the top half of its binary32
  // pattern is its exact BF16 pattern
  return static_cast<uint16_t>(__float_as_uint(v) >> 16);
}

template <>
__device__ __forceinline__ uint8_t encode_code<uint8_t>(float v) {
  return static_cast<uint8_t>(__nv_cvt_float_to_fp8(v, __NV_SATFINITE, __NV_E4M3));
}

// quantize tile: 64 rows x 128 columns, 256 threads.  Lane l owns columns 4l .. 4l+3 of
// the tile and warp w the eight rows 8w .. 8w+7: every load instruction of a warp reads 512
// contiguous bytes of one row, and all eight loads of a thread are in flight together.
// For the transposed copy each thread packs, per column, its eight codes (rows 8w..8w+7)
// into one chunk; chunk w of tile column c sits at slot c*8 + (w ^ ((c >> 2) & 7)) of the
// shared staging area, so the chunk stores of a warp and the row reads that follow both
// touch every bank equally.
constexpr int kQR = 64;
constexpr int kQC = 128;
constexpr int kQRowsPerWarp = kQR / 8;

__device__ __forceinline__ int chunk_slot(int col, int chunk) {
  return col * 8 + (chunk ^ ((col >> 2) & 7));
}

// The thread's eight input rows of the block's 64 x 128 tile (four columns each), all
// loads in flight together; outside the tensor the values are 0.  FULL: the tile lies
// inside the tensor and its rows are 16-byte aligned.
template <bool FULL>
__device__ __forceinline__ void load_quant_tile(const QuantArgs& a, float4 (&xin)[kQRowsPerWarp]) {
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int wq = tid >> 5;
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kQR;
  const int64_t cb = static_cast<int64_t>(blockIdx.x) * kQC + lane * 4;
#pragma unroll
  for (int i = 0; i < kQRowsPerWarp; ++i) {
    const int64_t r = r0 + wq * 8 + i;
    const float* row = a.x + r * a.ld;
    if (FULL) {
      xin[i] = ld_stream_v4(row + cb);
    } else {
      xin[i] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      if (r < a.R) {
        if (a.vec_in && cb + 3 < a.C) {
          xin[i] = __ldg(reinterpret_cast<const float4*>(row + cb));
        } else {
          if (cb + 0 < a.C) xin[i].x = __ldg(row + cb + 0);
          if (cb + 1 < a.C) xin[i].y = __ldg(row + cb + 1);
          if (cb + 2 < a.C) xin[i].z = __ldg(row + cb + 2);
          if (cb + 3 < a.C) xin[i].w = __ldg(row + cb + 3);
        }
      }
    }
  }
}

// One 64 x 128 tile.  GRAN: SQ_GRAN_*; MODE: SQ_ROUND_*; FOLD: weight codes carry the
// ShiftMM shift 2^(G-1-fold[i]); FULL: the tile lies inside the tensor and every access
// is vector-aligned, so no element needs a bounds check.  LOAD: the tile's loads are
// issued here; otherwise `pre` holds the thread's eight rows, loaded by the caller
// (load_quant_tile) -- the weight kernel quantizes one load for both roles.
template <typename CodeT, int GRAN, int MODE, bool FOLD, bool FULL, bool LOAD = true>
__device__ __forceinline__ void quantize_tile(const QuantArgs& a, uint8_t* tile_t,
                                              const float4* pre = nullptr) {
  constexpr int kChunkBytes = 8 * sizeof(CodeT);  // eight codes of one column
  constexpr int kWords = kChunkBytes / 4;         // 32-bit words per packed column chunk
  constexpr int kPerWord = 4 / sizeof(CodeT);
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int wq = tid >> 5;
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kQR;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kQC;
  const int64_t cb = c0 + lane * 4;
  const float Qf = static_cast<float>(a.Q);

  // all eight input rows of this thread first, so their loads overlap
  float4 xin[kQRowsPerWarp];
#pragma unroll
  for (int i = 0; i < kQRowsPerWarp; ++i) {
    if (!LOAD) {
      xin[i] = pre[i];
      continue;
    }
    const int64_t r = r0 + wq * 8 + i;
    const float* row = a.x + r * a.ld;
    if (FULL) {
      xin[i] = ld_stream_v4(row + cb);
    } else {
      xin[i] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      if (r < a.R) {
        if (a.vec_in && cb + 3 < a.C) {
          xin[i] = __ldg(reinterpret_cast<const float4*>(row + cb));
        } else {
          if (cb + 0 < a.C) xin[i].x = __ldg(row + cb + 0);
          if (cb + 1 < a.C) xin[i].y = __ldg(row + cb + 1);
          if (cb + 2 < a.C) xin[i].z = __ldg(row + cb + 2);
          if (cb + 3 < a.C) xin[i].w = __ldg(row + cb + 3);
        }
      }
    }
  }

  // per-column multipliers: 2^e_c (SHIFT) or Q / range_c (PER_COL); per-column shifts
  float colmul[4];
  bool colzero[4];
  int colfold[4];
  float invS = 0.0f;
  bool zero_all = false;
  if (GRAN == SQ_GRAN_SHIFT) {
    const float tau = __ldg(a.rt);
    invS = __fdiv_rn(Qf, tau);
    zero_all = !(tau > 0.0f) || !isfinite(tau) || !isfinite(invS);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int64_t c = cb + j;
    colmul[j] = 1.0f;
    colzero[j] = false;
    colfold[j] = 0;
    if (FULL || c < a.C) {
      if (GRAN == SQ_GRAN_SHIFT) {
        colmul[j] = pow2f(__ldg(a.exp + c));
      } else if (GRAN == SQ_GRAN_PER_COL) {
        const float rg = __ldg(a.rt + c);
        colmul[j] = __fdiv_rn(Qf, rg);
        colzero[j] = !(rg > 0.0f) || !isfinite(rg) || !isfinite(colmul[j]);
      }
      if (GRAN == SQ_GRAN_PER_ROW && FOLD) colfold[j] = a.G - 1 - __ldg(a.fold + c);
    }
  }

  uint32_t packed[4][kWords];
#pragma unroll
  for (int j = 0; j < 4; ++j)
#pragma unroll
    for (int k = 0; k < kWords; ++k) packed[j][k] = 0u;

  // stochastic rounding: the generator state of element (r, c) is seed + (idx+1) gamma with
  // idx = (row0 + r) C + c; it advances by gamma per column and by C gamma per row
  uint64_t sr_state = 0;
  if (MODE == SQ_ROUND_STOCHASTIC)
    sr_state = a.seed + (static_cast<uint64_t>(a.row0 + r0 + wq * 8) * static_cast<uint64_t>(a.C) +
                         static_cast<uint64_t>(cb) + 1ull) * kSplitMixGamma;
  const uint64_t sr_row_step = static_cast<uint64_t>(a.C) * kSplitMixGamma;

#pragma unroll
  for (int i = 0; i < kQRowsPerWarp; ++i) {
    const int64_t r = r0 + wq * 8 + i;
    const bool row_in = FULL || r < a.R;
    float rowmul = 1.0f;
    bool rowzero = false;
    int rowfold = 0;
    if (row_in) {
      if (GRAN == SQ_GRAN_PER_ROW) {
        const float rg = __ldg(a.rt + r);
        rowmul = __fdiv_rn(Qf, rg);
        rowzero = !(rg > 0.0f) || !isfinite(rg) || !isfinite(rowmul);
      }
      if (GRAN == SQ_GRAN_PER_COL && FOLD) rowfold = a.G - 1 - __ldg(a.fold + r);
    }
    const float xv[4] = {xin[i].x, xin[i].y, xin[i].z, xin[i].w};
    CodeT out[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float v;
      bool z;
      if (GRAN == SQ_GRAN_SHIFT) {
        v = __fmul_rn(__fmul_rn(xv[j], colmul[j]), invS);  // x 2^e exactly, then * Q/tau
        z = zero_all;
      } else if (GRAN == SQ_GRAN_PER_COL) {
        v = __fmul_rn(xv[j], colmul[j]);
        z = colzero[j];
      } else {
        v = __fmul_rn(xv[j], rowmul);
        z = rowzero;
      }
      if (!FULL) z = z || !row_in || cb + j >= a.C;
      float q;
      if (MODE == SQ_ROUND_NEAREST_EVEN) {
        // |x| <= range gives |v| <= Q (1 + 2^-23), so rint never leaves [-Q, Q]
        q = rintf(v);
      } else {
        const float l = floorf(v);
        const float frac = __fsub_rn(v, l);
        const uint32_t h24 = splitmix64_top24(sr_state + static_cast<uint64_t>(j) * kSplitMixGamma +
                                              static_cast<uint64_t>(i) * sr_row_step);
        const float u = __fmul_rn(static_cast<float>(h24), 5.9604644775390625e-08f);  // * 2^-24, exact
        q = (u < frac) ? __fadd_rn(l, 1.0f) : l;
        q = fminf(fmaxf(q, -Qf), Qf);
      }
      if (z) q = 0.0f;
      if (FOLD) {
        const int f = (GRAN == SQ_GRAN_PER_ROW) ? colfold[j] : rowfold;
        q = __fmul_rn(q, pow2f(f));
      }
      out[j] = encode_code<CodeT>(__fadd_rn(q, 0.0f));  // +0 for a zero code
      packed[j][i / kPerWord] |= static_cast<uint32_t>(out[j]) << (8 * sizeof(CodeT) * (i % kPerWord));
    }
    if (a.codes && row_in && a.pos_cols != nullptr) {
      CodeT* dst = static_cast<CodeT*>(a.codes) + r * a.ldc;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (FULL || cb + j < a.C) dst[__ldg(a.pos_cols + cb + j)] = out[j];
    } else if (a.codes && row_in) {
      CodeT* dst = static_cast<CodeT*>(a.codes) + r * a.ldc + cb;
      if (FULL || (a.vec_out && cb + 3 < a.C)) {
        if constexpr (sizeof(CodeT) == 2) {
          uint2 w;
          w.x = static_cast<uint32_t>(out[0]) | (static_cast<uint32_t>(out[1]) << 16);
          w.y = static_cast<uint32_t>(out[2]) | (static_cast<uint32_t>(out[3]) << 16);
          *reinterpret_cast<uint2*>(dst) = w;
        } else {
          const uint32_t w = static_cast<uint32_t>(out[0]) | (static_cast<uint32_t>(out[1]) << 8) |
                             (static_cast<uint32_t>(out[2]) << 16) |
                             (static_cast<uint32_t>(out[3]) << 24);
          *reinterpret_cast<uint32_t*>(dst) = w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (cb + j < a.C) dst[j] = out[j];
      }
    }
  }

  if (a.codes_t) {
    const uint32_t base = smem_u32(tile_t);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t dst = base + chunk_slot(lane * 4 + j, wq) * kChunkBytes;
      if constexpr (kWords == 4)
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(packed[j][0]),
                     "r"(packed[j][1]), "r"(packed[j][2]), "r"(packed[j][3]) : "memory");
      else
        asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(dst), "r"(packed[j][0]),
                     "r"(packed[j][1]) : "memory");
    }
    __syncthreads();
    if (a.pos_rows != nullptr) {
      // group-ordered transposed copy: element (column c, row r) goes to pos_rows[r]
      CodeT* ctp = static_cast<CodeT*>(a.codes_t);
      for (int idx = tid; idx < kQC * kQR; idx += 256) {
        const int lc = idx / kQR, rr = idx % kQR;
        const int64_t c = c0 + lc, r = r0 + rr;
        if (!FULL && (c >= a.C || r >= a.R)) continue;
        const CodeT v = reinterpret_cast<const CodeT*>(tile_t + chunk_slot(lc, rr >> 3) * kChunkBytes)[rr & 7];
        ctp[c * a.ldt + __ldg(a.pos_rows + r)] = v;
      }
      goto scales;
    }
    {
    // each transposed row (one tile column) holds 64 codes = 8 chunks; 16-byte stores
    constexpr int kChunksPerStore = 16 / kChunkBytes;            // 1 (BF16) or 2 (E4M3)
    constexpr int kStoresPerRow = 8 / kChunksPerStore;
    constexpr int E = 16 / sizeof(CodeT);                         // codes per 16-byte store
    uint8_t* ct = static_cast<uint8_t*>(a.codes_t);
#pragma unroll
    for (int idx = tid; idx < kQC * kStoresPerRow; idx += 256) {
      const int lc = idx / kStoresPerRow, st = idx % kStoresPerRow;
      const int64_t c = c0 + lc;
      const int64_t rs = r0 + st * E;
      if (!FULL && (c >= a.C || rs >= a.R)) continue;
      uint4 v;
      if constexpr (kChunksPerStore == 1) {
        v = *reinterpret_cast<const uint4*>(tile_t + chunk_slot(lc, st) * kChunkBytes);
      } else {
        const uint2 lo = *reinterpret_cast<const uint2*>(tile_t + chunk_slot(lc, 2 * st) * kChunkBytes);
        const uint2 hi = *reinterpret_cast<const uint2*>(tile_t + chunk_slot(lc, 2 * st + 1) * kChunkBytes);
        v = make_uint4(lo.x, lo.y, hi.x, hi.y);
      }
      uint8_t* dst = ct + (c * a.ldt + rs) * static_cast<int64_t>(sizeof(CodeT));
      if (FULL || (a.vec_t && rs + E <= a.R)) {
        *reinterpret_cast<uint4*>(dst) = v;
      } else {
        const uint8_t* vb = reinterpret_cast<const uint8_t*>(&v);
        for (int e = 0; e < E && rs + e < a.R; ++e)
          for (int b = 0; b < static_cast<int>(sizeof(CodeT)); ++b)
            dst[e * sizeof(CodeT) + b] = vb[e * sizeof(CodeT) + b];
      }
    }
    }
  }
scales:
  // scales: s = tau_0 / Q, or range / Q per channel (0 for an all-zero channel)
  if (GRAN == SQ_GRAN_SHIFT) {
    if (blockIdx.x == 0 && blockIdx.y == 0 && tid == 0) {
      const float tau = __ldg(a.rt);
      *a.scale_out = zero_all ? 0.0f : __fdiv_rn(tau, Qf);
    }
  } else if (GRAN == SQ_GRAN_PER_COL) {
    if (blockIdx.y == 0 && wq == 0) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (FULL || cb + j < a.C)
          a.scale_out[cb + j] = colzero[j] ? 0.0f : __fdiv_rn(__ldg(a.rt + cb + j), Qf);
    }
  } else {
    if (blockIdx.x == 0 && lane == 0) {
#pragma unroll
      for (int i = 0; i < kQRowsPerWarp; ++i) {
        const int64_t r = r0 + wq * 8 + i;
        if (FULL || r < a.R) {
          const float rg = __ldg(a.rt + r);
          const float inv = __fdiv_rn(Qf, rg);
          const bool z = !(rg > 0.0f) || !isfinite(rg) || !isfinite(inv);
          a.scale_out[r] = z ? 0.0f : __fdiv_rn(rg, Qf);
        }
      }
    }
  }
}

template <typename CodeT, int GRAN, int MODE, bool FOLD>
__global__ void __launch_bounds__(256) quantize_kernel(const QuantArgs a) {
  __shared__ __align__(16) uint8_t tile_t[kQC * 8 * 8 * sizeof(CodeT)];
  // launched early behind the range pass: nothing it wrote (nor x) is read before it is done
  griddep_wait();
  const bool full = (static_cast<int64_t>(blockIdx.y) + 1) * kQR <= a.R &&
                    (static_cast<int64_t>(blockIdx.x) + 1) * kQC <= a.C && a.vec_in &&
                    (a.codes == nullptr || a.vec_out) && (a.codes_t == nullptr || a.vec_t);
  if (full)
    quantize_tile<CodeT, GRAN, MODE, FOLD, true>(a, tile_t);
  else
    quantize_tile<CodeT, GRAN, MODE, FOLD, false>(a, tile_t);
}

// Launch with programmatic stream serialization: the kernel may begin launching while the
// preceding kernel of the stream finishes, and waits for it (griddep_wait) before reading
// anything.
template <typename... Params, typename... Args>
static cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, cudaStream_t s,
                              Args... args) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <typename CodeT>
static void launch_quantize(const QuantArgs& a, dim3 grid, cudaStream_t s) {
  const bool fold = a.fold != nullptr;
  if (a.gran == SQ_GRAN_SHIFT) {
    if (a.mode == SQ_ROUND_NEAREST_EVEN)
      launch_pdl(quantize_kernel<CodeT, SQ_GRAN_SHIFT, SQ_ROUND_NEAREST_EVEN, false>, grid, dim3(256), s, a);
    else
      launch_pdl(quantize_kernel<CodeT, SQ_GRAN_SHIFT, SQ_ROUND_STOCHASTIC, false>, grid, dim3(256), s, a);
  } else if (a.gran == SQ_GRAN_PER_COL) {
    if (a.mode == SQ_ROUND_NEAREST_EVEN) {
      if (fold) launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_NEAREST_EVEN, true>, grid, dim3(256), s, a);
      else launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_NEAREST_EVEN, false>, grid, dim3(256), s, a);
    } else {
      if (fold) launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_STOCHASTIC, true>, grid, dim3(256), s, a);
      else launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_STOCHASTIC, false>, grid, dim3(256), s, a);
    }
  } else {
    if (a.mode == SQ_ROUND_NEAREST_EVEN) {
      if (fold) launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_NEAREST_EVEN, true>, grid, dim3(256), s, a);
      else launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_NEAREST_EVEN, false>, grid, dim3(256), s, a);
    } else {
      if (fold) launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_STOCHASTIC, true>, grid, dim3(256), s, a);
      else launch_pdl(quantize_kernel<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_STOCHASTIC, false>, grid, dim3(256), s, a);
    }
  }
}

// Both roles of a weight from one pass over it (Sec. 5.1): the forward GEMM's
// per-out-channel codes (gran PER_COL, written transposed, the fold indexed by row) and loss
// propagation's per-in-channel codes (gran PER_ROW, natural layout, the fold indexed by
// column), both from the one load of the block's tile held in registers.  Re-reading the
// tile for the second role (from L2) put a second load latency in every block: 87 us for
// large_linear's [4096, 11008] weight against 76 us now.  The tile held across both roles
// needs about 98 registers; three blocks per SM (80, a few bytes spilled) measured 76 us, two (98) 93 us,
// four (64, spilling) 73 us on the wide weights but slower on small ones.
template <typename CodeT, bool FF, bool FD>
__global__ void __launch_bounds__(256, 3) quantize_weight_kernel(const QuantArgs af, const QuantArgs ad) {
  __shared__ __align__(16) uint8_t tile_t[kQC * 8 * 8 * sizeof(CodeT)];
  griddep_wait();
  const bool inside = (static_cast<int64_t>(blockIdx.y) + 1) * kQR <= af.R &&
                      (static_cast<int64_t>(blockIdx.x) + 1) * kQC <= af.C && af.vec_in;
  float4 xin[kQRowsPerWarp];   // both roles read the same tensor: af and ad share x, R, C, ld
  if (inside)
    load_quant_tile<true>(af, xin);
  else
    load_quant_tile<false>(af, xin);
  if (inside && af.vec_t)
    quantize_tile<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_NEAREST_EVEN, FF, true, false>(af, tile_t, xin);
  else
    quantize_tile<CodeT, SQ_GRAN_PER_COL, SQ_ROUND_NEAREST_EVEN, FF, false, false>(af, tile_t, xin);
  if (inside && ad.vec_out)
    quantize_tile<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_NEAREST_EVEN, FD, true, false>(ad, tile_t, xin);
  else
    quantize_tile<CodeT, SQ_GRAN_PER_ROW, SQ_ROUND_NEAREST_EVEN, FD, false, false>(ad, tile_t, xin);
}

template <typename CodeT>
static void launch_quantize_weight(const QuantArgs& af, const QuantArgs& ad, dim3 grid,
                                   cudaStream_t s) {
  const bool ff = af.fold != nullptr, fd = ad.fold != nullptr;
  if (ff && fd) launch_pdl(quantize_weight_kernel<CodeT, true, true>, grid, dim3(256), s, af, ad);
  else if (ff) launch_pdl(quantize_weight_kernel<CodeT, true, false>, grid, dim3(256), s, af, ad);
  else if (fd) launch_pdl(quantize_weight_kernel<CodeT, false, true>, grid, dim3(256), s, af, ad);
  else launch_pdl(quantize_weight_kernel<CodeT, false, false>, grid, dim3(256), s, af, ad);
}

// ============================================================ group order (Sec. 3.2)
// The inner index of a forward or loss-propagation GEMM in group order: every group's
// channels contiguous (stable: in channel order within a group), each group's segment
// starting on a K-block boundary (bk elements), so that the contraction can accumulate a
// group unshifted and apply its shift once per segment.  seg[0..G] = segment starts (seg[G]
// = the padded width), seg[G+1..2G] = channels per group; pos[c] = the position of channel
// c.  One block: counts per group, then stable ranks chunk by chunk with warp ballots.
constexpr int kOrderThreads = 1024;

__global__ void __launch_bounds__(kOrderThreads)
    group_order_kernel(const uint8_t* __restrict__ exp, int64_t C, int G, int bk,
                       int* __restrict__ pos, int* __restrict__ seg) {
  __shared__ int cnt[8];
  __shared__ int start[9];
  __shared__ int base[8];
  __shared__ int wtot[kOrderThreads / 32][8];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid < 8) cnt[tid] = 0;
  __syncthreads();
  int mine[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int64_t c = tid; c < C; c += kOrderThreads) {
    const int e = min(static_cast<int>(exp[c]), G - 1);
#pragma unroll
    for (int g = 0; g < 8; ++g) mine[g] += (e == g);
  }
#pragma unroll
  for (int g = 0; g < 8; ++g) {
    const int v = __reduce_add_sync(0xFFFFFFFFu, mine[g]);
    if (lane == 0 && v) atomicAdd(&cnt[g], v);
  }
  __syncthreads();
  if (tid == 0) {
    int o = 0;
    for (int g = 0; g < G; ++g) {
      start[g] = o;
      o += (cnt[g] + bk - 1) / bk * bk;
      base[g] = 0;
    }
    start[G] = o;
    for (int g = 0; g <= G; ++g) seg[g] = start[g];
    for (int g = 0; g < G; ++g) seg[G + 1 + g] = cnt[g];
  }
  __syncthreads();
  for (int64_t c0 = 0; c0 < C; c0 += kOrderThreads) {
    const int64_t c = c0 + tid;
    const int e = c < C ? min(static_cast<int>(exp[c]), G - 1) : -1;
    const unsigned below = (1u << lane) - 1u;
    int rank = 0;
#pragma unroll
    for (int g = 0; g < 8; ++g) {
      const unsigned b = __ballot_sync(0xFFFFFFFFu, e == g);
      if (e == g) rank = __popc(b & below);
      if (lane == 0) wtot[w][g] = __popc(b);
    }
    __syncthreads();
    if (e >= 0) {
      int before = 0;
      for (int k = 0; k < w; ++k) before += wtot[k][e];
      pos[c] = start[e] + base[e] + before + rank;
    }
    __syncthreads();
    if (tid < G) {
      int t = 0;
      for (int k = 0; k < kOrderThreads / 32; ++k) t += wtot[k][tid];
      base[tid] += t;
    }
    __syncthreads();
  }
}

// zero the padding positions of a group-ordered code buffer [rows, ld]: the tail
// [seg[g] + count_g, seg[g+1]) of every segment, one warp per row
template <typename CodeT>
__global__ void __launch_bounds__(256)
    order_pad_kernel(CodeT* __restrict__ codes, int64_t rows, int64_t ld, const int* __restrict__ seg,
                     int G) {
  const int lane = threadIdx.x & 31;
  for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) / 32; r < rows;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x / 32) {
    CodeT* row = codes + r * ld;
    for (int g = 0; g < G; ++g) {
      const int from = seg[g] + seg[G + 1 + g], to = seg[g + 1];
      for (int i = from + lane; i < to; i += 32) row[i] = CodeT(0);
    }
  }
}

// The range pass of x [rows, cols] (0 < rows, 0 < cols < 2^36, checked by the callers):
// one block per tile, narrow tensors in whole clusters along the rows; with
// row_bits also the per-row maxima.
static cudaError_t launch_range(const float* x, int64_t rows, int64_t cols, int64_t ld,
                                unsigned* col_bits, unsigned* row_bits, int* status,
                                cudaStream_t s) {
  // the tile: the column count rounded up to a power of two (4 .. 128) wide, 1024 elements;
  // a weight's row ranges need whole 128-column warp rows
  int lg = 5;
  if (row_bits == nullptr)
    for (lg = 0; lg < 5 && (int64_t(4) << lg) < cols; ++lg) {
    }
  const int64_t tc = int64_t(4) << lg;
  const int64_t cblocks = (cols + tc - 1) / tc;   // < 2^29: cols < 2^36, tc = 128 past 64
  const int64_t tiles = (rows + 8 * (256 >> lg) - 1) / (8 * (256 >> lg));
  const int cl = cols <= kRangeClusterMaxCols ? kRangeCluster : 1;
  const int vec = (ld % 4 == 0) && aligned16(x);
  if (row_bits != nullptr && cl == 1) {
    // a wide weight: runs of column blocks per block (weight_range_kernel)
    const int64_t runs = (cblocks + kWeightRun - 1) / kWeightRun;
    cudaLaunchConfig_t cfg;
    memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3(static_cast<unsigned>(runs), static_cast<unsigned>(tiles < 65535 ? tiles : 65535));
    cfg.blockDim = dim3(kColTx, kColTy);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t err = cudaLaunchKernelEx(&cfg, weight_range_kernel, x, rows, cols, ld, vec,
                                         col_bits, row_bits, status);
    if (err == cudaSuccess) err = cudaGetLastError();
    return err;
  }
  const int64_t max_rblocks = 65535 / cl * cl;
  int64_t rblocks = (tiles + cl - 1) / cl * cl;
  if (rblocks > max_rblocks) rblocks = max_rblocks;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(static_cast<unsigned>(cblocks), static_cast<unsigned>(rblocks));
  cfg.blockDim = dim3(kColTx, kColTy);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = cl;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cl > 1 ? 2 : 1;
  cudaError_t err;
  if (row_bits != nullptr)   // a narrow weight (wide ones returned above)
    err = cudaLaunchKernelEx(&cfg, colmax_kernel<kRangeCluster, true>, x, rows, cols, ld, vec, lg,
                             col_bits, row_bits, status);
  else
    err = cl > 1 ? cudaLaunchKernelEx(&cfg, colmax_kernel<kRangeCluster, false>, x, rows, cols, ld, vec,
                                      lg, col_bits, row_bits, status)
                 : cudaLaunchKernelEx(&cfg, colmax_kernel<1, false>, x, rows, cols, ld, vec, lg, col_bits,
                                      row_bits, status);
  if (err == cudaSuccess) err = cudaGetLastError();
  return err;
}

}  // namespace sq

using namespace sq;

// ===================================================================== C entry points
extern "C" int shiftquant_code_type(int bits, int n_groups) {
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "bits must be in [2, 8] and n_groups in [1, 8] (got %d, %d)", bits,
                n_groups);
  return code_type(bits, n_groups);
}

extern "C" int shiftquant_code_bytes(int bits, int n_groups) {
  const int t = shiftquant_code_type(bits, n_groups);
  return t < 0 ? t : code_bytes(t);
}

extern "C" const char* shiftquant_status_string(sq_status s) {
  switch (s) {
    case SQ_OK: return "ok";
    case SQ_EINVAL: return "invalid argument";
    case SQ_EALIGN: return "alignment";
    case SQ_EUNSUPPORTED: return "unsupported combination";
    case SQ_ECUDA: return "CUDA error";
    default: return "unknown status";
  }
}

extern "C" const char* shiftquant_last_error(void) { return g_last_error; }

extern "C" sq_status shiftquant_calibrate(const float* x, int64_t rows, int64_t cols,
                                          int64_t ld, int gran, int n_groups,
                                          float* range_out, float* tau0_out, uint8_t* exp_out,
                                          int32_t* dev_status, void* stream) {
  clear_error();
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "calibrate: negative size");
  if (cols >= (int64_t(1) << 36)) return fail(SQ_EINVAL, "calibrate: too many columns");
  if (gran < SQ_GRAN_SHIFT || gran > SQ_GRAN_PER_ROW) return fail(SQ_EINVAL, "calibrate: bad gran %d", gran);
  if (gran == SQ_GRAN_SHIFT && !groups_ok(n_groups))
    return fail(SQ_EINVAL, "calibrate: n_groups must be in [1, 8]");
  if (rows > 0 && cols > 0 && (x == nullptr || ld < cols))
    return fail(SQ_EINVAL, "calibrate: x is NULL or ld < cols");
  const int64_t channels = gran == SQ_GRAN_PER_ROW ? rows : cols;
  if (dev_status == nullptr || (channels > 0 && range_out == nullptr))
    return fail(SQ_EINVAL, "calibrate: range_out and dev_status are required");
  if (gran == SQ_GRAN_SHIFT && (tau0_out == nullptr || (cols > 0 && exp_out == nullptr)))
    return fail(SQ_EINVAL, "calibrate: SHIFT needs tau0_out and exp_out");
  cudaStream_t s = as_stream(stream);
  cudaError_t err;
  if (gran == SQ_GRAN_PER_ROW) {
    if (rows == 0) return SQ_OK;
    if (cols == 0) {
      err = cudaMemsetAsync(range_out, 0, sizeof(float) * rows, s);
      return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemsetAsync");
    }
    const int vec = (ld % 4 == 0) && aligned16(x);
    const int per_block = 8;
    const int64_t blocks = (rows + per_block - 1) / per_block;
    rowmax_kernel<<<static_cast<unsigned>(blocks), per_block * 32, 0, s>>>(x, rows, cols, ld, vec,
                                                                           range_out, dev_status);
    err = cudaGetLastError();
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "rowmax_kernel launch");
  }
  const bool shift = gran == SQ_GRAN_SHIFT;
  if (rows == 0 || cols == 0) {
    // every range is 0: tau_0 = 0 and every channel in the last group
    if (cols > 0) {
      err = cudaMemsetAsync(range_out, 0, sizeof(float) * cols, s);
      if (err == cudaSuccess && shift) err = cudaMemsetAsync(exp_out, n_groups - 1, cols, s);
      if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
    }
    if (shift) {
      err = cudaMemsetAsync(tau0_out, 0, sizeof(float), s);
      if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
    }
    return SQ_OK;
  }
  {
    const int64_t iblocks = (cols + 255) / 256;
    calib_init_kernel<<<static_cast<unsigned>(iblocks < 1024 ? iblocks : 1024), 256, 0, s>>>(
        reinterpret_cast<unsigned*>(range_out), cols, nullptr, 0);
    err = cudaGetLastError();
    if (err != cudaSuccess) return cuda_fail(err, "calib_init_kernel launch");
  }
  unsigned* bits = reinterpret_cast<unsigned*>(range_out);
  err = launch_range(x, rows, cols, ld, bits, nullptr, dev_status, s);
  if (err != cudaSuccess) return cuda_fail(err, "colmax_kernel launch");
  if (!shift) return SQ_OK;
  // grouping (Eq. 3) by one block behind the range pass
  err = cols <= static_cast<int64_t>(kGroupSmallThreads) * kGroupPerThread
            ? launch_pdl(group_kernel<kGroupSmallThreads>, dim3(1), dim3(kGroupSmallThreads), s,
                         static_cast<const unsigned*>(bits), cols, n_groups, tau0_out, exp_out, dev_status)
            : launch_pdl(group_kernel<kGroupLargeThreads>, dim3(1), dim3(kGroupLargeThreads), s,
                         static_cast<const unsigned*>(bits), cols, n_groups, tau0_out, exp_out, dev_status);
  if (err == cudaSuccess) err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "group_kernel launch");
}

extern "C" sq_status shiftquant_group(const float* range, int64_t channels, int n_groups,
                                      float* tau0_out, uint8_t* exp_out, int32_t* dev_status,
                                      void* stream) {
  clear_error();
  if (!groups_ok(n_groups)) return fail(SQ_EINVAL, "group: n_groups must be in [1, 8]");
  if (channels < 0) return fail(SQ_EINVAL, "group: negative size");
  if (tau0_out == nullptr || dev_status == nullptr || (channels > 0 && (range == nullptr || exp_out == nullptr)))
    return fail(SQ_EINVAL, "group: range, tau0_out, exp_out and dev_status are required");
  cudaStream_t s = as_stream(stream);
  if (channels == 0) {
    const cudaError_t err = cudaMemsetAsync(tau0_out, 0, sizeof(float), s);
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemsetAsync");
  }
  const unsigned* rb = reinterpret_cast<const unsigned*>(range);
  if (channels <= static_cast<int64_t>(kGroupSmallThreads) * kGroupPerThread)
    group_kernel<kGroupSmallThreads><<<1, kGroupSmallThreads, 0, s>>>(rb, channels, n_groups, tau0_out,
                                                                     exp_out, dev_status);
  else
    group_kernel<kGroupLargeThreads><<<1, kGroupLargeThreads, 0, s>>>(rb, channels, n_groups, tau0_out,
                                                                     exp_out, dev_status);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "group_kernel launch");
}

extern "C" sq_status shiftquant_quantize(const float* x, int64_t rows, int64_t cols, int64_t ld,
                                         int gran, int bits, int n_groups,
                                         const float* range_or_tau0, const uint8_t* exp,
                                         const uint8_t* fold_exp, int mode, uint64_t seed,
                                         int64_t row0, void* codes, int64_t ld_codes,
                                         void* codes_t, int64_t ld_t, float* scale_out,
                                         void* stream) {
  clear_error();
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "quantize: bits must be in [2, 8] and n_groups in [1, 8]");
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "quantize: negative size");
  if (row0 < 0) return fail(SQ_EINVAL, "quantize: negative row0");
  if (gran < SQ_GRAN_SHIFT || gran > SQ_GRAN_PER_ROW) return fail(SQ_EINVAL, "quantize: bad gran");
  if (mode != SQ_ROUND_NEAREST_EVEN && mode != SQ_ROUND_STOCHASTIC)
    return fail(SQ_EINVAL, "quantize: bad rounding mode");
  if (gran == SQ_GRAN_SHIFT && fold_exp != nullptr)
    return fail(SQ_EINVAL, "quantize: SHIFT takes no fold_exp");
  cudaStream_t s = as_stream(stream);
  const int type = code_type(bits, n_groups);
  const int cbytes = code_bytes(type);
  if (rows == 0 || cols == 0) {
    // every range is 0: scales are 0 and there is no code to write
    const int64_t n = gran == SQ_GRAN_SHIFT ? 1 : (gran == SQ_GRAN_PER_COL ? cols : rows);
    if (n == 0) return SQ_OK;
    if (scale_out == nullptr) return fail(SQ_EINVAL, "quantize: scale_out is required");
    cudaError_t err = cudaMemsetAsync(scale_out, 0, sizeof(float) * n, s);
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemsetAsync");
  }
  if (range_or_tau0 == nullptr || scale_out == nullptr)
    return fail(SQ_EINVAL, "quantize: range_or_tau0 and scale_out are required");
  if (gran == SQ_GRAN_SHIFT && exp == nullptr)
    return fail(SQ_EINVAL, "quantize: SHIFT needs exp");
  if (codes == nullptr && codes_t == nullptr)
    return fail(SQ_EINVAL, "quantize: at least one of codes / codes_t is required");
  if (codes && ld_codes < cols) return fail(SQ_EINVAL, "quantize: ld_codes < cols");
  if (codes_t && ld_t < rows) return fail(SQ_EINVAL, "quantize: ld_t < rows");
  if (x == nullptr || ld < cols) return fail(SQ_EINVAL, "quantize: x is NULL or ld < cols");
  QuantArgs a;
  a.x = x;
  a.R = rows;
  a.C = cols;
  a.ld = ld;
  a.gran = gran;
  a.Q = q_of_bits(bits);
  a.G = n_groups;
  a.mode = mode;
  a.seed = seed;
  a.row0 = row0;
  a.rt = range_or_tau0;
  a.exp = exp;
  a.fold = fold_exp;
  a.codes = codes;
  a.ldc = ld_codes;
  a.codes_t = codes_t;
  a.ldt = ld_t;
  a.scale_out = scale_out;
  a.vec_in = (ld % 4 == 0) && aligned16(x);
  a.vec_out = codes != nullptr && ((ld_codes * cbytes) % (4 * cbytes) == 0) &&
              (reinterpret_cast<uintptr_t>(codes) % (4 * cbytes) == 0);
  a.vec_t = codes_t != nullptr && ((ld_t * cbytes) % 16 == 0) && aligned16(codes_t);
  a.pos_cols = g_order_cols;
  a.pos_rows = g_order_rows;
  const int64_t gx = (cols + kQC - 1) / kQC, gy = (rows + kQR - 1) / kQR;
  if (gx > 0x7FFFFFFF || gy > 65535)
    return fail(SQ_EUNSUPPORTED, "quantize: tensor too large for one launch (%lld x %lld)",
                static_cast<long long>(rows), static_cast<long long>(cols));
  dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
  if (type == SQ_CODE_E4M3)
    launch_quantize<uint8_t>(a, grid, s);
  else
    launch_quantize<uint16_t>(a, grid, s);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "quantize_kernel launch");
}

// ------------------------------------------------------------------ group order
extern "C" int64_t shiftquant_group_order_width(int64_t channels, int bits, int n_groups) {
  if (channels < 0 || !bits_ok(bits) || !groups_ok(n_groups)) return -1;
  const int64_t bk = 128 / code_bytes(code_type(bits, n_groups));
  return (channels + bk - 1) / bk * bk + (n_groups - 1) * bk;
}

extern "C" sq_status shiftquant_group_order(const uint8_t* exp, int64_t channels, int bits,
                                            int n_groups, int32_t* pos_out, int32_t* seg_out,
                                            void* stream) {
  clear_error();
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "group_order: bits must be in [2, 8] and n_groups in [1, 8]");
  if (channels < 0 || channels > INT32_MAX / 2) return fail(SQ_EINVAL, "group_order: bad channel count");
  if (seg_out == nullptr || (channels > 0 && (exp == nullptr || pos_out == nullptr)))
    return fail(SQ_EINVAL, "group_order: exp, pos_out and seg_out are required");
  const int bk = 128 / code_bytes(code_type(bits, n_groups));
  group_order_kernel<<<1, kOrderThreads, 0, as_stream(stream)>>>(exp, channels, n_groups, bk,
                                                                   pos_out, seg_out);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "group_order_kernel launch");
}

extern "C" sq_status shiftquant_quantize_ordered(const float* x, int64_t rows, int64_t cols,
                                                 int64_t ld, int gran, int bits, int n_groups,
                                                 const float* range_or_tau0, const uint8_t* exp,
                                                 int mode, uint64_t seed, int64_t row0,
                                                 const int32_t* pos, const int32_t* seg,
                                                 void* codes, int64_t ld_codes, void* codes_t,
                                                 int64_t ld_t, float* scale_out, void* stream) {
  clear_error();
  if (pos == nullptr || seg == nullptr) return fail(SQ_EINVAL, "quantize_ordered: pos and seg are required");
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "quantize_ordered: bits must be in [2, 8] and n_groups in [1, 8]");
  // the ordered output: codes for ShiftQuant and per-row grans, codes_t for per-column
  const bool on_t = gran == SQ_GRAN_PER_COL;
  void* ordered = on_t ? codes_t : codes;
  const int64_t ord_rows = on_t ? cols : rows;       // rows of the ordered buffer
  const int64_t ord_ld = on_t ? ld_t : ld_codes;
  const int64_t chans = on_t ? rows : cols;          // the ordered (inner) index
  if (ordered == nullptr)
    return fail(SQ_EINVAL, "quantize_ordered: the group-ordered output (%s) is required",
                on_t ? "codes_t" : "codes");
  const int64_t width = shiftquant_group_order_width(chans, bits, n_groups);
  if (ord_ld < width)
    return fail(SQ_EINVAL, "quantize_ordered: the ordered output needs a leading dimension of "
                "at least %lld (shiftquant_group_order_width)", static_cast<long long>(width));
  // the other output (if any) keeps the natural order; a leading dimension >= the natural
  // width is checked by the plain quantizer below
  g_order_cols = on_t ? nullptr : pos;
  g_order_rows = on_t ? pos : nullptr;
  const sq_status st = shiftquant_quantize(x, rows, cols, ld, gran, bits, n_groups, range_or_tau0,
                                           exp, nullptr, mode, seed, row0, codes, ld_codes, codes_t,
                                           ld_t, scale_out, stream);
  g_order_cols = g_order_rows = nullptr;
  if (st != SQ_OK || ord_rows == 0) return st;
  cudaStream_t s = as_stream(stream);
  int64_t blocks = (ord_rows + 7) / 8;
  if (blocks > 4096) blocks = 4096;
  if (code_type(bits, n_groups) == SQ_CODE_E4M3)
    order_pad_kernel<uint8_t><<<static_cast<unsigned>(blocks), 256, 0, s>>>(
        static_cast<uint8_t*>(ordered), ord_rows, ord_ld, seg, n_groups);
  else
    order_pad_kernel<uint16_t><<<static_cast<unsigned>(blocks), 256, 0, s>>>(
        static_cast<uint16_t*>(ordered), ord_rows, ord_ld, seg, n_groups);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "order_pad_kernel launch");
}

extern "C" sq_status shiftquant_calibrate_weight(const float* w, int64_t rows, int64_t cols,
                                                 int64_t ld, float* range_out_ch,
                                                 float* range_in_ch, int32_t* dev_status,
                                                 void* stream) {
  clear_error();
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "calibrate_weight: negative size");
  if (cols >= (int64_t(1) << 36)) return fail(SQ_EINVAL, "calibrate_weight: too many columns");
  if (rows > 0 && cols > 0 && (w == nullptr || ld < cols))
    return fail(SQ_EINVAL, "calibrate_weight: w is NULL or ld < cols");
  if (dev_status == nullptr || (cols > 0 && range_out_ch == nullptr) ||
      (rows > 0 && range_in_ch == nullptr))
    return fail(SQ_EINVAL, "calibrate_weight: range_out_ch, range_in_ch and dev_status are required");
  cudaStream_t s = as_stream(stream);
  cudaError_t err;
  if (rows == 0 || cols == 0) {
    // every range is 0
    if (cols > 0 && (err = cudaMemsetAsync(range_out_ch, 0, sizeof(float) * cols, s)) != cudaSuccess)
      return cuda_fail(err, "cudaMemsetAsync");
    if (rows > 0 && (err = cudaMemsetAsync(range_in_ch, 0, sizeof(float) * rows, s)) != cudaSuccess)
      return cuda_fail(err, "cudaMemsetAsync");
    return SQ_OK;
  }
  unsigned* cb = reinterpret_cast<unsigned*>(range_out_ch);
  unsigned* rb = reinterpret_cast<unsigned*>(range_in_ch);
  // Both ranges from one read.  On wide weights the blocks of one row tile run together and
  // their per-row atomics (one per 128 columns) partly serialise; measured on a
  // [4096, 11008] weight this pass (58 us) still beats a column pass plus a one-warp-per-row
  // pass (34 + 30 us).
  const int64_t n = rows > cols ? rows : cols;
  const int64_t iblocks = (n + 255) / 256;
  calib_init_kernel<<<static_cast<unsigned>(iblocks < 1024 ? iblocks : 1024), 256, 0, s>>>(
      cb, cols, rb, rows);
  err = cudaGetLastError();
  if (err != cudaSuccess) return cuda_fail(err, "calib_init_kernel launch");
  err = launch_range(w, rows, cols, ld, cb, rb, dev_status, s);
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "colmax_kernel launch");
}

extern "C" sq_status shiftquant_quantize_weight(const float* w, int64_t rows, int64_t cols,
                                                int64_t ld, int bits, int n_groups,
                                                const float* range_out_ch, const float* range_in_ch,
                                                const uint8_t* fold_fwd, const uint8_t* fold_dgrad,
                                                void* codes_fwd, int64_t ld_fwd, float* scale_fwd,
                                                void* codes_dgrad, int64_t ld_dgrad,
                                                float* scale_dgrad, void* stream) {
  clear_error();
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "quantize_weight: bits must be in [2, 8] and n_groups in [1, 8]");
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "quantize_weight: negative size");
  cudaStream_t s = as_stream(stream);
  const int type = code_type(bits, n_groups);
  const int cbytes = code_bytes(type);
  if (rows == 0 || cols == 0) {
    // every range is 0: the scales are 0 and there is no code to write
    cudaError_t err;
    if (cols > 0) {
      if (scale_fwd == nullptr) return fail(SQ_EINVAL, "quantize_weight: scale_fwd is required");
      if ((err = cudaMemsetAsync(scale_fwd, 0, sizeof(float) * cols, s)) != cudaSuccess)
        return cuda_fail(err, "cudaMemsetAsync");
    }
    if (rows > 0) {
      if (scale_dgrad == nullptr) return fail(SQ_EINVAL, "quantize_weight: scale_dgrad is required");
      if ((err = cudaMemsetAsync(scale_dgrad, 0, sizeof(float) * rows, s)) != cudaSuccess)
        return cuda_fail(err, "cudaMemsetAsync");
    }
    return SQ_OK;
  }
  if (w == nullptr || ld < cols) return fail(SQ_EINVAL, "quantize_weight: w is NULL or ld < cols");
  if (range_out_ch == nullptr || range_in_ch == nullptr || scale_fwd == nullptr ||
      scale_dgrad == nullptr || codes_fwd == nullptr || codes_dgrad == nullptr)
    return fail(SQ_EINVAL, "quantize_weight: ranges, codes and scales of both roles are required");
  if (ld_fwd < rows) return fail(SQ_EINVAL, "quantize_weight: ld_fwd < rows");
  if (ld_dgrad < cols) return fail(SQ_EINVAL, "quantize_weight: ld_dgrad < cols");
  QuantArgs af;
  memset(&af, 0, sizeof(af));
  af.x = w;
  af.R = rows;
  af.C = cols;
  af.ld = ld;
  af.gran = SQ_GRAN_PER_COL;
  af.Q = q_of_bits(bits);
  af.G = n_groups;
  af.mode = SQ_ROUND_NEAREST_EVEN;
  af.vec_in = (ld % 4 == 0) && aligned16(w);
  QuantArgs ad = af;
  af.rt = range_out_ch;
  af.fold = fold_fwd;
  af.codes_t = codes_fwd;
  af.ldt = ld_fwd;
  af.scale_out = scale_fwd;
  af.vec_t = ((ld_fwd * cbytes) % 16 == 0) && aligned16(codes_fwd);
  ad.gran = SQ_GRAN_PER_ROW;
  ad.rt = range_in_ch;
  ad.fold = fold_dgrad;
  ad.codes = codes_dgrad;
  ad.ldc = ld_dgrad;
  ad.scale_out = scale_dgrad;
  ad.vec_out = ((ld_dgrad * cbytes) % (4 * cbytes) == 0) &&
               (reinterpret_cast<uintptr_t>(codes_dgrad) % (4 * cbytes) == 0);
  const int64_t gx = (cols + kQC - 1) / kQC, gy = (rows + kQR - 1) / kQR;
  if (gx > 0x7FFFFFFF || gy > 65535)
    return fail(SQ_EUNSUPPORTED, "quantize_weight: tensor too large for one launch (%lld x %lld)",
                static_cast<long long>(rows), static_cast<long long>(cols));
  const dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
  if (type == SQ_CODE_E4M3)
    launch_quantize_weight<uint8_t>(af, ad, grid, s);
  else
    launch_quantize_weight<uint16_t>(af, ad, grid, s);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "quantize_weight_kernel launch");
}
