// Fully-quantized L1 batch normalization (Sec. 4, App. C) on sm_103a.
//
// Forward over x [R, C] (channels = columns; the R rows are the batch and spatial
// positions), with the readings of the paper that the oracle states:
//   - x by ShiftQuant (round to nearest) to int8 codes q with per-channel steps s_c;
//   - the mean onto the channel's code grid, m_c = round-half-even(sum_r q / R), so that
//     x^q - mu^q = (q - m) s_c is an integer code difference;
//   - sigma_c = (sum_r |q - m| / R) s_c, the mean absolute deviation (L1 normalization);
//   - sigma, gamma and beta on 8-bit symmetric per-tensor grids;
//   - y = gamma^q (x^q - mu^q) / sigma^q + beta^q (beta^q where sigma^q = 0).
// Backward from dy: ShiftQuant with stochastic rounding to int8 codes p, then
//   dx = (gamma / sigma)(g - mean g - mean(g xhat)(sign(q - m) - mean sign(q - m))),
//   dgamma = sum g xhat, dbeta = sum g.
// Every sum over a channel is an exact integer (sums of codes, of |q - m|, of signs, of
// p (q - m)); each binary32 step is one IEEE operation in a fixed order (this file compiles
// with -fmad=false), so the results are reproducible bit for bit.
//
// Kernels, all streaming HBM passes over a tile of TC columns (the channel count rounded
// up to a power of two, at most 128) whose 256 threads each own one four-column quad and
// every (1024 / TC)-th row, with 8 (fp32) or 16 (code) loads in flight: a column-reduction
// pass that quantizes and sums, a second reduction over the 1-byte codes for the deviation
// sums, a one-block pass for the per-channel values, and an elementwise output pass whose
// threads keep their quad's per-channel constants in registers.  Channel sums go from
// shared memory to global 64-bit atomics into one of kSpread slots per sum (the block row
// modulo kSpread), so that same-address atomics from hundreds of blocks do not serialise;
// readers add the slots.  Every kernel after the range pass is launched behind the one
// before it (programmatic stream serialization).
#include <cuda_runtime.h>

#include <cstring>

#include "sq_device.cuh"
#include "sq_host.h"
#include "sq_quant_dev.cuh"

namespace sq {

// per-channel float arrays of the state
enum {
  kChXRange, kChGRange, kChS, kChM, kChSig, kChSq, kChGq, kChBq, kChT, kChU, kChMg, kChMgx,
  kChZs, kNumChan
};
// per-channel int64 sums of the state, each kept in kSpread slots (block row y adds to slot
// y mod kSpread, so that same-address atomics from many blocks do not serialise; a reader
// adds the slots)
enum { kStS1, kStS, kStZ, kStP, kStD, kNumStats };
constexpr int kSpread = 8;
// scalars of the state
enum { kScXTau, kScXScale, kScGTau, kScGScale, kNumScal };

struct L1bnLayout {
  size_t xq, gq, stats, chan, lut, exps, scal, sync, total;
};

// the forward output of every code value per channel: lut[c][q + 127]
constexpr int kLutStride = 256;

static L1bnLayout l1bn_layout(int64_t R, int64_t C) {
  auto up = [](size_t n) { return (n + 255) & ~size_t(255); };
  const size_t n = static_cast<size_t>(R) * static_cast<size_t>(C);
  L1bnLayout L;
  size_t o = 0;
  L.xq = o;    o += up(n);
  L.gq = o;    o += up(n);
  L.stats = o; o += up(kNumStats * kSpread * static_cast<size_t>(C) * sizeof(long long));
  L.chan = o;  o += up(kNumChan * static_cast<size_t>(C) * sizeof(float));
  L.lut = o;   o += up(kLutStride * static_cast<size_t>(C) * sizeof(float));
  L.exps = o;  o += up(2 * static_cast<size_t>(C));
  L.scal = o;  o += 256;
  // the single-launch form's barrier counter (first 256 bytes) and the range pass's
  // per-column maxima in kSpread slot rows, zeroed before each call
  L.sync = o;  o += up(256 + kSpread * static_cast<size_t>(C) * sizeof(unsigned));
  L.total = o;
  return L;
}

struct L1bnArgs {
  int64_t R, C, ld_in, ld_out;
  int Q;
  uint64_t seed;
  const float* in;  // x (forward) or dy (backward)
  float* out;       // y or dx
  int8_t* xq;
  int8_t* gq;
  long long* st;  // [kNumStats][kSpread][C]
  float* ch;      // [kNumChan][C]
  float* lut;     // [C][kLutStride]
  uint8_t* xe;
  uint8_t* ge;
  float* scal;
  const float* gamma;
  const float* beta;
  float* dgamma;
  float* dbeta;
  int vec_in, vec_out;  // 16-byte rows: four elements per load / store
  unsigned* sync;       // single-launch form: barrier counter, then range slots [kSpread][C]
};

constexpr int kL1Threads = 256;
constexpr int kL1MaxCols = 128;   // widest tile: 32 quads
constexpr int kL1PassesF32 = 4;    // rows in flight per thread in the passes that read fp32
constexpr int kL1PassesCodes = 8;  // ... and in those that read only codes

__device__ __forceinline__ long long rne_div(long long a, long long b) {
  long long q = a / b, r = a % b;
  if (r < 0) {
    q -= 1;
    r += b;
  }
  if (2 * r > b || (2 * r == b && (q & 1))) q += 1;
  return q;
}

// channel sum k of column c: its slots added
__device__ __forceinline__ long long stat_sum(const long long* st, int k, int64_t C, int64_t c) {
  long long v = 0;
#pragma unroll
  for (int i = 0; i < kSpread; ++i) v += __ldcg(st + (static_cast<int64_t>(k) * kSpread + i) * C + c);
  return v;
}

// the slot row of statistic k that block row y adds to
__device__ __forceinline__ long long* stat_slot(long long* st, int k, int64_t C, int64_t y) {
  return st + (static_cast<int64_t>(k) * kSpread + y % kSpread) * C;
}

// A pass's block: its column tile x and row slab y of a gx x gy grid (the launch's own
// grid, or the part of a cooperative launch's blocks that runs the pass).
struct Blk {
  int64_t x, y, gx, gy;
};

__device__ __forceinline__ Blk launch_blk() {
  return Blk{blockIdx.x, blockIdx.y, gridDim.x, gridDim.y};
}

// The thread's place in a tile: its quad (four consecutive columns) and its first row.
struct TilePos {
  int tc;        // tile columns: 4 << lg
  int rpp;       // rows per pass: 256 / (tc / 4)
  int qc, ro;    // this thread's quad and row offset
  int64_t c;     // its first column
};

__device__ __forceinline__ TilePos tile_pos(int lg, const Blk& b) {
  TilePos t;
  t.tc = 4 << lg;
  t.rpp = kL1Threads >> lg;
  t.qc = threadIdx.x & ((1 << lg) - 1);
  t.ro = threadIdx.x >> lg;
  t.c = b.x * t.tc + 4 * t.qc;
  return t;
}

// the four elements of a quad at p (its first column c; zeros past C)
__device__ __forceinline__ void load4(const float* p, int64_t c, int64_t C, bool vec, float v[4]) {
  if (vec && c + 3 < C) {
    const float4 t = ld_stream_v4(p);
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) v[j] = c + j < C ? __ldg(p + j) : 0.0f;
  }
}

// the four codes of a quad at p packed in one word, byte j = column c + j (zeros past C).
// COH: codes written earlier in the same launch (the single-launch form): coherent loads
// through L2, not the read-only path, which holds only data no part of the launch writes.
template <bool COH = false>
__device__ __forceinline__ uint32_t load_codes_w(const int8_t* p, int64_t c, int64_t C) {
  if ((C & 3) == 0)
    return COH ? __ldcg(reinterpret_cast<const unsigned int*>(p)) : __ldg(reinterpret_cast<const unsigned int*>(p));
  uint32_t w = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (c + j < C) {
      const int8_t v = COH ? __ldcg(p + j) : p[j];
      w |= static_cast<uint32_t>(static_cast<uint8_t>(v)) << (8 * j);
    }
  return w;
}

__device__ __forceinline__ int code_at(uint32_t w, int j) {
  return static_cast<int>(static_cast<int8_t>(static_cast<uint8_t>(w >> (8 * j))));
}

__device__ __forceinline__ void store_codes4(int8_t* p, int64_t c, int64_t C, const int q[4]) {
  if ((C & 3) == 0) {
    *reinterpret_cast<char4*>(p) = make_char4(static_cast<signed char>(q[0]), static_cast<signed char>(q[1]),
                                              static_cast<signed char>(q[2]), static_cast<signed char>(q[3]));
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (c + j < C) p[j] = static_cast<int8_t>(q[j]);
  }
}

__device__ __forceinline__ void store4(float* p, int64_t c, int64_t C, bool vec, const float y[4]) {
  if (vec && c + 3 < C) {
    *reinterpret_cast<float4*>(p) = make_float4(y[0], y[1], y[2], y[3]);
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (c + j < C) p[j] = y[j];
  }
}

// The rows of a thread: block row y takes rows y rpp + ro, then every S = gridDim.y rpp-th
// row after it; U of them are in flight per step (their loads first, then their work).
struct RowWalk {
  int64_t r, S;
};

__device__ __forceinline__ RowWalk row_walk(const TilePos& t, const Blk& b) {
  RowWalk w;
  w.r = b.y * t.rpp + t.ro;
  w.S = b.gy * t.rpp;
  return w;
}

// Shared memory of a reduction block: every thread's NS x 4 partial sums.
template <int NS>
struct RedSmem {
  long long part[NS][kL1Threads * 4];
};

// The block's column sums of NS statistics -> global (dst[k]: the block's slot row of
// statistic k): acc[k][j] is this thread's sum over its rows for column t.c + j.
template <int NS>
__device__ __forceinline__ void red_end(const long long (&acc)[NS][4], long long* const (&dst)[NS],
                                        const TilePos& t, int64_t C, RedSmem<NS>& sm, const Blk& b) {
#pragma unroll
  for (int k = 0; k < NS; ++k)
#pragma unroll
    for (int j = 0; j < 4; ++j) sm.part[k][t.ro * t.tc + t.qc * 4 + j] = acc[k][j];
  __syncthreads();
  const int tid = threadIdx.x;
  long long tot[NS];
#pragma unroll
  for (int k = 0; k < NS; ++k) {
    tot[k] = 0;
    if (tid < t.tc)
      for (int r = 0; r < t.rpp; ++r) tot[k] += sm.part[k][r * t.tc + tid];
  }
  const int64_t c = b.x * t.tc + tid;
  if (tid < t.tc && c < C) {
#pragma unroll
    for (int k = 0; k < NS; ++k)
      if (tot[k] != 0)
        atomicAdd(reinterpret_cast<unsigned long long*>(dst[k] + c), static_cast<unsigned long long>(tot[k]));
  }
}

// Forward pass 1: x -> int8 ShiftQuant codes (round to nearest), sum of codes per channel.
// tau: tau_0; the exponent of column c is ex[c - ex0].
__device__ __forceinline__ void fwd_quant_pass(const L1bnArgs& a, int lg, const Blk& b, float tau,
                                               const uint8_t* ex, int64_t ex0, RedSmem<1>& sm) {
  const TilePos t = tile_pos(lg, b);
  const float Qf = static_cast<float>(a.Q);
  const float invS = __fdiv_rn(Qf, tau);
  const bool zero = !(tau > 0.0f) || !isfinite(tau) || !isfinite(invS);
  int e[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) e[j] = t.c + j < a.C ? ex[t.c + j - ex0] : 0;
  long long acc[1][4] = {{0, 0, 0, 0}};
  constexpr int U = kL1PassesF32;
  if (t.c < a.C) {
    RowWalk w = row_walk(t, b);
    const float* px = a.in + w.r * a.ld_in + t.c;
    int8_t* pq = a.xq + w.r * a.C + t.c;
    const int64_t sx = w.S * a.ld_in, sq = w.S * a.C;
    for (; w.r < a.R; w.r += U * w.S, px += U * sx, pq += U * sq) {
      float v[U][4];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (w.r + u * w.S < a.R) load4(px + u * sx, t.c, a.C, a.vec_in, v[u]);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (w.r + u * w.S >= a.R) break;
        int q[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          q[j] = t.c + j < a.C ? shift_code(v[u][j], e[j], invS, zero, Qf, false, 0, 0) : 0;
          acc[0][j] += q[j];
        }
        store_codes4(pq + u * sq, t.c, a.C, q);
      }
    }
  }
  long long* const dst[1] = {stat_slot(a.st, kStS1, a.C, b.y)};
  red_end<1>(acc, dst, t, a.C, sm, b);
  if (b.x == 0 && b.y == 0 && threadIdx.x == 0) a.scal[kScXScale] = zero ? 0.0f : __fdiv_rn(tau, Qf);
}

__global__ void __launch_bounds__(kL1Threads, 3) l1bn_fwd_quant_kernel(const L1bnArgs a, int lg) {
  // launched behind the previous kernel (programmatic stream serialization): wait for it
  // before reading anything it wrote, and let the next kernel start launching
  griddep_wait();
  griddep_launch_dependents();
  __shared__ RedSmem<1> sm;
  fwd_quant_pass(a, lg, launch_blk(), a.scal[kScXTau], a.xe, 0, sm);
}

// Forward pass 2: over the codes, sum |q - m| and sum sign(q - m) per channel, with
// m = round-half-even(sum q / R).  mean: shared scratch for the block's columns.
template <bool COH>
__device__ __forceinline__ void fwd_dev_pass(const L1bnArgs& a, int lg, const Blk& b, RedSmem<2>& sm,
                                             int* mean) {
  const TilePos t = tile_pos(lg, b);
  // the block's columns' means, from their sum slots, once per block
  {
    long long* fold = &sm.part[0][0];   // free until the block's reduction at the end
    const int64_t cb = b.x * t.tc;
    for (int i = threadIdx.x; i < kSpread * t.tc; i += kL1Threads) {
      const int slot = i / t.tc, col = i - slot * t.tc;
      fold[i] = cb + col < a.C ? __ldcg(a.st + (static_cast<int64_t>(kStS1) * kSpread + slot) * a.C + cb + col) : 0;
    }
    __syncthreads();
    if (threadIdx.x < t.tc) {
      long long v = 0;
#pragma unroll
      for (int k = 0; k < kSpread; ++k) v += fold[k * t.tc + threadIdx.x];
      mean[threadIdx.x] = static_cast<int>(rne_div(v, a.R));
    }
    __syncthreads();
  }
  int m[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) m[j] = t.c + j < a.C ? mean[4 * t.qc + j] : 0;
  long long acc[2][4] = {{0, 0, 0, 0}, {0, 0, 0, 0}};
  constexpr int U = kL1PassesCodes;
  if (t.c < a.C) {
    RowWalk w = row_walk(t, b);
    const int8_t* pq = a.xq + w.r * a.C + t.c;
    const int64_t sq = w.S * a.C;
    int sabs[4] = {0, 0, 0, 0}, ssgn[4] = {0, 0, 0, 0};
    int n = 0;
    for (; w.r < a.R; w.r += U * w.S, pq += U * sq) {
      uint32_t q[U];
#pragma unroll
      for (int u = 0; u < U; ++u) q[u] = w.r + u * w.S < a.R ? load_codes_w<COH>(pq + u * sq, t.c, a.C) : 0u;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (w.r + u * w.S >= a.R) break;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int d = code_at(q[u], j) - m[j];
          sabs[j] += abs(d);
          ssgn[j] += (d > 0) - (d < 0);
        }
      }
      // |d| <= 255: int sums of up to 2^23 rows stay exact; fold them into 64 bits by then
      if (++n == (1 << 20) / U) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[0][j] += sabs[j];
          acc[1][j] += ssgn[j];
          sabs[j] = ssgn[j] = 0;
        }
        n = 0;
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {   // columns past C: zero codes and m = 0, so d = 0
      acc[0][j] += sabs[j];
      acc[1][j] += ssgn[j];
    }
  }
  long long* const dst[2] = {stat_slot(a.st, kStS, a.C, b.y), stat_slot(a.st, kStZ, a.C, b.y)};
  red_end<2>(acc, dst, t, a.C, sm, b);
}

__global__ void __launch_bounds__(kL1Threads, 3) l1bn_fwd_dev_kernel(const L1bnArgs a, int lg) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ RedSmem<2> sm;
  __shared__ int mean[kL1MaxCols];
  fwd_dev_pass<false>(a, lg, launch_blk(), sm, mean);
}

// max over the block of non-negative values given as bit patterns
__device__ __forceinline__ uint32_t block_max(uint32_t v, uint32_t* red) {
  v = __reduce_max_sync(0xFFFFFFFFu, v);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) red[w] = v;
  __syncthreads();
  uint32_t m = 0;
  for (int k = 0; k < static_cast<int>(blockDim.x) / 32; ++k) m = max(m, red[k]);
  __syncthreads();
  return m;
}

// 8-bit symmetric per-tensor quantization of one value with the vector's maximum vmax
__device__ __forceinline__ float quant8(float v, float vmax) {
  const float inv = __fdiv_rn(127.0f, vmax), step = __fdiv_rn(vmax, 127.0f);
  const bool zero = !(vmax > 0.0f) || !isfinite(inv);
  float k = zero ? 0.0f : rintf(__fmul_rn(v, inv));
  k = fminf(fmaxf(k, -127.0f), 127.0f);
  return __fmul_rn(k, step);
}

// The forward statistics of channel c: its step s_c = s 2^-e_c, mean code m_c =
// round-half-even(sum q / R) and sigma_c = (sum |q - m| / R) s_c.
struct FwdChan {
  float s, m, sig;
};

__device__ __forceinline__ FwdChan fwd_chan_of(const L1bnArgs& a, int64_t c, float scale, float Rf) {
  FwdChan f;
  f.s = __fmul_rn(scale, pow2f(-static_cast<int>(__ldcg(a.xe + c))));
  f.m = static_cast<float>(rne_div(stat_sum(a.st, kStS1, a.C, c), a.R));
  f.sig = __fmul_rn(__fdiv_rn(__ll2float_rn(stat_sum(a.st, kStS, a.C, c)), Rf), f.s);
  return f;
}

// The output for code q of a channel with step s, mean code m and quantized sigma^q,
// gamma^q, beta^q: y = gamma^q (q s - m s) / sigma^q + beta^q (beta^q where sigma^q = 0).
__device__ __forceinline__ float l1bn_out_of(int q, float s, float m, float sq, float gq, float bq) {
  const float xq = __fmul_rn(static_cast<float>(q), s);
  const float mq = __fmul_rn(m, s);
  const float xhat = sq > 0.0f ? __fdiv_rn(__fsub_rn(xq, mq), sq) : 0.0f;
  return __fadd_rn(__fmul_rn(gq, xhat), bq);
}

// Forward pass 3 (one block): s_c, m_c, sigma_c, then sigma^q, gamma^q, beta^q.
__global__ void __launch_bounds__(1024) l1bn_fwd_chan_kernel(const L1bnArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ uint32_t red[32];
  const float Rf = __ll2float_rn(a.R);
  const float scale = a.scal[kScXScale];
  float* ch = a.ch;
  const int64_t C = a.C;
  uint32_t ms = 0, mg = 0, mb = 0;
  for (int64_t c = threadIdx.x; c < C; c += blockDim.x) {
    const FwdChan f = fwd_chan_of(a, c, scale, Rf);
    ch[kChS * C + c] = f.s;
    ch[kChM * C + c] = f.m;
    ch[kChSig * C + c] = f.sig;
    ms = max(ms, __float_as_uint(f.sig) & 0x7FFFFFFFu);
    mg = max(mg, __float_as_uint(a.gamma[c]) & 0x7FFFFFFFu);
    mb = max(mb, __float_as_uint(a.beta[c]) & 0x7FFFFFFFu);
  }
  const float smax = __uint_as_float(block_max(ms, red));
  const float gmax = __uint_as_float(block_max(mg, red));
  const float bmax = __uint_as_float(block_max(mb, red));
  for (int64_t c = threadIdx.x; c < C; c += blockDim.x) {
    ch[kChSq * C + c] = quant8(ch[kChSig * C + c], smax);
    ch[kChGq * C + c] = quant8(a.gamma[c], gmax);
    ch[kChBq * C + c] = quant8(a.beta[c], bmax);
  }
}

// Forward pass 3b (one block per channel): the output of every code value q in [-127, 127]
// in the output pass's operations and order.  A code takes at most 255 values, so the
// output pass looks its result up instead of dividing per element.
__global__ void __launch_bounds__(kLutStride) l1bn_fwd_lut_kernel(const L1bnArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t C = a.C, c = blockIdx.x;
  const float* ch = a.ch;
  const int q = static_cast<int>(threadIdx.x) - 127;
  a.lut[c * kLutStride + threadIdx.x] = l1bn_out_of(q, ch[kChS * C + c], ch[kChM * C + c],
                                                    ch[kChSq * C + c], ch[kChGq * C + c],
                                                    ch[kChBq * C + c]);
}

// zero n 64-bit channel sums (the first kernel of a call: nothing before it in the call)
__global__ void __launch_bounds__(256) l1bn_zero_kernel(long long* __restrict__ p, int64_t n) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    p[i] = 0;
}

// Forward pass 4: y = gamma^q ((x^q - mu^q) / sigma^q) + beta^q, looked up per code from
// lut, the block's columns' tables in shared memory.
template <bool COH>
__device__ __forceinline__ void fwd_out_pass(const L1bnArgs& a, int lg, const Blk& b, const float* lut) {
  const TilePos t = tile_pos(lg, b);
  const int64_t C = a.C;
  if (t.c >= C) return;
  constexpr int U = kL1PassesCodes;
  RowWalk w = row_walk(t, b);
  const int8_t* pq = a.xq + w.r * C + t.c;
  float* py = a.out + w.r * a.ld_out + t.c;
  const int64_t sq = w.S * C, sy = w.S * a.ld_out;
  const int col0 = 4 * t.qc * kLutStride + 127;
  for (; w.r < a.R; w.r += U * w.S, pq += U * sq, py += U * sy) {
    uint32_t q[U];
#pragma unroll
    for (int u = 0; u < U; ++u) q[u] = w.r + u * w.S < a.R ? load_codes_w<COH>(pq + u * sq, t.c, C) : 0u;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (w.r + u * w.S >= a.R) break;
      float y[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) y[j] = t.c + j < C ? lut[col0 + j * kLutStride + code_at(q[u], j)] : 0.0f;
      store4(py + u * sy, t.c, C, a.vec_out, y);
    }
  }
}

__global__ void __launch_bounds__(kL1Threads, 3) l1bn_fwd_out_kernel(const L1bnArgs a, int lg) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ float lut[];   // [tile columns][kLutStride]
  const int64_t cbase = static_cast<int64_t>(blockIdx.x) * (int64_t(4) << lg);
  const int ncol = static_cast<int>(min(int64_t(4) << lg, a.C - cbase));
  for (int i = threadIdx.x; i < ncol * kLutStride; i += kL1Threads)
    lut[i] = a.lut[cbase * kLutStride + i];
  __syncthreads();
  fwd_out_pass<false>(a, lg, launch_blk(), lut);
}

// Backward pass 1: dy -> int8 ShiftQuant codes p (stochastic rounding of element r C + c),
// sums of p and of p (q - m) per channel.  tau: dy's tau_0; the exponent of column c is
// ex[c - ex0].
__device__ __forceinline__ void bwd_quant_pass(const L1bnArgs& a, int lg, const Blk& b, float tau,
                                               const uint8_t* ex, int64_t ex0, RedSmem<2>& sm) {
  const TilePos t = tile_pos(lg, b);
  const float Qf = static_cast<float>(a.Q);
  const float invS = __fdiv_rn(Qf, tau);
  const bool zero = !(tau > 0.0f) || !isfinite(tau) || !isfinite(invS);
  int e[4], m[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    e[j] = t.c + j < a.C ? ex[t.c + j - ex0] : 0;
    m[j] = t.c + j < a.C ? static_cast<int>(a.ch[kChM * a.C + t.c + j]) : 0;
  }
  long long acc[2][4] = {{0, 0, 0, 0}, {0, 0, 0, 0}};
  constexpr int U = kL1PassesF32;
  if (t.c < a.C) {
    RowWalk w = row_walk(t, b);
    const float* pg = a.in + w.r * a.ld_in + t.c;
    const int8_t* px = a.xq + w.r * a.C + t.c;
    int8_t* pp = a.gq + w.r * a.C + t.c;
    const int64_t sg = w.S * a.ld_in, sc = w.S * a.C;
    for (; w.r < a.R; w.r += U * w.S, pg += U * sg, px += U * sc, pp += U * sc) {
      float v[U][4];
      uint32_t qx[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        qx[u] = 0u;
        if (w.r + u * w.S < a.R) {
          load4(pg + u * sg, t.c, a.C, a.vec_in, v[u]);
          qx[u] = load_codes_w(px + u * sc, t.c, a.C);
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t r = w.r + u * w.S;
        if (r >= a.R) break;
        int pc[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          pc[j] = t.c + j < a.C ? shift_code(v[u][j], e[j], invS, zero, Qf, true, a.seed,
                                             static_cast<uint64_t>(r * a.C + t.c + j))
                                : 0;
          acc[0][j] += pc[j];
          acc[1][j] += pc[j] * (code_at(qx[u], j) - m[j]);
        }
        store_codes4(pp + u * sc, t.c, a.C, pc);
      }
    }
  }
  long long* const dst[2] = {stat_slot(a.st, kStP, a.C, b.y), stat_slot(a.st, kStD, a.C, b.y)};
  red_end<2>(acc, dst, t, a.C, sm, b);
  if (b.x == 0 && b.y == 0 && threadIdx.x == 0) a.scal[kScGScale] = zero ? 0.0f : __fdiv_rn(tau, Qf);
}

__global__ void __launch_bounds__(kL1Threads, 3) l1bn_bwd_quant_kernel(const L1bnArgs a, int lg) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ RedSmem<2> sm;
  bwd_quant_pass(a, lg, launch_blk(), a.scal[kScGTau], a.ge, 0, sm);
}

// The backward constants of channel c: dy's step t_c, u = gamma^q / sigma^q, mean g,
// mean(g xhat), mean sign(q - m), dgamma and dbeta.
struct BwdChan {
  float t, u, mg, mgx, zs, dg, db;
};

__device__ __forceinline__ BwdChan bwd_chan_of(const L1bnArgs& a, int64_t c, float gscale, float Rf) {
  const int64_t C = a.C;
  const float* ch = a.ch;
  BwdChan k;
  k.t = __fmul_rn(gscale, pow2f(-static_cast<int>(__ldcg(a.ge + c))));
  const float sq = ch[kChSq * C + c], s = ch[kChS * C + c];
  const float P = __ll2float_rn(stat_sum(a.st, kStP, C, c));
  k.u = sq > 0.0f ? __fdiv_rn(ch[kChGq * C + c], sq) : 0.0f;
  k.mg = __fdiv_rn(__fmul_rn(P, k.t), Rf);
  k.dg = sq > 0.0f ? __fdiv_rn(__fmul_rn(__fmul_rn(__ll2float_rn(stat_sum(a.st, kStD, C, c)), k.t), s), sq)
                   : 0.0f;
  k.mgx = __fdiv_rn(k.dg, Rf);
  k.zs = __fdiv_rn(__ll2float_rn(stat_sum(a.st, kStZ, C, c)), Rf);
  k.db = __fmul_rn(P, k.t);
  return k;
}

// channel c's backward constants into the state (for the output pass), dgamma and dbeta
__device__ __forceinline__ void put_bwd_chan(const L1bnArgs& a, int64_t c, const BwdChan& k) {
  const int64_t C = a.C;
  float* ch = a.ch;
  ch[kChT * C + c] = k.t;
  ch[kChU * C + c] = k.u;
  ch[kChMg * C + c] = k.mg;
  ch[kChMgx * C + c] = k.mgx;
  ch[kChZs * C + c] = k.zs;
  a.dgamma[c] = k.dg;
  a.dbeta[c] = k.db;
}

// Backward pass 2: the per-channel constants of the input gradient, dgamma and dbeta.
__global__ void __launch_bounds__(256) l1bn_bwd_chan_kernel(const L1bnArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  const float Rf = __ll2float_rn(a.R);
  const float gscale = a.scal[kScGScale];
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; c < a.C;
       c += static_cast<int64_t>(gridDim.x) * blockDim.x)
    put_bwd_chan(a, c, bwd_chan_of(a, c, gscale, Rf));
}

// Backward pass 3: dx = u ((g - mean g) - mean(g xhat) (sign(q - m) - mean sign)), the
// per-channel values of each thread's quad in registers; mean(g xhat) (sign - mean sign)
// takes one of three values per channel, formed once.  FROM_STATE: the constants come
// from the state (the channel pass wrote them); otherwise from kc[c - first column of the
// block's tile], formed by the caller with bwd_chan_of (the same operations), and the codes
// are read coherently (the single-launch form writes them in the same launch).
template <bool FROM_STATE>
__device__ __forceinline__ void bwd_out_pass(const L1bnArgs& a, int lg, const Blk& b, const BwdChan* kc) {
  const TilePos t = tile_pos(lg, b);
  if (t.c >= a.C) return;
  const float* ch = a.ch;
  const int64_t C = a.C;
  int m[4];
  float tt[4], mg[4], u4[4], k[4][3];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int64_t c = t.c + j < C ? t.c + j : C - 1;
    m[j] = static_cast<int>(ch[kChM * C + c]);
    float mgx, zs;
    if (FROM_STATE) {
      tt[j] = ch[kChT * C + c];
      mg[j] = ch[kChMg * C + c];
      u4[j] = ch[kChU * C + c];
      mgx = ch[kChMgx * C + c];
      zs = ch[kChZs * C + c];
    } else {
      const BwdChan& v = kc[c - b.x * t.tc];
      tt[j] = v.t;
      mg[j] = v.mg;
      u4[j] = v.u;
      mgx = v.mgx;
      zs = v.zs;
    }
#pragma unroll
    for (int sgn = -1; sgn <= 1; ++sgn) k[j][sgn + 1] = __fmul_rn(mgx, __fsub_rn(static_cast<float>(sgn), zs));
  }
  constexpr int U = kL1PassesCodes;
  RowWalk w = row_walk(t, b);
  const int8_t* pq = a.xq + w.r * C + t.c;
  const int8_t* pp = a.gq + w.r * C + t.c;
  float* pd = a.out + w.r * a.ld_out + t.c;
  const int64_t sc = w.S * C, sd = w.S * a.ld_out;
  for (; w.r < a.R; w.r += U * w.S, pq += U * sc, pp += U * sc, pd += U * sd) {
    uint32_t q[U], p[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const bool in = w.r + u * w.S < a.R;
      q[u] = in ? load_codes_w<!FROM_STATE>(pq + u * sc, t.c, C) : 0u;
      p[u] = in ? load_codes_w<!FROM_STATE>(pp + u * sc, t.c, C) : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (w.r + u * w.S >= a.R) break;
      float dx[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int d = code_at(q[u], j) - m[j];
        const float g = __fmul_rn(static_cast<float>(code_at(p[u], j)), tt[j]);
        const float kj = d > 0 ? k[j][2] : (d < 0 ? k[j][0] : k[j][1]);
        dx[j] = __fmul_rn(u4[j], __fsub_rn(__fsub_rn(g, mg[j]), kj));
      }
      store4(pd + u * sd, t.c, C, a.vec_out, dx);
    }
  }
}

__global__ void __launch_bounds__(kL1Threads, 3) l1bn_bwd_out_kernel(const L1bnArgs a, int lg) {
  griddep_wait();
  griddep_launch_dependents();
  bwd_out_pass<true>(a, lg, launch_blk(), nullptr);
}

// ------------------------------------------------------------- single-launch form
// For up to kCoopMaxChannels channels the passes of a call run as the phases of one
// cooperative launch (every block resident), separated by grid barriers: on the ResNet
// shapes the launch-to-launch gaps of the chain of kernels cost more than its HBM traffic.
// Each phase runs the same pass body as the multi-kernel form (the same operations in the
// same order, so the results are bit for bit the same); what the multi-kernel form reads
// back from the state between launches (tau_0, exponents, channel constants) each block
// forms here from the channel sums itself, for the columns it needs.
constexpr int kCoopMaxChannels = 1024;
constexpr int kCoopOutLg = 3;   // output-pass tiles of 32 columns (a 32 KB table per block)

// Grid barrier of a cooperative launch: the k-th barrier of a call waits until the
// counter (zeroed before the launch) reaches k gridDim.x.  A block's writes are ordered
// before its arrival by the block barrier and the arrival's release; the acquire load that
// sees the count orders the other blocks' writes before what the block reads next.
// (Measured with 456 blocks: 1.6 us a barrier; with full fences around a relaxed atomic,
// 2.0-2.2 us, also with the arrivals spread over up to 32 counters.)  Bounded: after
// kWaitBudgetNs the block records SQ_DEV_TIMEOUT and the call's blocks unwind (each gives
// up at its own next barrier).
// (arrive = false: the block waits without arriving -- the self-test of the expiry path.)
__device__ __forceinline__ bool grid_barrier(unsigned* ctr, unsigned target, int* status,
                                             bool arrive = true) {
  __shared__ int ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    if (arrive) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
    int good = 1;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if (v >= target) break;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        atomicOr(status, kDevTimeout);
        good = 0;
        break;
      }
      __nanosleep(32);
    }
    ok = good;
  }
  __syncthreads();
  return ok != 0;
}

// zero n 64-bit channel sums, spread over the launch's blocks
__device__ __forceinline__ void zero_sums(long long* p, int64_t n) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    p[i] = 0;
}

// Range pass of x (or dy): the per-column max |x| of the block's rows into slot row
// b.y mod kSpread of `slots` (ordered bit patterns), as shiftquant_calibrate forms them.
__device__ __forceinline__ void range_pass(const L1bnArgs& a, int lg, const Blk& b, unsigned* slots,
                                           RedSmem<1>& sm, int* status) {
  const TilePos t = tile_pos(lg, b);
  unsigned mx[4] = {0u, 0u, 0u, 0u};
  constexpr int U = kL1PassesF32;
  if (t.c < a.C) {
    RowWalk w = row_walk(t, b);
    const float* px = a.in + w.r * a.ld_in + t.c;
    const int64_t sx = w.S * a.ld_in;
    for (; w.r < a.R; w.r += U * w.S, px += U * sx) {
      float v[U][4];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (w.r + u * w.S < a.R) load4(px + u * sx, t.c, a.C, a.vec_in, v[u]);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (w.r + u * w.S >= a.R) break;
#pragma unroll
        for (int j = 0; j < 4; ++j) mx[j] = max(mx[j], __float_as_uint(v[u][j]) & 0x7FFFFFFFu);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) sm.part[0][t.ro * t.tc + t.qc * 4 + j] = mx[j];
  __syncthreads();
  const int tid = threadIdx.x;
  const int64_t c = b.x * t.tc + tid;
  if (tid < t.tc && c < a.C) {
    unsigned m = 0;
    for (int r = 0; r < t.rpp; ++r) m = max(m, static_cast<unsigned>(sm.part[0][r * t.tc + tid]));
    if (m != 0u) atomicMax(slots + (b.y % kSpread) * a.C + c, m);
    if (m >= 0x7F800000u) atomicOr(status, kDevNonFinite);
  }
  __syncthreads();   // sm is reused by the next phase
}

// range of column c: its slot rows' maximum (bit pattern)
__device__ __forceinline__ unsigned slot_range(const unsigned* slots, int64_t C, int64_t c) {
  unsigned m = 0;
#pragma unroll
  for (int i = 0; i < kSpread; ++i) m = max(m, __ldcg(slots + i * C + c));
  return m;
}

// After the range pass: tau_0 (the largest range) and the exponents of the block's tile
// columns (Eq. 3, as group_kernel forms them) into sexp; block 0 also stores the ranges,
// tau_0 and every exponent in the state.  Returns tau_0.
__device__ __forceinline__ float coop_group(const L1bnArgs& a, int lg, const Blk& b, int G,
                                            const unsigned* slots, float* range_out, float* tau_out,
                                            uint8_t* exp_out, uint8_t* sexp, uint32_t* red,
                                            int* status) {
  unsigned m = 0;
  for (int64_t c = threadIdx.x; c < a.C; c += kL1Threads) m = max(m, slot_range(slots, a.C, c));
  const unsigned tb = block_max(m, red);
  const float tau = __uint_as_float(tb);
  const bool nonfinite = tb >= 0x7F800000u;
  const int tc = 4 << lg;
  const int64_t c0 = b.x * tc;
  if (threadIdx.x < tc && c0 + threadIdx.x < a.C) {
    const unsigned r = slot_range(slots, a.C, c0 + threadIdx.x);
    sexp[threadIdx.x] = static_cast<uint8_t>(nonfinite ? 0 : group_exponent(__uint_as_float(r), tau, G));
  }
  if (blockIdx.x == 0) {
    for (int64_t c = threadIdx.x; c < a.C; c += kL1Threads) {
      const unsigned r = slot_range(slots, a.C, c);
      range_out[c] = __uint_as_float(r);
      exp_out[c] = static_cast<uint8_t>(nonfinite ? 0 : group_exponent(__uint_as_float(r), tau, G));
    }
    if (threadIdx.x == 0) {
      *tau_out = tau;
      if (nonfinite) atomicOr(status, kDevNonFinite);
    }
  }
  __syncthreads();
  return tau;
}

struct CoopGeom {
  int lg, gx, gy;     // reduction passes: tile columns 4 << lg, gx x gy blocks
  int lgo, gxo, gyo;  // output pass: tile columns 4 << lgo, gxo x gyo blocks
  int G;
  int* status;
};

__device__ __forceinline__ Blk red_blk(const CoopGeom& g) {
  return Blk{blockIdx.x % g.gx, blockIdx.x / g.gx, g.gx, g.gy};
}
__device__ __forceinline__ Blk out_blk(const CoopGeom& g) {
  return Blk{blockIdx.x % g.gxo, blockIdx.x / g.gxo, g.gxo, g.gyo};
}

// The forward as one launch: range pass -> tau_0, exponents, codes and code sums -> the
// deviation sums -> channel constants and output tables, spread over the blocks by channel
// -> output.  (Each block building the tables of its own output columns instead -- 8192
// entries, a division each -- took 8.7 us of a 29 us call on [12544, 256].)
__global__ void __launch_bounds__(kL1Threads, 3) l1bn_fwd_coop_kernel(const L1bnArgs a, const CoopGeom g) {
  extern __shared__ __align__(16) unsigned char dyn[];   // reductions, then the output table
  __shared__ uint8_t sexp[kL1MaxCols];
  __shared__ int mean[kL1MaxCols];
  __shared__ uint32_t red[32];
  __shared__ float cs[1], cm[1], csq[1], cgq[1], cbq[1];
  RedSmem<2>& sm2 = *reinterpret_cast<RedSmem<2>*>(dyn);
  RedSmem<1>& sm1 = *reinterpret_cast<RedSmem<1>*>(dyn);
  unsigned* ctr = a.sync;
  unsigned* slots = a.sync + 64;
  const unsigned nb = gridDim.x;
  const bool red_on = blockIdx.x < static_cast<unsigned>(g.gx * g.gy);
  const Blk b = red_blk(g);
  // 1. range pass; the sums the later phases add into start at zero
  zero_sums(a.st, 3 * kSpread * a.C);   // kStS1, kStS, kStZ
  if (red_on) range_pass(a, g.lg, b, slots, sm1, g.status);
  if (!grid_barrier(ctr, nb, g.status)) return;
  // 2. tau_0, exponents; codes and their sums
  if (red_on) {
    const float tau = coop_group(a, g.lg, b, g.G, slots, a.ch + kChXRange * a.C, a.scal + kScXTau,
                                 a.xe, sexp, red, g.status);
    fwd_quant_pass(a, g.lg, b, tau, sexp, b.x * (int64_t(4) << g.lg), sm1);
  }
  if (!grid_barrier(ctr, 2 * nb, g.status)) return;
  // 3. deviation sums
  if (red_on) fwd_dev_pass<true>(a, g.lg, b, sm2, mean);
  if (!grid_barrier(ctr, 3 * nb, g.status)) return;
  // 4. per-tensor maxima of sigma, |gamma|, |beta| over all channels
  const float Rf = __ll2float_rn(a.R);
  const float scale = __ldcg(a.scal + kScXScale);
  uint32_t ms = 0, mg = 0, mb = 0;
  for (int64_t c = threadIdx.x; c < a.C; c += kL1Threads) {
    ms = max(ms, __float_as_uint(fwd_chan_of(a, c, scale, Rf).sig) & 0x7FFFFFFFu);
    mg = max(mg, __float_as_uint(a.gamma[c]) & 0x7FFFFFFFu);
    mb = max(mb, __float_as_uint(a.beta[c]) & 0x7FFFFFFFu);
  }
  const float smax = __uint_as_float(block_max(ms, red));
  const float gmax = __uint_as_float(block_max(mg, red));
  const float bmax = __uint_as_float(block_max(mb, red));
  // 5. block b: the constants of channels b, b + gridDim.x, ... into the state (the
  // backward reads them) and their output tables (one entry per thread)
  for (int64_t c = blockIdx.x; c < a.C; c += gridDim.x) {
    if (threadIdx.x == 0) {
      const int64_t C = a.C;
      const FwdChan f = fwd_chan_of(a, c, scale, Rf);
      cs[0] = f.s;
      cm[0] = f.m;
      csq[0] = quant8(f.sig, smax);
      cgq[0] = quant8(a.gamma[c], gmax);
      cbq[0] = quant8(a.beta[c], bmax);
      a.ch[kChS * C + c] = f.s;
      a.ch[kChM * C + c] = f.m;
      a.ch[kChSig * C + c] = f.sig;
      a.ch[kChSq * C + c] = csq[0];
      a.ch[kChGq * C + c] = cgq[0];
      a.ch[kChBq * C + c] = cbq[0];
    }
    __syncthreads();
    a.lut[c * kLutStride + threadIdx.x] =
        l1bn_out_of(static_cast<int>(threadIdx.x) - 127, cs[0], cm[0], csq[0], cgq[0], cbq[0]);
    __syncthreads();
  }
  if (!grid_barrier(ctr, 4 * nb, g.status)) return;
  // 6. output: the block's columns' tables into shared memory, then y
  if (blockIdx.x >= static_cast<unsigned>(g.gxo * g.gyo)) return;
  const Blk bo = out_blk(g);
  const int64_t cbase = bo.x * (int64_t(4) << g.lgo);
  const int ncol = static_cast<int>(min(int64_t(4) << g.lgo, a.C - cbase));
  float* lut = reinterpret_cast<float*>(dyn);
  for (int i = threadIdx.x; i < ncol * kLutStride; i += kL1Threads) lut[i] = __ldcg(a.lut + cbase * kLutStride + i);
  __syncthreads();
  fwd_out_pass<true>(a, g.lgo, bo, lut);
}

// The backward as one launch: range pass of dy -> its tau_0, exponents, codes and the sums
// of p and p (q - m) -> channel constants (dgamma, dbeta) and the input gradient.
__global__ void __launch_bounds__(kL1Threads, 2) l1bn_bwd_coop_kernel(const L1bnArgs a, const CoopGeom g) {
  __shared__ RedSmem<2> sm2;
  __shared__ uint8_t sexp[kL1MaxCols];
  __shared__ uint32_t red[32];
  __shared__ BwdChan sc[4 << kCoopOutLg];
  RedSmem<1>& sm1 = *reinterpret_cast<RedSmem<1>*>(&sm2);
  unsigned* ctr = a.sync;
  unsigned* slots = a.sync + 64;
  const unsigned nb = gridDim.x;
  const bool red_on = blockIdx.x < static_cast<unsigned>(g.gx * g.gy);
  const Blk b = red_blk(g);
  zero_sums(a.st + kStP * kSpread * a.C, 2 * kSpread * a.C);   // kStP, kStD
  if (red_on) range_pass(a, g.lg, b, slots, sm1, g.status);
  if (!grid_barrier(ctr, nb, g.status)) return;
  if (red_on) {
    const float tau = coop_group(a, g.lg, b, g.G, slots, a.ch + kChGRange * a.C, a.scal + kScGTau,
                                 a.ge, sexp, red, g.status);
    bwd_quant_pass(a, g.lg, b, tau, sexp, b.x * (int64_t(4) << g.lg), sm2);
  }
  if (!grid_barrier(ctr, 2 * nb, g.status)) return;
  if (blockIdx.x >= static_cast<unsigned>(g.gxo * g.gyo)) return;
  const Blk bo = out_blk(g);
  const float gscale = __ldcg(a.scal + kScGScale);
  const float Rf = __ll2float_rn(a.R);
  const int64_t c = bo.x * (int64_t(4) << g.lgo) + threadIdx.x;
  if (threadIdx.x < (4 << g.lgo) && c < a.C) {
    sc[threadIdx.x] = bwd_chan_of(a, c, gscale, Rf);
    if (bo.y == 0) put_bwd_chan(a, c, sc[threadIdx.x]);   // dgamma, dbeta, the state: once per column
  }
  __syncthreads();
  bwd_out_pass<false>(a, g.lgo, bo, sc);
}

// Self-test of the grid barrier's expiry path: block 0 never arrives, so every block's
// bounded wait runs out (about 1 s), records SQ_DEV_TIMEOUT and returns.
__global__ void __launch_bounds__(kL1Threads) l1bn_selftest_barrier_kernel(unsigned* ctr, int* status) {
  grid_barrier(ctr, gridDim.x, status, blockIdx.x != 0);
}

// ------------------------------------------------------------------ host side
static int l1bn_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
  return n;
}

// the argument block over a checked state buffer
static L1bnArgs l1bn_args(int64_t R, int64_t C, int bits, void* state) {
  const L1bnLayout L = l1bn_layout(R, C);
  char* b = static_cast<char*>(state);
  L1bnArgs a;
  memset(&a, 0, sizeof(a));
  a.R = R;
  a.C = C;
  a.Q = q_of_bits(bits);
  a.xq = reinterpret_cast<int8_t*>(b + L.xq);
  a.gq = reinterpret_cast<int8_t*>(b + L.gq);
  a.st = reinterpret_cast<long long*>(b + L.stats);
  a.ch = reinterpret_cast<float*>(b + L.chan);
  a.lut = reinterpret_cast<float*>(b + L.lut);
  a.xe = reinterpret_cast<uint8_t*>(b + L.exps);
  a.ge = a.xe + C;
  a.scal = reinterpret_cast<float*>(b + L.scal);
  a.sync = reinterpret_cast<unsigned*>(b + L.sync);
  return a;
}

static int l1bn_check(const char* nm, int64_t R, int64_t C, int64_t ld_in, int64_t ld_out,
                      int bits, int G, const void* in, const void* out, void* state,
                      size_t state_bytes, int32_t* dev_status) {
  if (!bits_ok(bits) || !groups_ok(G))
    return fail(SQ_EINVAL, "%s: bits must be in [2, 8] and n_groups in [1, 8]", nm);
  if (R < 0 || C < 0) return fail(SQ_EINVAL, "%s: negative size", nm);
  if (C > 0 && R == 0) return fail(SQ_EINVAL, "%s: a channel needs at least one element", nm);
  if (C == 0) return SQ_OK;
  if (R > (int64_t(1) << 40) || C >= (int64_t(1) << 31) || R * C > (int64_t(1) << 40))
    return fail(SQ_EUNSUPPORTED, "%s: tensor too large", nm);
  if (in == nullptr || out == nullptr || state == nullptr || dev_status == nullptr)
    return fail(SQ_EINVAL, "%s: NULL argument", nm);
  if (ld_in < C || ld_out < C) return fail(SQ_EINVAL, "%s: leading dimension < channels", nm);
  if (!aligned16(state)) return fail(SQ_EALIGN, "%s: state must be 16-byte aligned", nm);
  if (state_bytes < l1bn_layout(R, C).total)
    return fail(SQ_EINVAL, "%s: state smaller than shiftquant_l1bn_state_bytes()", nm);
  return SQ_OK;
}

// The tile of a tensor with C channels: TC = 4 << lg columns, the channel count rounded up
// to a power of two (at least 4, at most 128).
static int tile_lg(int64_t C) {
  int lg = 0;
  while (lg < 5 && (int64_t(4) << lg) < C) ++lg;
  return lg;
}

// A reduction launch: the column tiles by about three blocks per SM (one resident wave),
// each block taking every gridDim.y-th tile of `rows_per_tile` rows.
static dim3 reduction_grid(int64_t R, int64_t C, int lg, int rows_per_tile, int sms) {
  const int64_t gx = (C + (int64_t(4) << lg) - 1) / (int64_t(4) << lg);
  const int64_t tiles = (R + rows_per_tile - 1) / rows_per_tile;
  int64_t gy = (3 * static_cast<int64_t>(sms) + gx - 1) / gx;   // one wave at three blocks per SM
  if (gy > tiles) gy = tiles;
  if (gy > 65535) gy = 65535;
  if (gy < 1) gy = 1;
  return dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
}

// An elementwise launch: the column tiles by about three blocks per SM, each block walking
// its rows (at most one step of kL1PassesCodes rows per thread when there are few rows).
static dim3 elementwise_grid(int64_t R, int64_t C, int lg, int sms) {
  const int64_t gx = (C + (int64_t(4) << lg) - 1) / (int64_t(4) << lg);
  const int64_t rows_per_step = kL1PassesCodes * (int64_t(kL1Threads) >> lg);
  int64_t gy = (R + rows_per_step - 1) / rows_per_step;
  const int64_t want = (3 * static_cast<int64_t>(sms) + gx - 1) / gx;
  if (gy > want) gy = want;
  if (gy > 65535) gy = 65535;
  return dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy < 1 ? 1 : gy));
}

// The output pass's tile: at most 32 columns, so that the table it keeps in shared memory
// (32 KB) leaves room for three blocks per SM.
constexpr int kL1OutMaxLg = 3;

// Launch a kernel behind the previous one of the stream with programmatic stream
// serialization (it waits for that kernel before reading its results).
template <typename... Params, typename... Args>
static cudaError_t launch_behind(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                                 cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

static int launched(const char* what) {
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, what);
}

// The single-launch form's block count on the current device (one resident wave: every
// block of a cooperative launch must be resident at once), 0 where it cannot run.
template <bool FWD>
static int coop_blocks() {
  static int cached[64][2];   // [device][fwd]: blocks + 1, 0 = not asked yet
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int& slot = cached[dev][FWD ? 1 : 0];
  if (slot == 0) {
    int coop = 0, sms = 0, per_sm = 0;
    cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const size_t dyn = FWD ? size_t(4 << kCoopOutLg) * kLutStride * sizeof(float) : 0;
    if (coop && sms > 0 &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &per_sm, FWD ? l1bn_fwd_coop_kernel : l1bn_bwd_coop_kernel, kL1Threads, dyn) == cudaSuccess)
      slot = 1 + (per_sm > 3 ? 3 : per_sm) * sms;
    else
      slot = 1;
    cudaGetLastError();
  }
  return slot - 1;
}

// The single-launch form of a call: the counter and range slots zeroed, then one
// cooperative launch of `blocks` blocks.
template <bool FWD>
static int launch_coop(const L1bnArgs& a, int G, int blocks, int32_t* dev_status, cudaStream_t s) {
  cudaError_t err = cudaMemsetAsync(a.sync, 0, 256 + kSpread * static_cast<size_t>(a.C) * sizeof(unsigned), s);
  if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync (l1bn sync)");
  CoopGeom g;
  g.lg = tile_lg(a.C);
  g.gx = static_cast<int>((a.C + (int64_t(4) << g.lg) - 1) / (int64_t(4) << g.lg));
  g.gy = blocks / g.gx;
  g.lgo = g.lg < kCoopOutLg ? g.lg : kCoopOutLg;
  g.gxo = static_cast<int>((a.C + (int64_t(4) << g.lgo) - 1) / (int64_t(4) << g.lgo));
  g.gyo = blocks / g.gxo;
  g.G = G;
  g.status = dev_status;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(static_cast<unsigned>(blocks));
  cfg.blockDim = dim3(kL1Threads);
  cfg.dynamicSmemBytes = FWD ? size_t(4 << g.lgo) * kLutStride * sizeof(float) : 0;
  if (FWD && cfg.dynamicSmemBytes < sizeof(RedSmem<2>)) cfg.dynamicSmemBytes = sizeof(RedSmem<2>);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = FWD ? cudaLaunchKernelEx(&cfg, l1bn_fwd_coop_kernel, a, g)
            : cudaLaunchKernelEx(&cfg, l1bn_bwd_coop_kernel, a, g);
  if (err == cudaSuccess) err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, FWD ? "l1bn_fwd_coop_kernel launch" : "l1bn_bwd_coop_kernel launch");
}

// the single-launch form serves this call: few enough channels for every block to form
// the per-tensor maxima over all of them, and a device that runs cooperative launches
// with at least one block per output column tile
template <bool FWD>
static int coop_use(int64_t C) {
  if (C > kCoopMaxChannels) return 0;
  const int blocks = coop_blocks<FWD>();
  const int lgo = tile_lg(C) < kCoopOutLg ? tile_lg(C) : kCoopOutLg;
  const int64_t gxo = (C + (int64_t(4) << lgo) - 1) / (int64_t(4) << lgo);
  return blocks >= gxo && blocks >= 8 ? blocks : 0;
}

}  // namespace sq

using namespace sq;

extern "C" size_t shiftquant_l1bn_state_bytes(int64_t rows, int64_t channels) {
  if (rows < 0 || channels < 0) return 0;
  return l1bn_layout(rows, channels).total;
}

extern "C" sq_status shiftquant_selftest_grid_barrier_timeout(void* scratch, int32_t* dev_status,
                                                              void* stream) {
  fail(SQ_OK, "");
  if (scratch == nullptr || dev_status == nullptr || !aligned16(scratch))
    return fail(SQ_EINVAL, "selftest_grid_barrier_timeout: scratch (16-byte aligned) and dev_status are required");
  cudaStream_t s = as_stream(stream);
  cudaError_t err = cudaMemsetAsync(scratch, 0, 256, s);
  if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(8);
  cfg.blockDim = dim3(kL1Threads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, l1bn_selftest_barrier_kernel, static_cast<unsigned*>(scratch),
                           reinterpret_cast<int*>(dev_status));
  if (err == cudaSuccess) err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "l1bn_selftest_barrier_kernel launch");
}

extern "C" int shiftquant_l1bn_kernel_launches(int64_t channels, int backward) {
  if (channels < 0 || channels >= (int64_t(1) << 31)) return -1;
  if (channels == 0) return 0;
  if (l1bn_sms() <= 0) return -1;
  if (backward ? coop_use<false>(channels) : coop_use<true>(channels)) return 1;
  // zeroing, the range pass (zeroing, range, grouping), then the passes
  return backward ? 1 + 3 + 3 : 1 + 3 + 5;
}

extern "C" sq_status shiftquant_l1bn_forward(const float* x, int64_t rows, int64_t channels,
                                             int64_t ld_x, const float* gamma, const float* beta,
                                             int bits, int n_groups, float* y, int64_t ld_y,
                                             void* state, size_t state_bytes,
                                             int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  int st = l1bn_check("l1bn_forward", rows, channels, ld_x, ld_y, bits, n_groups, x, y, state,
                      state_bytes, dev_status);
  if (st != SQ_OK || channels == 0) return st;
  if (gamma == nullptr || beta == nullptr) return fail(SQ_EINVAL, "l1bn_forward: gamma and beta are required");
  const int sms = l1bn_sms();
  if (sms <= 0) return fail(SQ_ECUDA, "l1bn_forward: no current CUDA device");
  cudaStream_t s = as_stream(stream);
  L1bnArgs a = l1bn_args(rows, channels, bits, state);
  a.in = x;
  a.ld_in = ld_x;
  a.out = y;
  a.ld_out = ld_y;
  a.gamma = gamma;
  a.beta = beta;
  a.vec_in = (ld_x % 4 == 0) && aligned16(x);
  a.vec_out = (ld_y % 4 == 0) && aligned16(y);
  if (const int blocks = coop_use<true>(channels)) return launch_coop<true>(a, n_groups, blocks, dev_status, s);
  // the channel sums start at zero (a kernel, not a memset, so that the launches after the
  // range pass stay a chain of kernels, each launched behind the one before)
  const int64_t nz = 3 * kSpread * channels;
  l1bn_zero_kernel<<<static_cast<unsigned>((nz + 255) / 256 < 1024 ? (nz + 255) / 256 : 1024), 256, 0, s>>>(a.st, nz);
  if ((st = launched("l1bn_zero_kernel launch")) != SQ_OK) return st;
  // range pass and grouping of x (the library's own), into the state
  st = shiftquant_calibrate(x, rows, channels, ld_x, SQ_GRAN_SHIFT, n_groups,
                            a.ch + kChXRange * channels, a.scal + kScXTau, a.xe, dev_status, stream);
  if (st != SQ_OK) return st;
  cudaError_t err;
  const int lg = tile_lg(channels);
  const int rpp = kL1Threads >> lg;
  err = launch_behind(l1bn_fwd_quant_kernel, reduction_grid(rows, channels, lg, kL1PassesF32 * rpp, sms),
                      dim3(kL1Threads), 0, s, a, lg);
  if (err != cudaSuccess) return cuda_fail(err, "l1bn_fwd_quant_kernel launch");
  err = launch_behind(l1bn_fwd_dev_kernel, reduction_grid(rows, channels, lg, kL1PassesCodes * rpp, sms),
                      dim3(kL1Threads), 0, s, a, lg);
  if (err != cudaSuccess) return cuda_fail(err, "l1bn_fwd_dev_kernel launch");
  if ((err = launch_behind(l1bn_fwd_chan_kernel, dim3(1), dim3(1024), 0, s, a)) != cudaSuccess)
    return cuda_fail(err, "l1bn_fwd_chan_kernel launch");
  if ((err = launch_behind(l1bn_fwd_lut_kernel, dim3(static_cast<unsigned>(channels)), dim3(kLutStride),
                           0, s, a)) != cudaSuccess)
    return cuda_fail(err, "l1bn_fwd_lut_kernel launch");
  const int lgo = lg < kL1OutMaxLg ? lg : kL1OutMaxLg;
  const size_t lut_bytes = (size_t(4) << lgo) * kLutStride * sizeof(float);
  err = launch_behind(l1bn_fwd_out_kernel, elementwise_grid(rows, channels, lgo, sms), dim3(kL1Threads),
                      lut_bytes, s, a, lgo);
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "l1bn_fwd_out_kernel launch");
}

extern "C" sq_status shiftquant_l1bn_backward(const float* dy, int64_t rows, int64_t channels,
                                              int64_t ld_dy, int bits, int n_groups,
                                              uint64_t seed, void* state, size_t state_bytes,
                                              float* dx, int64_t ld_dx, float* dgamma,
                                              float* dbeta, int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  int st = l1bn_check("l1bn_backward", rows, channels, ld_dy, ld_dx, bits, n_groups, dy, dx,
                      state, state_bytes, dev_status);
  if (st != SQ_OK || channels == 0) return st;
  if (dgamma == nullptr || dbeta == nullptr)
    return fail(SQ_EINVAL, "l1bn_backward: dgamma and dbeta are required");
  const int sms = l1bn_sms();
  if (sms <= 0) return fail(SQ_ECUDA, "l1bn_backward: no current CUDA device");
  cudaStream_t s = as_stream(stream);
  L1bnArgs a = l1bn_args(rows, channels, bits, state);
  a.in = dy;
  a.ld_in = ld_dy;
  a.out = dx;
  a.ld_out = ld_dx;
  a.seed = seed;
  a.dgamma = dgamma;
  a.dbeta = dbeta;
  a.vec_in = (ld_dy % 4 == 0) && aligned16(dy);
  a.vec_out = (ld_dx % 4 == 0) && aligned16(dx);
  if (const int blocks = coop_use<false>(channels)) return launch_coop<false>(a, n_groups, blocks, dev_status, s);
  const int64_t nz = 2 * kSpread * channels;
  l1bn_zero_kernel<<<static_cast<unsigned>((nz + 255) / 256 < 1024 ? (nz + 255) / 256 : 1024), 256, 0, s>>>(
      a.st + kStP * kSpread * channels, nz);
  if ((st = launched("l1bn_zero_kernel launch")) != SQ_OK) return st;
  st = shiftquant_calibrate(dy, rows, channels, ld_dy, SQ_GRAN_SHIFT, n_groups,
                            a.ch + kChGRange * channels, a.scal + kScGTau, a.ge, dev_status, stream);
  if (st != SQ_OK) return st;
  cudaError_t err;
  const int lg = tile_lg(channels);
  const int rpp = kL1Threads >> lg;
  err = launch_behind(l1bn_bwd_quant_kernel, reduction_grid(rows, channels, lg, kL1PassesF32 * rpp, sms),
                      dim3(kL1Threads), 0, s, a, lg);
  if (err != cudaSuccess) return cuda_fail(err, "l1bn_bwd_quant_kernel launch");
  const unsigned cb = static_cast<unsigned>((channels + 255) / 256);
  if ((err = launch_behind(l1bn_bwd_chan_kernel, dim3(cb), dim3(256), 0, s, a)) != cudaSuccess)
    return cuda_fail(err, "l1bn_bwd_chan_kernel launch");
  err = launch_behind(l1bn_bwd_out_kernel, elementwise_grid(rows, channels, lg, sms), dim3(kL1Threads), 0,
                      s, a, lg);
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "l1bn_bwd_out_kernel launch");
}
