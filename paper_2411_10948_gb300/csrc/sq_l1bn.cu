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
// Kernels, all streaming HBM passes: a column-reduction pass that quantizes and sums
// (128 columns x a slab of rows per block, four columns per thread with 16-byte loads,
// sums combined across warps in shared memory and across blocks with 64-bit atomics), a
// second reduction over the 1-byte codes for the deviation sums, a one-block pass for the
// per-channel values, and an elementwise output pass (four outputs per thread).
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
// per-channel int64 sums of the state
enum { kStS1, kStS, kStZ, kStP, kStD, kNumStats };
// scalars of the state
enum { kScXTau, kScXScale, kScGTau, kScGScale, kNumScal };

struct L1bnLayout {
  size_t xq, gq, stats, chan, exps, scal, total;
};

static L1bnLayout l1bn_layout(int64_t R, int64_t C) {
  auto up = [](size_t n) { return (n + 255) & ~size_t(255); };
  const size_t n = static_cast<size_t>(R) * static_cast<size_t>(C);
  L1bnLayout L;
  size_t o = 0;
  L.xq = o;    o += up(n);
  L.gq = o;    o += up(n);
  L.stats = o; o += up(kNumStats * static_cast<size_t>(C) * sizeof(long long));
  L.chan = o;  o += up(kNumChan * static_cast<size_t>(C) * sizeof(float));
  L.exps = o;  o += up(2 * static_cast<size_t>(C));
  L.scal = o;  o += 256;
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
  long long* st;  // [kNumStats][C]
  float* ch;      // [kNumChan][C]
  uint8_t* xe;
  uint8_t* ge;
  float* scal;
  const float* gamma;
  const float* beta;
  float* dgamma;
  float* dbeta;
  int vec_in, vec_out;  // 16-byte rows: four elements per load / store
};

constexpr int kL1Cols = 128;  // columns of a reduction block (four per lane)
constexpr int kL1Threads = 256;

__device__ __forceinline__ long long rne_div(long long a, long long b) {
  long long q = a / b, r = a % b;
  if (r < 0) {
    q -= 1;
    r += b;
  }
  if (2 * r > b || (2 * r == b && (q & 1))) q += 1;
  return q;
}

// four consecutive elements of row r from column c (zeros past C)
__device__ __forceinline__ void load4(const float* row, int64_t c, int64_t C, bool vec, float v[4]) {
  if (vec && c + 3 < C) {
    const float4 t = __ldg(reinterpret_cast<const float4*>(row + c));
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) v[j] = c + j < C ? __ldg(row + c + j) : 0.0f;
  }
}

__device__ __forceinline__ void load_codes4(const int8_t* codes, int64_t off, int64_t c, int64_t C,
                                            int q[4]) {
  if ((C & 3) == 0) {
    const char4 t = *reinterpret_cast<const char4*>(codes + off);
    q[0] = t.x; q[1] = t.y; q[2] = t.z; q[3] = t.w;
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) q[j] = c + j < C ? codes[off + j] : 0;
  }
}

__device__ __forceinline__ void store_codes4(int8_t* codes, int64_t off, int64_t c, int64_t C,
                                             const int q[4]) {
  if ((C & 3) == 0) {
    *reinterpret_cast<char4*>(codes + off) = make_char4(static_cast<signed char>(q[0]),
                                                        static_cast<signed char>(q[1]),
                                                        static_cast<signed char>(q[2]),
                                                        static_cast<signed char>(q[3]));
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (c + j < C) codes[off + j] = static_cast<int8_t>(q[j]);
  }
}

// Per-block column sums -> global: each thread holds sums of its four columns over its
// rows; the eight warps combine in shared memory and 128 threads add one column each.
template <typename T>
__device__ __forceinline__ void add_columns(const T (&acc)[4], long long* dst, int64_t c0,
                                            int64_t C, T* red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int j = 0; j < 4; ++j) red[w * kL1Cols + lane * 4 + j] = acc[j];
  __syncthreads();
  if (threadIdx.x < kL1Cols) {
    long long s = 0;
#pragma unroll
    for (int k = 0; k < kL1Threads / 32; ++k) s += static_cast<long long>(red[k * kL1Cols + threadIdx.x]);
    const int64_t c = c0 + threadIdx.x;
    if (c < C && s != 0)
      atomicAdd(reinterpret_cast<unsigned long long*>(dst + c), static_cast<unsigned long long>(s));
  }
}

// rows of this block: [r0, r1); the block's warps take rows r0 + w, r0 + w + 8, ...
__device__ __forceinline__ void block_rows(int64_t R, int64_t* r0, int64_t* r1) {
  const int64_t per = (R + gridDim.y - 1) / gridDim.y;
  *r0 = static_cast<int64_t>(blockIdx.y) * per;
  *r1 = min(R, *r0 + per);
}

// Forward pass 1: x -> int8 ShiftQuant codes (round to nearest), sum of codes per channel.
__global__ void __launch_bounds__(kL1Threads) l1bn_fwd_quant_kernel(const L1bnArgs a) {
  __shared__ int red[kL1Threads / 32 * kL1Cols];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kL1Cols;
  const int64_t c = c0 + lane * 4;
  const float tau = a.scal[kScXTau];
  const float Qf = static_cast<float>(a.Q);
  const float invS = __fdiv_rn(Qf, tau);
  const bool zero = !(tau > 0.0f) || !isfinite(tau) || !isfinite(invS);
  int e[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) e[j] = c + j < a.C ? a.xe[c + j] : 0;
  int acc[4] = {0, 0, 0, 0};
  int64_t r0, r1;
  block_rows(a.R, &r0, &r1);
  if (c < a.C) {
#pragma unroll 4
    for (int64_t r = r0 + w; r < r1; r += kL1Threads / 32) {
      float v[4];
      load4(a.in + r * a.ld_in, c, a.C, a.vec_in, v);
      int q[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        q[j] = c + j < a.C ? shift_code(v[j], e[j], invS, zero, Qf, false, 0, 0) : 0;
        acc[j] += q[j];
      }
      store_codes4(a.xq, r * a.C + c, c, a.C, q);
    }
  }
  add_columns(acc, a.st + kStS1 * a.C, c0, a.C, red);
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0)
    a.scal[kScXScale] = zero ? 0.0f : __fdiv_rn(tau, Qf);
}

// Forward pass 2: over the codes, sum |q - m| and sum sign(q - m) per channel, with
// m = round-half-even(sum q / R).
__global__ void __launch_bounds__(kL1Threads) l1bn_fwd_dev_kernel(const L1bnArgs a) {
  __shared__ int red[kL1Threads / 32 * kL1Cols];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kL1Cols;
  const int64_t c = c0 + lane * 4;
  int m[4];
#pragma unroll
  for (int j = 0; j < 4; ++j)
    m[j] = c + j < a.C ? static_cast<int>(rne_div(a.st[kStS1 * a.C + c + j], a.R)) : 0;
  int sabs[4] = {0, 0, 0, 0}, ssgn[4] = {0, 0, 0, 0};
  int64_t r0, r1;
  block_rows(a.R, &r0, &r1);
  if (c < a.C) {
#pragma unroll 4
    for (int64_t r = r0 + w; r < r1; r += kL1Threads / 32) {
      int q[4];
      load_codes4(a.xq, r * a.C + c, c, a.C, q);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (c + j >= a.C) continue;
        const int d = q[j] - m[j];
        sabs[j] += d < 0 ? -d : d;
        ssgn[j] += (d > 0) - (d < 0);
      }
    }
  }
  add_columns(sabs, a.st + kStS * a.C, c0, a.C, red);
  __syncthreads();
  add_columns(ssgn, a.st + kStZ * a.C, c0, a.C, red);
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

// Forward pass 3 (one block): s_c, m_c, sigma_c, then sigma^q, gamma^q, beta^q.
__global__ void __launch_bounds__(1024) l1bn_fwd_chan_kernel(const L1bnArgs a) {
  __shared__ uint32_t red[32];
  const float Rf = __ll2float_rn(a.R);
  const float scale = a.scal[kScXScale];
  float* ch = a.ch;
  const int64_t C = a.C;
  uint32_t ms = 0, mg = 0, mb = 0;
  for (int64_t c = threadIdx.x; c < C; c += blockDim.x) {
    const float s = __fmul_rn(scale, pow2f(-static_cast<int>(a.xe[c])));
    const long long m = rne_div(a.st[kStS1 * C + c], a.R);
    const float sig = __fmul_rn(__fdiv_rn(__ll2float_rn(a.st[kStS * C + c]), Rf), s);
    ch[kChS * C + c] = s;
    ch[kChM * C + c] = static_cast<float>(m);
    ch[kChSig * C + c] = sig;
    ms = max(ms, __float_as_uint(sig) & 0x7FFFFFFFu);
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

// Forward pass 4: y = gamma^q ((x^q - mu^q) / sigma^q) + beta^q, four outputs per thread.
__global__ void __launch_bounds__(256) l1bn_fwd_out_kernel(const L1bnArgs a) {
  const int64_t nq = (a.C + 3) / 4;
  const int64_t quads = a.R * nq;
  const float* ch = a.ch;
  const int64_t C = a.C;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < quads;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / nq;
    const int64_t c = (i - r * nq) * 4;
    int q[4];
    load_codes4(a.xq, r * C + c, c, C, q);
    float y[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      y[j] = 0.0f;
      if (c + j >= C) continue;
      const float s = ch[kChS * C + c + j], sq = ch[kChSq * C + c + j];
      const float xq = __fmul_rn(static_cast<float>(q[j]), s);
      const float mq = __fmul_rn(ch[kChM * C + c + j], s);
      const float xhat = sq > 0.0f ? __fdiv_rn(__fsub_rn(xq, mq), sq) : 0.0f;
      y[j] = __fadd_rn(__fmul_rn(ch[kChGq * C + c + j], xhat), ch[kChBq * C + c + j]);
    }
    float* dst = a.out + r * a.ld_out + c;
    if (a.vec_out && c + 3 < C) {
      *reinterpret_cast<float4*>(dst) = make_float4(y[0], y[1], y[2], y[3]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (c + j < C) dst[j] = y[j];
    }
  }
}

// Backward pass 1: dy -> int8 ShiftQuant codes p (stochastic rounding of element r C + c),
// sums of p and of p (q - m) per channel.
__global__ void __launch_bounds__(kL1Threads) l1bn_bwd_quant_kernel(const L1bnArgs a) {
  __shared__ long long red[kL1Threads / 32 * kL1Cols];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kL1Cols;
  const int64_t c = c0 + lane * 4;
  const float tau = a.scal[kScGTau];
  const float Qf = static_cast<float>(a.Q);
  const float invS = __fdiv_rn(Qf, tau);
  const bool zero = !(tau > 0.0f) || !isfinite(tau) || !isfinite(invS);
  int e[4], m[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    e[j] = c + j < a.C ? a.ge[c + j] : 0;
    m[j] = c + j < a.C ? static_cast<int>(a.ch[kChM * a.C + c + j]) : 0;
  }
  long long sp[4] = {0, 0, 0, 0}, spd[4] = {0, 0, 0, 0};
  int64_t r0, r1;
  block_rows(a.R, &r0, &r1);
  if (c < a.C) {
#pragma unroll 4
    for (int64_t r = r0 + w; r < r1; r += kL1Threads / 32) {
      float v[4];
      load4(a.in + r * a.ld_in, c, a.C, a.vec_in, v);
      int qx[4];
      load_codes4(a.xq, r * a.C + c, c, a.C, qx);
      int p[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        p[j] = c + j < a.C ? shift_code(v[j], e[j], invS, zero, Qf, true, a.seed,
                                        static_cast<uint64_t>(r * a.C + c + j))
                           : 0;
        sp[j] += p[j];
        spd[j] += static_cast<long long>(p[j]) * (qx[j] - m[j]);
      }
      store_codes4(a.gq, r * a.C + c, c, a.C, p);
    }
  }
  add_columns(sp, a.st + kStP * a.C, c0, a.C, red);
  __syncthreads();
  add_columns(spd, a.st + kStD * a.C, c0, a.C, red);
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0)
    a.scal[kScGScale] = zero ? 0.0f : __fdiv_rn(tau, Qf);
}

// Backward pass 2: the per-channel constants of the input gradient, dgamma and dbeta.
__global__ void __launch_bounds__(256) l1bn_bwd_chan_kernel(const L1bnArgs a) {
  const float Rf = __ll2float_rn(a.R);
  const float gscale = a.scal[kScGScale];
  const int64_t C = a.C;
  float* ch = a.ch;
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; c < C;
       c += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float t = __fmul_rn(gscale, pow2f(-static_cast<int>(a.ge[c])));
    const float sq = ch[kChSq * C + c], s = ch[kChS * C + c];
    const float P = __ll2float_rn(a.st[kStP * C + c]);
    const float u = sq > 0.0f ? __fdiv_rn(ch[kChGq * C + c], sq) : 0.0f;
    const float mg = __fdiv_rn(__fmul_rn(P, t), Rf);
    const float dg =
        sq > 0.0f ? __fdiv_rn(__fmul_rn(__fmul_rn(__ll2float_rn(a.st[kStD * C + c]), t), s), sq) : 0.0f;
    ch[kChT * C + c] = t;
    ch[kChU * C + c] = u;
    ch[kChMg * C + c] = mg;
    ch[kChMgx * C + c] = __fdiv_rn(dg, Rf);
    ch[kChZs * C + c] = __fdiv_rn(__ll2float_rn(a.st[kStZ * C + c]), Rf);
    a.dgamma[c] = dg;
    a.dbeta[c] = __fmul_rn(P, t);
  }
}

// Backward pass 3: dx = u ((g - mean g) - mean(g xhat) (sign(q - m) - mean sign)).
__global__ void __launch_bounds__(256) l1bn_bwd_out_kernel(const L1bnArgs a) {
  const int64_t nq = (a.C + 3) / 4;
  const int64_t quads = a.R * nq;
  const float* ch = a.ch;
  const int64_t C = a.C;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < quads;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / nq;
    const int64_t c = (i - r * nq) * 4;
    int q[4], p[4];
    load_codes4(a.xq, r * C + c, c, C, q);
    load_codes4(a.gq, r * C + c, c, C, p);
    float dx[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      dx[j] = 0.0f;
      if (c + j >= C) continue;
      const int d = q[j] - static_cast<int>(ch[kChM * C + c + j]);
      const float g = __fmul_rn(static_cast<float>(p[j]), ch[kChT * C + c + j]);
      const float sg = static_cast<float>((d > 0) - (d < 0));
      const float inner = __fsub_rn(__fsub_rn(g, ch[kChMg * C + c + j]),
                                    __fmul_rn(ch[kChMgx * C + c + j], __fsub_rn(sg, ch[kChZs * C + c + j])));
      dx[j] = __fmul_rn(ch[kChU * C + c + j], inner);
    }
    float* dst = a.out + r * a.ld_out + c;
    if (a.vec_out && c + 3 < C) {
      *reinterpret_cast<float4*>(dst) = make_float4(dx[0], dx[1], dx[2], dx[3]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (c + j < C) dst[j] = dx[j];
    }
  }
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
  a.xe = reinterpret_cast<uint8_t*>(b + L.exps);
  a.ge = a.xe + C;
  a.scal = reinterpret_cast<float*>(b + L.scal);
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
  if (R > (int64_t(1) << 40) || C > (int64_t(1) << 31) || R * C > (int64_t(1) << 40))
    return fail(SQ_EUNSUPPORTED, "%s: tensor too large", nm);
  if (in == nullptr || out == nullptr || state == nullptr || dev_status == nullptr)
    return fail(SQ_EINVAL, "%s: NULL argument", nm);
  if (ld_in < C || ld_out < C) return fail(SQ_EINVAL, "%s: leading dimension < channels", nm);
  if (!aligned16(state)) return fail(SQ_EALIGN, "%s: state must be 16-byte aligned", nm);
  if (state_bytes < l1bn_layout(R, C).total)
    return fail(SQ_EINVAL, "%s: state smaller than shiftquant_l1bn_state_bytes()", nm);
  return SQ_OK;
}

static dim3 reduction_grid(int64_t R, int64_t C, int sms) {
  const int64_t gx = (C + kL1Cols - 1) / kL1Cols;
  int64_t gy = (4 * static_cast<int64_t>(sms) + gx - 1) / gx;  // about four blocks per SM
  const int64_t max_gy = (R + 7) / 8;                          // at least eight rows a block
  if (gy > max_gy) gy = max_gy;
  if (gy > 65535) gy = 65535;
  if (gy < 1) gy = 1;
  return dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy));
}

static unsigned elementwise_blocks(int64_t R, int64_t C, int sms) {
  const int64_t quads = R * ((C + 3) / 4);
  int64_t b = (quads + 255) / 256;
  if (b > static_cast<int64_t>(sms) * 16) b = static_cast<int64_t>(sms) * 16;
  return static_cast<unsigned>(b < 1 ? 1 : b);
}

static int launched(const char* what) {
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, what);
}

}  // namespace sq

using namespace sq;

extern "C" size_t shiftquant_l1bn_state_bytes(int64_t rows, int64_t channels) {
  if (rows < 0 || channels < 0) return 0;
  return l1bn_layout(rows, channels).total;
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
  // range pass and grouping of x (the library's own), into the state
  st = shiftquant_calibrate(x, rows, channels, ld_x, SQ_GRAN_SHIFT, n_groups,
                            a.ch + kChXRange * channels, a.scal + kScXTau, a.xe, dev_status, stream);
  if (st != SQ_OK) return st;
  cudaError_t err = cudaMemsetAsync(a.st, 0, 3 * static_cast<size_t>(channels) * sizeof(long long), s);
  if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  const dim3 rg = reduction_grid(rows, channels, sms);
  l1bn_fwd_quant_kernel<<<rg, kL1Threads, 0, s>>>(a);
  if ((st = launched("l1bn_fwd_quant_kernel launch")) != SQ_OK) return st;
  l1bn_fwd_dev_kernel<<<rg, kL1Threads, 0, s>>>(a);
  if ((st = launched("l1bn_fwd_dev_kernel launch")) != SQ_OK) return st;
  l1bn_fwd_chan_kernel<<<1, 1024, 0, s>>>(a);
  if ((st = launched("l1bn_fwd_chan_kernel launch")) != SQ_OK) return st;
  l1bn_fwd_out_kernel<<<elementwise_blocks(rows, channels, sms), 256, 0, s>>>(a);
  return launched("l1bn_fwd_out_kernel launch");
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
  st = shiftquant_calibrate(dy, rows, channels, ld_dy, SQ_GRAN_SHIFT, n_groups,
                            a.ch + kChGRange * channels, a.scal + kScGTau, a.ge, dev_status, stream);
  if (st != SQ_OK) return st;
  cudaError_t err = cudaMemsetAsync(a.st + kStP * channels, 0,
                                    2 * static_cast<size_t>(channels) * sizeof(long long), s);
  if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  const dim3 rg = reduction_grid(rows, channels, sms);
  l1bn_bwd_quant_kernel<<<rg, kL1Threads, 0, s>>>(a);
  if ((st = launched("l1bn_bwd_quant_kernel launch")) != SQ_OK) return st;
  const unsigned cb = static_cast<unsigned>((channels + 255) / 256);
  l1bn_bwd_chan_kernel<<<cb, 256, 0, s>>>(a);
  if ((st = launched("l1bn_bwd_chan_kernel launch")) != SQ_OK) return st;
  l1bn_bwd_out_kernel<<<elementwise_blocks(rows, channels, sms), 256, 0, s>>>(a);
  return launched("l1bn_bwd_out_kernel launch");
}
