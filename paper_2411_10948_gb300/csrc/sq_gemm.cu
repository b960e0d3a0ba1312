// ShiftMM on sm_103a: the quantized training GEMMs of ShiftQuant (Eq. 4, App. D) on the
// 5th-generation tensor cores.
//
// sm_103a has no integer MMA, so the integer contraction runs on the float MMA with
// exact operands: a code q (|q| <= 127) times a power of two is exact in BF16, and in
// FP8 E4M3 when |q| <= 15 and the shifted value stays <= 448.  Products are exact in
// FP32, and a sum of integers is exact in FP32 while every partial sum stays within
// 2^24.  The K loop is therefore cut into chunks whose worst case
// (max|product| x chunk length) is at most 2^24; each chunk accumulates in its own TMEM
// buffer and the epilogue warps convert it to int32 and add it to a register
// accumulator (two TMEM buffers ping-pong so the tensor core never waits on them).
// The ShiftMM shift 2^(G-1-e_k) of inner index k is already inside the weight codes
// (the quantizer folds it in), so the tensor core applies it to every product before
// accumulation at no cost, exactly as ShiftMM prescribes (Sec. 3.2).
//
// One CTA per SM, persistent over output tiles of 128 x 256:
//   warp 0      TMA producer: A and B tiles (128-byte rows, 128-byte swizzle) into a
//               4-stage shared-memory ring
//   warp 1      TMEM allocation and the MMA issuer (one thread)
//   warps 4-11  epilogue: tcgen05.ld, int32 accumulation across chunks, dequantizing
//               multiply, stores (or int32 reductions into a split-K workspace)
// Every wait is bounded (about 1 s); on expiry the kernel records SQ_DEV_TIMEOUT,
// drains its own copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "sq_device.cuh"
#include "sq_host.h"

namespace sq {

constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kBKBytes = 128;                 // one 128-byte swizzle row of K per stage
constexpr int kStages = 3;
constexpr int kABytes = kBM * kBKBytes;       // 16 KB
constexpr int kBBytes = kBN * kBKBytes;       // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kThreads = 384;
constexpr int kEpiWarp0 = 4;
constexpr int kNumEpiWarps = 8;
constexpr uint32_t kTmemCols = 2 * kBN;       // two FP32 accumulator buffers
constexpr int64_t kExactSum = int64_t(1) << 24;  // every partial sum of a chunk stays within this
// shared memory: the operand ring, two 32 x 32 output boxes per epilogue warp (staging for
// TMA stores, double-buffered), two per-tile column-factor tables, then the barriers
constexpr int kOutBox = 32;
constexpr int kOutStageBytes = kOutBox * kOutBox * 4;
constexpr int kOutOffset = kStages * kStageBytes;
constexpr int kFacOffset = kOutOffset + kNumEpiWarps * 2 * kOutStageBytes;
constexpr int kBarOffset = kFacOffset + 2 * kBN * 4;
constexpr int kNumBars = 2 * kStages + 2 + 2 + 2 + 1;   // full, empty, tfull, tempty, fac, drain
constexpr size_t kSmemBytes = kBarOffset + kNumBars * 8 + 16;
static_assert(kSmemBytes <= 232448, "shared memory beyond the 227 KB per-CTA limit");
static_assert(kOutOffset % 1024 == 0 && kOutStageBytes % 1024 == 0, "swizzle atoms need 1 KB");

struct GemmParams {
  int M, N, K;
  int m_tiles, n_tiles, splits, kb_total, kb_per_split, chunk_kb;
  int mode;  // 0: per-column scale (forward, loss propagation); 1: row/column shifts (wgrad)
  int G;
  int use_tma_y;  // outputs leave through TMA stores (else plain stores)
  const float* a_scale;
  const float* b_scale;
  const uint8_t* row_exp;
  const uint8_t* col_exp;
  float* y;
  int64_t ldy;
  long long* acc;
  int64_t ld_acc;
  int* ws;  // split-K int32 partial sums [M, N], or null
  int* status;
};

__device__ __forceinline__ float pow2_neg(int k) { return __int_as_float((127 - k) << 23); }

// the dequantized value and the canonical integer of one output element
__device__ __forceinline__ void epilogue_value(const GemmParams& p, int64_t row, int64_t col,
                                               int32_t t, float a_fac, float* out_y,
                                               long long* out_t) {
  if (p.mode == 0) {
    // Y = T * (s_A 2^-(G-1) * s_B[col]);  T already carries the shifts
    const float f = __fmul_rn(a_fac, __ldg(p.b_scale + col));
    *out_y = __fmul_rn(__int2float_rn(t), f);
    *out_t = t;
  } else {
    // dW = T_raw * 2^-(eX + eY) * (s_X s_dY);  canonical T = T_raw << (2(G-1) - eX - eY)
    const int er = __ldg(p.row_exp + row), ec = __ldg(p.col_exp + col);
    *out_y = __fmul_rn(__fmul_rn(__int2float_rn(t), pow2_neg(er + ec)), a_fac);
    *out_t = static_cast<long long>(t) << (2 * (p.G - 1) - er - ec);
  }
}

__device__ __forceinline__ float epilogue_a_factor(const GemmParams& p) {
  return p.mode == 0 ? __fmul_rn(__ldg(p.a_scale), pow2_neg(p.G - 1))
                     : __fmul_rn(__ldg(p.a_scale), __ldg(p.b_scale));
}

// value of box element (rr, cc) in a staging buffer written with 128-byte swizzle
__device__ __forceinline__ uint32_t staged(uint32_t buf, int rr, int cc) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];"
               : "=r"(v)
               : "r"(buf + rr * 128 + ((((cc >> 2) ^ (rr & 7))) << 4) + (cc & 3) * 4));
  return v;
}

// plain stores of a staged fp32 box (lane = column, one row per step: coalesced)
__device__ __noinline__ void write_y_box(float* y, int64_t ldy, int64_t M, int64_t N, uint32_t buf,
                                         int64_t row0, int64_t col0, int lane) {
  const int64_t col = col0 + lane;
  for (int rr = 0; rr < 32; ++rr) {
    const int64_t row = row0 + rr;
    if (row < M && col < N) y[row * ldy + col] = __uint_as_float(staged(buf, rr, lane));
  }
}

// the canonical integers T of a staged int32 box as int64 (exactness-check output);
// row_exp / col_exp are null for the forward and loss-propagation GEMMs
__device__ __noinline__ void write_acc_box(long long* acc, int64_t ld_acc, int64_t M, int64_t N,
                                           const uint8_t* row_exp, const uint8_t* col_exp, int G,
                                           uint32_t buf, int64_t row0, int64_t col0, int lane) {
  const int64_t col = col0 + lane;
  if (col >= N) return;
  const int ec = col_exp ? __ldg(col_exp + col) : 0;
  for (int rr = 0; rr < 32; ++rr) {
    const int64_t row = row0 + rr;
    if (row >= M) break;
    const long long t = static_cast<int32_t>(staged(buf, rr, lane));
    acc[row * ld_acc + col] = row_exp ? t << (2 * (G - 1) - __ldg(row_exp + row) - ec) : t;
  }
}

// One 32 x 32 output box of an epilogue warp: lane = row, vals = the lane's 32 columns as
// exact integers (FP32 patterns when `as_float`, else int32).  Stages the box in shared
// memory and hands it to TMA (store of the dequantized fp32 values, or int32 reduce-add
// into the split-K workspace); writes the exactness-check integers when asked.
__device__ __forceinline__ void emit_box(const GemmParams& p, const CUtensorMap* tma_y,
                                         const CUtensorMap* tma_ws, const uint32_t (&vals)[32],
                                         bool as_float, const float* f, float rfac, uint32_t buf,
                                         int64_t row0, int64_t col0, int lane, bool via_tma) {
  if (lane == 0) bulk_wait_read<1>();
  __syncwarp();
  if (p.acc != nullptr && p.ws == nullptr) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      uint32_t o[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t a = vals[k * 4 + e];
        o[e] = as_float ? static_cast<uint32_t>(__float2int_rn(__uint_as_float(a))) : a;
      }
      st_shared_v4(buf + lane * 128 + ((k ^ (lane & 7)) << 4), o[0], o[1], o[2], o[3]);
    }
    __syncwarp();
    write_acc_box(p.acc, p.ld_acc, p.M, p.N, p.mode == 1 ? p.row_exp : nullptr,
                  p.mode == 1 ? p.col_exp : nullptr, p.G, buf, row0, col0, lane);
    __syncwarp();
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t a = vals[k * 4 + e];
      if (p.ws != nullptr) {
        o[e] = as_float ? static_cast<uint32_t>(__float2int_rn(__uint_as_float(a))) : a;
      } else {
        const float val = as_float ? __uint_as_float(a) : __int2float_rn(static_cast<int32_t>(a));
        o[e] = __float_as_uint(__fmul_rn(__fmul_rn(val, rfac), f[k * 4 + e]));
      }
    }
    st_shared_v4(buf + lane * 128 + ((k ^ (lane & 7)) << 4), o[0], o[1], o[2], o[3]);
  }
  if (via_tma) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (p.ws != nullptr)
        tma_reduce_add_2d(tma_ws, buf, static_cast<int32_t>(col0), static_cast<int32_t>(row0));
      else
        tma_store_2d(tma_y, buf, static_cast<int32_t>(col0), static_cast<int32_t>(row0));
      bulk_commit();
    }
  } else {
    __syncwarp();
    write_y_box(p.y, p.ldy, p.M, p.N, buf, row0, col0, lane);  // outputs TMA cannot address
    __syncwarp();
  }
}

struct Unit {
  int mb, nb, kb0, kb1;
};

// Work unit u -> (tile, K split).  Tiles go in groups of kGroupM row tiles: inside a group
// the row tile changes fastest, then the column tile.  The CTAs running at one time then
// cover a compact block of the output, so the A rows of a group stay in L2 while every
// column tile of B passes by, and neither operand is streamed from HBM more than once
// per group.
constexpr int kGroupM = 16;

__device__ __forceinline__ Unit decode_unit(const GemmParams& p, int u) {
  const int tiles = p.m_tiles * p.n_tiles;
  const int split = u / tiles;
  const int t = u - split * tiles;
  const int per_group = kGroupM * p.n_tiles;
  const int g = t / per_group;
  const int gm = min(kGroupM, p.m_tiles - g * kGroupM);  // row tiles in this group
  const int in = t - g * per_group;
  Unit r;
  r.mb = g * kGroupM + in % gm;
  r.nb = in / gm;
  r.kb0 = split * p.kb_per_split;
  r.kb1 = min(p.kb_total, r.kb0 + p.kb_per_split);
  return r;
}

// kMulti: the K loop of a tile spans several exact chunks, whose int32 sums the epilogue
// keeps in registers; otherwise every output streams from TMEM once.
template <int kF8, bool kMulti>
__global__ void __launch_bounds__(kThreads, 1)
    shiftmm_kernel(const __grid_constant__ CUtensorMap tma_a,
                   const __grid_constant__ CUtensorMap tma_b,
                   const __grid_constant__ CUtensorMap tma_y,
                   const __grid_constant__ CUtensorMap tma_ws, const GemmParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {  // the swizzled layouts need 1 KB alignment
    if (threadIdx.x == 0) atomicOr(p.status, kDevInternal);
    return;
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kBarOffset);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* tfull = bars + 2 * kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* facbar = tempty + 2;
  uint64_t* drain = facbar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kNumEpiWarps);
      mbar_init(&facbar[b], kNumEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tma_a);
    tma_prefetch_desc(&tma_b);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int units = p.m_tiles * p.n_tiles * p.splits;
  constexpr int kBKElems = kF8 ? kBKBytes : kBKBytes / 2;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    int s = 0;
    uint32_t ph = 0;
    long long issued = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      for (int kb = w.kb0; kb < w.kb1; ++kb) {
        if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t sa = smem_u32(smem + s * kStageBytes);
        mbar_arrive_expect_tx(&full[s], kStageBytes);
        tma_load_2d(sa, &tma_a, smem_u32(&full[s]), kb * kBKElems, w.mb * kBM);
        tma_load_2d(sa + kABytes, &tma_b, smem_u32(&full[s]), kb * kBKElems, w.nb * kBN);
        ++issued;
        if (++s == kStages) {
          s = 0;
          ph ^= 1u;
        }
      }
    }
    if (!ok) {
      atomicOr(p.status, kDevTimeout);
      *abort_flag = 1;
    }
    // every issued copy must have landed before the CTA may exit
    for (long long i = issued > kStages ? issued - kStages : 0; i < issued; ++i)
      mbar_wait(&full[i % kStages], static_cast<uint32_t>((i / kStages) & 1), nullptr);
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------- MMA issuer
    constexpr uint32_t idesc = make_idesc(kF8 ? 0u : 1u, kBM, kBN);
    int s = 0;
    uint32_t ph = 0;
    uint32_t c = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      const Unit w = decode_unit(p, u);
      for (int kc = w.kb0; kc < w.kb1 && ok; kc += p.chunk_kb) {
        const int kce = min(w.kb1, kc + p.chunk_kb);
        const uint32_t b = c & 1u, tph = (c >> 1) & 1u;
        if (!mbar_wait(&tempty[b], tph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + b * kBN;
        for (int kb = kc; kb < kce; ++kb) {
          if (!mbar_wait(&full[s], ph, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(smem + s * kStageBytes);
          const uint32_t b0 = a0 + kABytes;
#pragma unroll
          for (int k = 0; k < kBKBytes / 32; ++k) {
            const uint64_t ad = make_sdesc_k_sw128(a0 + k * 32);
            const uint64_t bd = make_sdesc_k_sw128(b0 + k * 32);
            const uint32_t accumulate = (kb > kc || k > 0) ? 1u : 0u;
            if (kF8)
              tc_mma_f8(d, ad, bd, idesc, accumulate);
            else
              tc_mma_f16(d, ad, bd, idesc, accumulate);
          }
          tc_commit(smem_u32(&empty[s]));  // frees the stage once these MMAs are done
          if (++s == kStages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(&tfull[b]));  // chunk complete in TMEM buffer b
        ++c;
      }
    }
    if (!ok) {
      atomicOr(p.status, kDevTimeout);
      *abort_flag = 1;
    }
    tc_commit(smem_u32(drain));
    mbar_wait(drain, 0, nullptr);
  } else if (warp >= kEpiWarp0) {
    // --------------------------------------------------------------- epilogue
    const int q = warp & 3;                       // TMEM lanes 32q .. 32q+31 (output rows)
    const int h = (warp - kEpiWarp0) >> 2;        // column half of the 256-wide tile
    const int et = threadIdx.x - kEpiWarp0 * 32;  // 0 .. 255: one tile column each
    const uint32_t stage_out0 =
        smem_u32(smem + kOutOffset + (warp - kEpiWarp0) * 2 * kOutStageBytes);
    uint32_t nbox = 0;  // boxes this warp has handed to TMA: selects the staging buffer
    float* fac_tab = reinterpret_cast<float*>(smem + kFacOffset);
    const float a_fac = epilogue_a_factor(p);
    const bool via_tma = p.ws != nullptr || p.use_tma_y;
    uint32_t c = 0;
    bool ok = true;
    int it = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++it) {
      const Unit w = decode_unit(p, u);
      const int nch = (w.kb1 - w.kb0 + p.chunk_kb - 1) / p.chunk_kb;
      const int64_t m0 = static_cast<int64_t>(w.mb) * kBM;
      const int64_t n0 = static_cast<int64_t>(w.nb) * kBN;
      // the dequantizing factor of each of the tile's 256 columns, computed once per tile
      // while the tensor core works: s_A 2^-(G-1) s_B[n] (forward, loss propagation) or
      // s_X s_dY 2^-eY_n (weight gradient; the row's 2^-eX_m is applied separately)
      float* fac = fac_tab + (it & 1) * kBN;
      {
        const int64_t col = n0 + et;
        float f = 0.0f;
        if (col < p.N)
          f = p.mode == 0 ? __fmul_rn(a_fac, __ldg(p.b_scale + col))
                          : __fmul_rn(a_fac, pow2_neg(__ldg(p.col_exp + col)));
        fac[et] = f;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&facbar[it & 1]);

      const int64_t row0 = m0 + q * 32;
      const int64_t row = row0 + lane;
      const bool row_ok = row < p.M;
      const float rfac = pow2_neg((p.mode == 1 && row_ok) ? __ldg(p.row_exp + row) : 0);
      if constexpr (!kMulti) {
        // one exact chunk: each TMEM value is already the integer T (as FP32)
        const uint32_t b = c & 1u, tph = (c >> 1) & 1u;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(&tfull[b], tph, abort_flag)) ||
            !__all_sync(0xFFFFFFFFu, mbar_wait(&facbar[it & 1], (it >> 1) & 1, abort_flag))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + b * kBN + h * 128;
#pragma unroll 1
        for (int s = 0; s < 4; ++s) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(taddr + s * 32, v);
          tmem_ld_wait();
          if (s == 3) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[b]);  // TMEM buffer b may take the next tile
          }
          const int64_t col0 = n0 + h * 128 + s * 32;
          if (row0 >= p.M || col0 >= p.N) continue;  // warp-uniform: nothing of this box exists
          const uint32_t buf = stage_out0 + (nbox & 1u) * kOutStageBytes;
          ++nbox;
          emit_box(p, &tma_y, &tma_ws, v, true, fac + h * 128 + s * 32, rfac, buf, row0, col0,
                   lane, via_tma);
        }
        ++c;
      } else {
        uint32_t acc[128];  // int32 sums of the chunks
        for (int ch = 0; ch < nch; ++ch) {
          const uint32_t b = c & 1u, tph = (c >> 1) & 1u;
          if (!__all_sync(0xFFFFFFFFu, mbar_wait(&tfull[b], tph, abort_flag))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + b * kBN + h * 128;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            uint32_t v[16];
            tmem_ld_32x32b_x16(taddr + j * 16, v);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              // the FP32 value is an integer of magnitude <= 2^24: the conversion is exact
              const int32_t t = __float2int_rn(__uint_as_float(v[i]));
              acc[j * 16 + i] =
                  static_cast<uint32_t>(ch == 0 ? t : static_cast<int32_t>(acc[j * 16 + i]) + t);
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[b]);  // TMEM buffer b may take the next chunk
          ++c;
        }
        if (!ok) break;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait(&facbar[it & 1], (it >> 1) & 1, abort_flag))) {
          ok = false;
          break;
        }
#pragma unroll
        for (int s = 0; s < 4; ++s) {
          const int64_t col0 = n0 + h * 128 + s * 32;
          if (row0 >= p.M || col0 >= p.N) continue;
          uint32_t v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = acc[s * 32 + i];
          const uint32_t buf = stage_out0 + (nbox & 1u) * kOutStageBytes;
          ++nbox;
          emit_box(p, &tma_y, &tma_ws, v, false, fac + h * 128 + s * 32, rfac, buf, row0, col0,
                   lane, via_tma);
        }
      }
    }
    if (!ok) {
      atomicOr(p.status, kDevTimeout);
      *abort_flag = 1;
    }
    if (lane == 0) bulk_wait_read<0>();  // no store still reads shared memory at exit
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// split-K: turn the summed int32 partials into the outputs
__global__ void __launch_bounds__(256) splitk_finalize_kernel(const GemmParams p) {
  const float a_fac = epilogue_a_factor(p);
  const int64_t total = static_cast<int64_t>(p.M) * p.N;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = i / p.N, col = i - row * p.N;
    float o;
    long long t;
    epilogue_value(p, row, col, p.ws[i], a_fac, &o, &t);
    p.y[row * p.ldy + col] = o;
    if (p.acc) p.acc[row * p.ld_acc + col] = t;
  }
}

// ----------------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// K-major operand [rows, K] with leading dimension ld (elements): boxes of
// (128 bytes of K) x box_rows, 128-byte swizzle, zero fill outside the tensor
static int make_operand_map(CUtensorMap* map, const void* base, int64_t rows, int64_t K,
                            int64_t ld, int elem_bytes, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  const CUtensorMapDataType dt =
      elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(ld * elem_bytes)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBKBytes / elem_bytes),
                       static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estride[2] = {1, 1};
  const CUresult r = fn(map, dt, 2, const_cast<void*>(base), gdim, gstride, box, estride,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return SQ_OK;
}

// fp32 output or int32 split-K workspace [rows, cols] (leading dimension ld elements):
// 32 x 32 boxes with 128-byte swizzle, matching the epilogue's staging layout
static int make_output_map(CUtensorMap* map, void* base, int64_t rows, int64_t cols, int64_t ld,
                           CUtensorMapDataType dt) {
  auto fn = encode_fn();
  if (!fn) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(ld * 4)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kOutBox), static_cast<cuuint32_t>(kOutBox)};
  cuuint32_t estride[2] = {1, 1};
  const CUresult r = fn(map, dt, 2, base, gdim, gstride, box, estride,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled (output) failed (%d)", static_cast<int>(r));
  return SQ_OK;
}

static int device_sms(int* dev_out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
  if (dev_out) *dev_out = dev;
  return n;
}

struct Plan {
  int m_tiles, n_tiles, kb_total, chunk_kb, splits, kb_per_split;
  int elem_bytes;
};

// max |product| of one inner index: q_A q_B 2^(G-1) with the shift folded into B
// (forward, loss propagation) or q_A q_B with the shifts applied after the sum (wgrad)
static int64_t max_product(int which, int bits, int G) {
  const int64_t Q = q_of_bits(bits);
  return (which == 2) ? Q * Q : (Q * Q) << (G - 1);
}

// the exactness limits, checked before anything touches the device
static int check_exact_range(int which, int64_t K, int bits, int G) {
  const int64_t P = max_product(which, bits, G);
  if (P * K > INT32_MAX)
    return fail(SQ_EUNSUPPORTED,
                "inner dimension %lld exceeds the exact int32 range for bits=%d, n_groups=%d "
                "(max |T| = %lld * K)",
                static_cast<long long>(K), bits, G, static_cast<long long>(P));
  const int bk = kBKBytes / code_bytes(code_type(bits, G));
  if (kExactSum / P < bk)
    return fail(SQ_EUNSUPPORTED,
                "bits=%d with n_groups=%d: one %d-wide K block can exceed the exact FP32 sum range",
                bits, G, bk);
  return SQ_OK;
}

static int make_plan(int which, int64_t M, int64_t N, int64_t K, int bits, int G, int sms,
                     bool allow_split, Plan* pl) {
  const int st = check_exact_range(which, K, bits, G);
  if (st != SQ_OK) return st;
  const int64_t P = max_product(which, bits, G);
  pl->elem_bytes = code_bytes(code_type(bits, G));
  const int bk = kBKBytes / pl->elem_bytes;
  pl->chunk_kb = static_cast<int>((kExactSum / P) / bk);
  if (pl->chunk_kb > (1 << 20)) pl->chunk_kb = 1 << 20;
  pl->m_tiles = static_cast<int>((M + kBM - 1) / kBM);
  pl->n_tiles = static_cast<int>((N + kBN - 1) / kBN);
  pl->kb_total = static_cast<int>((K + bk - 1) / bk);
  const int64_t tiles = static_cast<int64_t>(pl->m_tiles) * pl->n_tiles;
  int splits = 1;
  if (allow_split && tiles < sms && pl->kb_total >= 4) {
    splits = static_cast<int>(sms / tiles);
    if (splits > pl->kb_total / 2) splits = pl->kb_total / 2;
    if (splits < 1) splits = 1;
  }
  pl->kb_per_split = (pl->kb_total + splits - 1) / splits;
  pl->splits = (pl->kb_total + pl->kb_per_split - 1) / pl->kb_per_split;
  return SQ_OK;
}

template <int kF8, bool kMulti>
static int configure_kernel(int dev) {
  static bool done[64] = {};
  if (dev >= 0 && dev < 64 && done[dev]) return SQ_OK;
  const cudaError_t err = cudaFuncSetAttribute(shiftmm_kernel<kF8, kMulti>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(kSmemBytes));
  if (err != cudaSuccess) return cuda_fail(err, "cudaFuncSetAttribute");
  if (dev >= 0 && dev < 64) done[dev] = true;
  return SQ_OK;
}

static int run_gemm(int which, const void* a_codes, int64_t lda, const void* b_codes, int64_t ldb,
                    int64_t M, int64_t N, int64_t K, int bits, int G, const float* a_scale,
                    const float* b_scale, const uint8_t* row_exp, const uint8_t* col_exp,
                    float* y, int64_t ldy, int64_t* acc_out, int64_t ld_acc, void* workspace,
                    size_t workspace_bytes, int32_t* dev_status, void* stream) {
  static const char* names[3] = {"gemm_fwd", "gemm_dgrad", "gemm_wgrad"};
  const char* nm = names[which];
  if (!bits_ok(bits) || !groups_ok(G))
    return fail(SQ_EINVAL, "%s: bits must be in [2, 8] and n_groups in [1, 8]", nm);
  if (M < 0 || N < 0 || K < 0) return fail(SQ_EINVAL, "%s: negative size", nm);
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX)
    return fail(SQ_EUNSUPPORTED, "%s: dimensions beyond 2^31", nm);
  if (dev_status == nullptr) return fail(SQ_EINVAL, "%s: dev_status is required", nm);
  if (M == 0 || N == 0) return SQ_OK;
  if (y == nullptr || ldy < N) return fail(SQ_EINVAL, "%s: output is NULL or its ld < N", nm);
  if (acc_out != nullptr && ld_acc < N) return fail(SQ_EINVAL, "%s: ld_acc < N", nm);
  if (a_scale == nullptr || b_scale == nullptr) return fail(SQ_EINVAL, "%s: scales are required", nm);
  if (which == 2 && (row_exp == nullptr || col_exp == nullptr))
    return fail(SQ_EINVAL, "%s: exponents are required", nm);
  cudaStream_t s = as_stream(stream);
  if (K == 0) {
    // an empty inner sum: T = 0 everywhere
    cudaError_t err = cudaMemset2DAsync(y, ldy * sizeof(float), 0, N * sizeof(float), M, s);
    if (err == cudaSuccess && acc_out)
      err = cudaMemset2DAsync(acc_out, ld_acc * sizeof(int64_t), 0, N * sizeof(int64_t), M, s);
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemset2DAsync");
  }
  if (a_codes == nullptr || b_codes == nullptr) return fail(SQ_EINVAL, "%s: codes are NULL", nm);
  if (lda < K || ldb < K) return fail(SQ_EINVAL, "%s: operand ld smaller than K", nm);
  const int eb = code_bytes(code_type(bits, G));
  if (!aligned16(a_codes) || !aligned16(b_codes) || (lda * eb) % 16 != 0 || (ldb * eb) % 16 != 0)
    return fail(SQ_EALIGN, "%s: operand pointers must be 16-byte aligned and ld * %d bytes a "
                "multiple of 16", nm, eb);
  int st = check_exact_range(which, K, bits, G);
  if (st != SQ_OK) return st;
  int dev = 0;
  const int sms = device_sms(&dev);
  if (sms <= 0) return fail(SQ_ECUDA, "%s: no current CUDA device", nm);
  Plan pl;
  st = make_plan(which, M, N, K, bits, G, sms, true, &pl);
  if (st != SQ_OK) return st;
  if (pl.splits > 1) {
    // split-K partials are added by TMA into a [M, N] int32 workspace with N-element rows,
    // whose rows must stay 16-byte aligned
    const size_t need = static_cast<size_t>(M) * N * sizeof(int);
    if (workspace == nullptr || workspace_bytes < need || !aligned16(workspace) || N % 4 != 0) {
      st = make_plan(which, M, N, K, bits, G, sms, false, &pl);
      if (st != SQ_OK) return st;
    }
  }
  CUtensorMap ma, mb;
  st = make_operand_map(&ma, a_codes, M, K, lda, eb, kBM);
  if (st != SQ_OK) return st;
  st = make_operand_map(&mb, b_codes, N, K, ldb, eb, kBN);
  if (st != SQ_OK) return st;

  GemmParams p;
  p.M = static_cast<int>(M);
  p.N = static_cast<int>(N);
  p.K = static_cast<int>(K);
  p.m_tiles = pl.m_tiles;
  p.n_tiles = pl.n_tiles;
  p.splits = pl.splits;
  p.kb_total = pl.kb_total;
  p.kb_per_split = pl.kb_per_split;
  p.chunk_kb = pl.chunk_kb;
  p.mode = which == 2 ? 1 : 0;
  p.G = G;
  p.use_tma_y = (ldy % 4 == 0) && aligned16(y);
  p.a_scale = a_scale;
  p.b_scale = b_scale;
  p.row_exp = row_exp;
  p.col_exp = col_exp;
  p.y = y;
  p.ldy = ldy;
  p.acc = reinterpret_cast<long long*>(acc_out);
  p.ld_acc = ld_acc;
  p.ws = pl.splits > 1 ? static_cast<int*>(workspace) : nullptr;
  p.status = dev_status;

  CUtensorMap my, mw;
  memset(&my, 0, sizeof(my));
  memset(&mw, 0, sizeof(mw));
  if (p.ws) {
    st = make_output_map(&mw, p.ws, M, N, N, CU_TENSOR_MAP_DATA_TYPE_INT32);
    if (st != SQ_OK) return st;
  } else if (p.use_tma_y) {
    st = make_output_map(&my, y, M, N, ldy, CU_TENSOR_MAP_DATA_TYPE_FLOAT32);
    if (st != SQ_OK) return st;
  }
  cudaError_t err;
  if (p.ws) {
    err = cudaMemsetAsync(p.ws, 0, static_cast<size_t>(M) * N * sizeof(int), s);
    if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  }
  const int units = pl.m_tiles * pl.n_tiles * pl.splits;
  const int grid = units < sms ? units : sms;
  const bool multi = pl.kb_per_split > pl.chunk_kb;  // some unit spans several exact chunks
  if (eb == 1) {
    if (multi) {
      if ((st = configure_kernel<1, true>(dev)) != SQ_OK) return st;
      shiftmm_kernel<1, true><<<grid, kThreads, kSmemBytes, s>>>(ma, mb, my, mw, p);
    } else {
      if ((st = configure_kernel<1, false>(dev)) != SQ_OK) return st;
      shiftmm_kernel<1, false><<<grid, kThreads, kSmemBytes, s>>>(ma, mb, my, mw, p);
    }
  } else {
    if (multi) {
      if ((st = configure_kernel<0, true>(dev)) != SQ_OK) return st;
      shiftmm_kernel<0, true><<<grid, kThreads, kSmemBytes, s>>>(ma, mb, my, mw, p);
    } else {
      if ((st = configure_kernel<0, false>(dev)) != SQ_OK) return st;
      shiftmm_kernel<0, false><<<grid, kThreads, kSmemBytes, s>>>(ma, mb, my, mw, p);
    }
  }
  err = cudaGetLastError();
  if (err != cudaSuccess) return cuda_fail(err, "shiftmm_kernel launch");
  if (p.ws) {
    const int64_t total = static_cast<int64_t>(M) * N;
    int64_t blocks = (total + 255) / 256;
    if (blocks > static_cast<int64_t>(sms) * 16) blocks = static_cast<int64_t>(sms) * 16;
    splitk_finalize_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(p);
    err = cudaGetLastError();
    if (err != cudaSuccess) return cuda_fail(err, "splitk_finalize_kernel launch");
  }
  return SQ_OK;
}


// ----------------------------------------------- allocation-free weight gradient
// Scratch for callers that cannot allocate device memory themselves: a fixed array in
// the library's own device image, present on every GPU that loads the library until the
// process exits.  It serves as the split-K int32 workspace of
// shiftquant_gemm_wgrad_static().
constexpr size_t kStaticScratchBytes = size_t(4) << 20;  // 4 MiB: Ci * Co <= 1048576
static __device__ __align__(256) int g_wgrad_scratch[kStaticScratchBytes / sizeof(int)];

// Device address of g_wgrad_scratch on the current device.  In host code the array's
// name only stands in for the symbol, so the address is looked up once per device with
// that device current and cached.
static int static_scratch_address(void** out) {
  static void* addr[64] = {};
  static std::mutex mu;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return cuda_fail(err, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(SQ_EUNSUPPORTED, "device index %d beyond 63", dev);
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_wgrad_scratch);
    if (err != cudaSuccess) return cuda_fail(err, "cudaGetSymbolAddress");
    addr[dev] = p;
  }
  *out = addr[dev];
  return SQ_OK;
}
}  // namespace sq

using namespace sq;

extern "C" sq_status shiftquant_gemm_fwd(const void* a_codes, int64_t lda, const float* a_scale,
                                         const void* b_codes, int64_t ldb, const float* b_scale,
                                         int64_t M, int64_t N, int64_t K, int bits, int n_groups,
                                         float* y, int64_t ldy, int64_t* acc_out, int64_t ld_acc,
                                         void* workspace, size_t workspace_bytes,
                                         int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  return run_gemm(0, a_codes, lda, b_codes, ldb, M, N, K, bits, n_groups, a_scale, b_scale,
                  nullptr, nullptr, y, ldy, acc_out, ld_acc, workspace, workspace_bytes,
                  dev_status, stream);
}

extern "C" sq_status shiftquant_gemm_dgrad(const void* a_codes, int64_t lda, const float* a_scale,
                                           const void* b_codes, int64_t ldb, const float* b_scale,
                                           int64_t M, int64_t N_out, int64_t K_in, int bits,
                                           int n_groups, float* dx, int64_t ldx, int64_t* acc_out,
                                           int64_t ld_acc, void* workspace, size_t workspace_bytes,
                                           int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  return run_gemm(1, a_codes, lda, b_codes, ldb, M, N_out, K_in, bits, n_groups, a_scale, b_scale,
                  nullptr, nullptr, dx, ldx, acc_out, ld_acc, workspace, workspace_bytes,
                  dev_status, stream);
}

extern "C" sq_status shiftquant_gemm_wgrad(const void* xt_codes, int64_t ldx, const float* x_scale,
                                           const uint8_t* x_exp, const void* gt_codes, int64_t ldg,
                                           const float* g_scale, const uint8_t* g_exp, int64_t Ci,
                                           int64_t Co, int64_t T, int bits, int n_groups, float* dw,
                                           int64_t ld_dw, int64_t* acc_out, int64_t ld_acc,
                                           void* workspace, size_t workspace_bytes,
                                           int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  return run_gemm(2, xt_codes, ldx, gt_codes, ldg, Ci, Co, T, bits, n_groups, x_scale, g_scale,
                  x_exp, g_exp, dw, ld_dw, acc_out, ld_acc, workspace, workspace_bytes, dev_status,
                  stream);
}

extern "C" size_t shiftquant_gemm_workspace_bytes(int which, int64_t M, int64_t N, int64_t K,
                                                  int bits, int n_groups) {
  if (which < 0 || which > 2 || !bits_ok(bits) || !groups_ok(n_groups) || M <= 0 || N <= 0 ||
      K <= 0)
    return 0;
  const int sms = device_sms(nullptr);
  if (sms <= 0) return 0;
  Plan pl;
  if (make_plan(which, M, N, K, bits, n_groups, sms, true, &pl) != SQ_OK) return 0;
  return pl.splits > 1 ? static_cast<size_t>(M) * N * sizeof(int) : 0;
}

extern "C" sq_status shiftquant_gemm_wgrad_static(
    const void* xt_codes, int64_t ldx, const float* x_scale, const uint8_t* x_exp,
    const void* gt_codes, int64_t ldg, const float* g_scale, const uint8_t* g_exp, int64_t Ci,
    int64_t Co, int64_t T, int bits, int n_groups, float* dw, int64_t ld_dw, int64_t* acc_out,
    int64_t ld_acc, int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  if (Ci > 0 && Co > 0 &&
      static_cast<uint64_t>(Ci) * static_cast<uint64_t>(Co) * sizeof(int) > kStaticScratchBytes)
    return fail(SQ_EUNSUPPORTED,
                "gemm_wgrad_static: Ci * Co = %lld exceeds the %zu int32 entries of the "
                "library's static scratch; use shiftquant_gemm_wgrad with a caller workspace",
                static_cast<long long>(Ci) * static_cast<long long>(Co),
                kStaticScratchBytes / sizeof(int));
  void* scratch = nullptr;
  if (Ci > 0 && Co > 0 && T > 0) {
    const int st = static_scratch_address(&scratch);
    if (st != SQ_OK) return st;
  }
  return run_gemm(2, xt_codes, ldx, gt_codes, ldg, Ci, Co, T, bits, n_groups, x_scale, g_scale,
                  x_exp, g_exp, dw, ld_dw, acc_out, ld_acc, scratch,
                  scratch ? kStaticScratchBytes : 0, dev_status, stream);
}
