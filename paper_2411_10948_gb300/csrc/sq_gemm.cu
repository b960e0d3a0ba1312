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
// Chunk length: the worst case assumes the largest shift on every inner index.  Where the
// inner channels' exponents are given (the layer launch), warp 2 of every CTA bounds the
// shifts per K block from them at the start, and the chunks take as many K blocks as
// max|q_A| max|q_B| x (largest per-block shift sum) x blocks <= 2^24 allows; with most
// channels in the last group (the usual case: tau_0 set by a few outlier channels) an
// 8-bit chunk grows from 2 K blocks to about 10.
//
// Persistent over output tiles: one CTA per SM with 128 x 256 tiles, or (for launches
// whose K loops are long) 2-CTA clusters with 256 x 256 tiles and cta_group::2 MMAs.
// The roles of a CTA:
//   warp 0      TMA producer: A and B tiles (128-byte rows, 128-byte swizzle) into a
//               shared-memory ring of 4 (pair: 6) stages
//   warp 1      TMEM allocation and the MMA issuer (one thread; a pair's leader only)
//   warp 2      the chunk plan (see above); then the dequantizing column factors of each
//               tile, ahead of the epilogue
//   warps 4-11  epilogue: tcgen05.ld, int32 accumulation across chunks, dequantizing
//               multiply, TMA stores of 32 x 32 boxes (or int32 TMA reductions into a
//               split-K workspace; plain stores where the output rows are not 16-byte
//               aligned)
// Work units reach the roles through a small shared-memory ring that the producer of the
// CTA (a pair's leader) fills: with a scheduling counter it takes each next unit from it
// (units are handed out in list order as CTAs free up), without one it strides over the
// list.
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

constexpr int kBM = 128;                      // output rows of a CTA (its TMEM lanes)
constexpr int kBN = 256;                      // output columns of a tile
constexpr int kBKBytes = 128;                 // one 128-byte swizzle row of K per stage
constexpr int kABytes = kBM * kBKBytes;       // 16 KB
constexpr int kThreads = 384;
constexpr int kEpiWarp0 = 4;
constexpr int kNumEpiWarps = 8;
constexpr int kFacWarp = 2;   // chunk plan, then the column factors
constexpr uint32_t kTmemCols = 2 * kBN;       // two FP32 accumulator buffers
constexpr int64_t kExactSum = int64_t(1) << 24;  // every partial sum of a chunk stays within this
// Two tile modes.  Single (kPair false): a CTA runs a 128 x 256 tile; a stage holds its
// 128 A rows and all 256 B rows (48 KB).  Pair (kPair true): a 2-CTA cluster runs a
// 256 x 256 tile with cta_group::2 MMAs issued by the leader; a stage holds a CTA's 128 A
// rows and 128 of the 256 B rows (32 KB), so the operand bytes each SM's shared memory
// takes in and hands to the tensor core drop by a third: a single CTA's 128 x 256 MMA
// needs more shared-memory bandwidth than the SM has and runs at about 70% of the tensor
// rate.  The epilogue of a pair is slower, though (about 20% per output box), so
// launches whose K loops are short keep single tiles.
//
// Shared memory of a CTA: the operand ring (4 stages single, 6 pair: about 1.3-1.5 us of
// MMA work, more than an operand tile takes to land while other SMs stream outputs), one
// 32 x 32 output staging box per epilogue warp (the box turns the lane-per-row TMEM layout
// into row-contiguous stores, or is the source of a TMA store), two per-tile column-factor
// tables, the barriers and the unit ring.
constexpr int kOutBox = 32;
constexpr int kUnitRing = 8;  // work units published by the producer ahead of the consumers
constexpr int kMaxSegGemms = 3;  // a launch holds at most three GEMMs
constexpr int kSegSlots = 12;    // segment starts of up to 8 groups (9 used)
constexpr int kOutStageBytes = kOutBox * kOutBox * 4;

template <bool kPair>
struct Smem {
  static constexpr int b_rows = kPair ? kBN / 2 : kBN;    // B rows (output columns) held
  static constexpr int tile_m = kPair ? 2 * kBM : kBM;    // output rows of a unit
  static constexpr int stage_bytes = kABytes + b_rows * kBKBytes;
  static constexpr int stages = kPair ? 6 : 4;
  static constexpr int out_offset = stages * stage_bytes;
  static constexpr int fac_offset = out_offset + kNumEpiWarps * kOutStageBytes;
  static constexpr int bar_offset = fac_offset + 2 * kBN * 4;
  // full, empty, tfull, tempty, fac, drain, unit ring full / empty, fac free, chunk plan
  static constexpr int num_bars = 2 * stages + 2 + 2 + 2 + 1 + 2 * kUnitRing + 2 + 1;
  static constexpr int ring_offset = bar_offset + num_bars * 8 + 16;  // after TMEM slot, flag
  static constexpr int chunk_offset = ring_offset + kUnitRing * 32;  // K blocks per chunk, per GEMM
  // group-ordered GEMMs: segment starts in K blocks (G + 1 of them), per GEMM
  static constexpr int seg_offset = chunk_offset + 4 * 4;
  static constexpr size_t bytes = seg_offset + kMaxSegGemms * kSegSlots * 4;
  static_assert(bytes <= 232448, "shared memory beyond the 227 KB per-CTA limit");
  static_assert(ring_offset % 16 == 0, "unit-ring slots are read as 16-byte vectors");
  static_assert(out_offset % 1024 == 0 && kOutStageBytes % 1024 == 0, "swizzle atoms need 1 KB");
};

struct GemmParams {
  int M, N, K;
  int m_tiles, n_tiles, splits, kb_total, kb_per_split, chunk_kb;
  int mode;  // 0: per-column scale (forward, loss propagation); 1: row/column shifts (wgrad)
  int G;
  int vec_y;  // output rows 16-byte aligned: 16-byte stores
  const float* a_scale;
  const float* b_scale;
  const uint8_t* row_exp;
  const uint8_t* col_exp;
  float* y;
  int64_t ldy;
  long long* acc;
  int64_t ld_acc;
  int* ws;  // split-K partial sums [M, N] (int32, or int64 when `wide`), or null
  int wide;  // the K loop exceeds the exact int32 range: splits add int64 sums
  // per-column max |output| (the next consumer's range pass, formed here), as the ordered
  // bit patterns of non-negative floats, zeroed before the launch; or null
  unsigned* colmax;
  int* status;
};

// Up to three GEMMs run by one persistent launch (the three GEMMs of a layer are
// independent).  Work units of all of them form one list, GEMM by GEMM in the order given
// (the host puts the GEMM with the longest K loop per unit first).
constexpr int kMaxBatch = 3;
struct GemmBatch {
  CUtensorMap a[kMaxBatch];
  CUtensorMap b[kMaxBatch];
  CUtensorMap y[kMaxBatch];   // fp32 output maps (outputs with 16-byte aligned rows)
  CUtensorMap ws[kMaxBatch];  // split-K workspace maps (unused when a GEMM does not split)
  GemmParams p[kMaxBatch];
  int unit_end[kMaxBatch];  // cumulative unit counts
  int count;
  int* sched;  // unit counter (zero before launch) for dynamic scheduling, or null
  // per GEMM: exponents e_k of the inner channels (forward, loss propagation; null:
  // worst-case chunks) and the bound max|q_A| max|q_B| of an unshifted product
  const uint8_t* k_exp[kMaxBatch];
  int raw_prod[kMaxBatch];
  int planned;  // some GEMM sizes its chunks from exponents (warp 2 plans them)
  int* status;
  int lazy_from;  // with the counter: from this unit on, a pair takes one unit at a time
  // failure-path self-test: the producer arms every stage but issues no copy, so the first
  // consumer wait runs out (nothing is ever in flight) and the launch takes its abort path
  int no_copies;
  // per GEMM: the group order of its inner index (segment starts in elements, then the
  // channel counts; a device table), or null.  A group-ordered GEMM's operands hold each
  // group's inner channels contiguously and unshifted; its chunks end at segment boundaries
  // and each chunk's sum is multiplied by the segment's shift 2^(G-1-g) in the epilogue.
  const int* seg[kMaxBatch];
  int segmented;  // some GEMM is group-ordered (every role waits for the table)
  // per GEMM: bit 0 set when A, bit 1 when B is stored MN-major ([K, ld] with the M or N
  // index contiguous: the weight gradient reading the activation and gradient codes in
  // their own layout instead of transposed copies); clear: K-major ([M or N, ld])
  int mn[kMaxBatch];
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
// exact integers (FP32 patterns when `as_float`, else int32); fac = shared-memory address
// of the box's 32 column factors (16-byte aligned), rfac the row's factor (weight gradient
// only: the forward and loss-propagation outputs take the column factor alone).  The box is staged in shared
// memory (128-byte swizzle) and leaves either as dequantized fp32 values through
// row-contiguous 16-byte stores (eight lanes per 128-byte row, four rows per instruction),
// as int32 partial sums through a TMA reduce-add into the split-K workspace, or -- past the
// int32 range -- as int64 additions (64-bit atomics, a row of 32 columns per instruction)
// into the int64 workspace.  The exactness-check integers are written when asked.
__device__ __forceinline__ void emit_box(const GemmParams& p, const CUtensorMap* tma_y,
                                         const CUtensorMap* tma_ws, const uint32_t (&vals)[32],
                                         bool as_float, uint32_t fac, float rfac, uint32_t buf,
                                         int64_t row0, int64_t col0, int lane) {
  const bool tma_out = p.ws != nullptr ? !p.wide : p.vec_y != 0;
  if (lane == 0) {
    // the last TMA store has read the box (it may belong to another GEMM of the launch,
    // whatever this box's own way out)
    bulk_wait_read<0>();
  }
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
  const bool row_scaled = p.mode == 1;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    uint32_t o[4];
    const float4 f4 = p.ws != nullptr ? make_float4(0.f, 0.f, 0.f, 0.f) : ld_shared_v4_f32(fac + k * 16);
    const float f[4] = {f4.x, f4.y, f4.z, f4.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t a = vals[k * 4 + e];
      if (p.ws != nullptr) {
        o[e] = as_float ? static_cast<uint32_t>(__float2int_rn(__uint_as_float(a))) : a;
      } else {
        const float val = as_float ? __uint_as_float(a) : __int2float_rn(static_cast<int32_t>(a));
        // x * 1 is x exactly, so skipping the row factor of 1 changes no result
        o[e] = __float_as_uint(__fmul_rn(row_scaled ? __fmul_rn(val, rfac) : val, f[e]));
      }
    }
    st_shared_v4(buf + lane * 128 + ((k ^ (lane & 7)) << 4), o[0], o[1], o[2], o[3]);
  }
  if (p.colmax != nullptr && p.ws == nullptr) {
    // The column maxima of |output| over the box's 32 rows, from the staged box: lane l
    // reads the four columns 4 (l & 7) .. +3 of the eight rows 8 (l >> 3) .. +7 (16-byte
    // loads), the four row groups combine by two exchanges, and lanes 0-7 add each column's
    // maximum to the output range (ordered bit patterns of |y|).
    __syncwarp();
    const int cq = lane & 7, rg = lane >> 3;
    uint32_t m[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int rr = rg * 8 + i;
      if (row0 + rr < p.M) {
        uint32_t v[4];
        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
                     : "r"(buf + rr * 128 + ((cq ^ (rr & 7)) << 4)));
#pragma unroll
        for (int e = 0; e < 4; ++e) m[e] = max(m[e], v[e] & 0x7FFFFFFFu);
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      m[e] = max(m[e], __shfl_xor_sync(0xFFFFFFFFu, m[e], 8));
      m[e] = max(m[e], __shfl_xor_sync(0xFFFFFFFFu, m[e], 16));
    }
    if (rg == 0) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int64_t col = col0 + cq * 4 + e;
        if (m[e] != 0u && col < p.N) atomicMax(p.colmax + col, m[e]);
      }
    }
  }
  if (p.ws != nullptr && p.wide) {
    // a split of a K loop beyond the int32 range: its exact int32 sums are added into the
    // int64 workspace, row by row (the lanes cover 32 consecutive columns of a row)
    __syncwarp();
    unsigned long long* w64 = reinterpret_cast<unsigned long long*>(p.ws);
    const int64_t col = col0 + lane;
    if (col < p.N) {
      for (int rr = 0; rr < 32; ++rr) {
        const int64_t row = row0 + rr;
        if (row >= p.M) break;
        const long long t = static_cast<int32_t>(staged(buf, rr, lane));
        atomicAdd(w64 + row * p.N + col, static_cast<unsigned long long>(t));
      }
    }
    __syncwarp();  // the staging box is free for the next one
    return;
  }
  if (tma_out) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (p.ws != nullptr)
        tma_reduce_add_2d(tma_ws, buf, static_cast<int32_t>(col0), static_cast<int32_t>(row0));
      else
        tma_store_2d(tma_y, buf, static_cast<int32_t>(col0), static_cast<int32_t>(row0));
      bulk_commit();
    }
    return;
  }
  __syncwarp();
  const int lr = lane >> 3;         // row within a group of four
  const int lc = lane & 7;          // 16-byte chunk within the 128-byte row
  const int64_t col = col0 + lc * 4;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int rr = i * 4 + lr;
    const int64_t row = row0 + rr;
    uint32_t v0, v1, v2, v3;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
                 : "r"(buf + rr * 128 + ((lc ^ (rr & 7)) << 4)));
    if (row < p.M) {
      float* dst = p.y + row * p.ldy + col;
      if (p.vec_y && col + 3 < p.N) {
        *reinterpret_cast<uint4*>(dst) = make_uint4(v0, v1, v2, v3);
      } else {
        if (col + 0 < p.N) dst[0] = __uint_as_float(v0);
        if (col + 1 < p.N) dst[1] = __uint_as_float(v1);
        if (col + 2 < p.N) dst[2] = __uint_as_float(v2);
        if (col + 3 < p.N) dst[3] = __uint_as_float(v3);
      }
    }
  }
  __syncwarp();  // the staging box is free for the next one
}

struct Unit {
  int mb, nb, kb0, kb1;
};

// A unit as the producer publishes it in the ring (one 32-byte slot): its GEMM g and its
// decoded tile and K range, so that no consumer repeats the decode (integer divisions and
// indexed parameter loads, about 0.5 us between two epilogue tiles).  g < 0: the end of
// the list.
struct RingUnit {
  int g;
  Unit w;
};

__device__ __forceinline__ void ring_put(volatile int* slot, const RingUnit& r) {
  asm volatile("st.volatile.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(smem_u32(const_cast<int*>(slot))),
               "r"(r.g), "r"(r.w.mb), "r"(r.w.nb), "r"(r.w.kb0)
               : "memory");
  slot[4] = r.w.kb1;
}

__device__ __forceinline__ void ring_put_cluster(uint32_t cluster_slot, const RingUnit& r) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(cluster_slot), "r"(r.g),
               "r"(r.w.mb), "r"(r.w.nb), "r"(r.w.kb0)
               : "memory");
  st_cluster_u32(cluster_slot + 16, static_cast<uint32_t>(r.w.kb1));
}

__device__ __forceinline__ RingUnit ring_get(const volatile int* slot) {
  RingUnit r;
  asm volatile("ld.volatile.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.g), "=r"(r.w.mb), "=r"(r.w.nb), "=r"(r.w.kb0)
               : "r"(smem_u32(const_cast<int*>(slot)))
               : "memory");
  r.w.kb1 = slot[4];
  return r;
}

// Work unit u -> (tile, K split).  Tiles go in groups of kGroupM row tiles: inside a group
// the row tile changes fastest, then the column tile.  The CTAs running at one time then
// cover a compact block of the output, so the A rows of a group stay in L2 while every
// column tile of B passes by, and neither operand is streamed from HBM more than once
// per group.
template <bool kPair>
__device__ __forceinline__ Unit decode_unit(const GemmParams& p, int u) {
  constexpr int kGroupM = kPair ? 8 : 16;  // 2048 output rows either way
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

// the GEMM of global unit u, and u's index inside that GEMM
__device__ __forceinline__ int batch_member(const GemmBatch& bt, int u, int* local) {
  int g = 0;
  while (g + 1 < bt.count && u >= bt.unit_end[g]) ++g;
  *local = u - (g ? bt.unit_end[g - 1] : 0);
  return g;
}

// Waits on the unit ring and the TMEM-release barriers, and arrivals on the leader's
// barriers: at cluster scope in a pair (the other CTA arrives, or wrote the ring slot),
// at CTA scope otherwise.
template <bool kPair>
__device__ __forceinline__ bool ring_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  if constexpr (kPair)
    return mbar_wait_cluster(bar, parity, abort_flag);
  else
    return mbar_wait(bar, parity, abort_flag);
}

template <bool kPair>
__device__ __forceinline__ void leader_arrive(uint64_t* local_bar, uint32_t cluster_bar) {
  if constexpr (kPair)
    mbar_arrive_cluster(cluster_bar);
  else
    mbar_arrive(local_bar);
}

// The chunk that starts at K block kc of a unit whose K loop ends at kend: its end and its
// shift exponent.  Without a segment table chunks are chunk_kb blocks; with one (segkb =
// the G + 1 segment starts in K blocks) a chunk also ends at its segment's end and carries
// the segment's shift G-1-g.  The producer, the MMA issuer and the epilogue walk the same
// sequence.
__device__ __forceinline__ int chunk_end(const volatile int* segkb, int G, int kc, int kend,
                                         int chunk_kb, int* shift) {
  int e = min(kend, kc + chunk_kb);
  *shift = 0;
  if (segkb != nullptr) {
    int s = 0;
    while (s + 1 < G && kc >= segkb[s + 1]) ++s;
    *shift = G - 1 - s;
    e = min(e, segkb[s + 1]);
  }
  return e;
}

// The factor warp: the dequantizing factor of each of a tile's 256 columns, into one of
// two tables ahead of the epilogue: s_A 2^-(G-1) s_B[n] (forward, loss propagation) or
// s_X s_dY 2^-eY_n (weight gradient; the row's 2^-eX_m is the epilogue's).  It reads the
// units from the same ring as the other roles; a table is refilled once every epilogue
// warp has released it (facfree).  Kept out of line: its registers stay its own.
template <bool kPair>
__device__ __noinline__ void factor_warp(const GemmBatch& bt, uint64_t* ufull,
                                         uint64_t* uempty, uint32_t uempty_c,
                                         volatile int* unit_ring,
                                         uint64_t* facbar, uint64_t* facfree, float* fac_tab,
                                         volatile int* abort_flag, uint32_t peer_abort_c,
                                         int lane) {
  bool ok = true;
  int us = 0;
  uint32_t uph = 0;
  for (int it = 0; ok; ++it) {
    if (!__all_sync(0xFFFFFFFFu, ring_wait<kPair>(&ufull[us], uph, abort_flag))) {
      ok = false;
      break;
    }
    const RingUnit r = ring_get(unit_ring + us * 8);
    __syncwarp();
    if (lane == 0) leader_arrive<kPair>(&uempty[us], uempty_c + us * 8);
    if (++us == kUnitRing) {
      us = 0;
      uph ^= 1u;
    }
    if (r.g < 0) break;
    const GemmParams& p = bt.p[r.g];
    const float a_fac = epilogue_a_factor(p);
    const int64_t n0 = static_cast<int64_t>(r.w.nb) * kBN;
    float f[kBN / 32];
#pragma unroll
    for (int j = 0; j < kBN / 32; ++j) {
      const int64_t col = n0 + lane + 32 * j;
      f[j] = 0.0f;
      if (col < p.N)
        f[j] = p.mode == 0 ? __fmul_rn(a_fac, __ldg(p.b_scale + col))
                           : __fmul_rn(a_fac, pow2_neg(__ldg(p.col_exp + col)));
    }
    // table it & 1 last held unit it - 2: wait until the epilogue is done with it
    if (it >= 2 &&
        !__all_sync(0xFFFFFFFFu, mbar_wait(&facfree[it & 1], ((it >> 1) & 1) ^ 1u, abort_flag))) {
      ok = false;
      break;
    }
    float* fac = fac_tab + (it & 1) * kBN;
#pragma unroll
    for (int j = 0; j < kBN / 32; ++j) fac[lane + 32 * j] = f[j];
    __syncwarp();
    if (lane == 0) mbar_arrive(&facbar[it & 1]);
  }
  if (!ok && lane == 0) {
    atomicOr(bt.status, kDevTimeout);
    *abort_flag = 1;
    if (peer_abort_c != 0) st_cluster_u32(peer_abort_c, 1);
  }
}

// The chunk length (K blocks) of every GEMM of the batch, into out[g], by one warp.  With
// the inner channels' exponents, a K block of channels c contributes products of at most
// raw_prod x sum_c 2^(G-1-e_c); the chunk takes as many blocks as keep the largest such
// sum times the block count within 2^24.  Never shorter than the worst-case chunk.
// block: inner elements per K block (128 bytes of codes: 64 or 128).  The exponents are
// read 16 at a time, four 16-byte loads of a lane in flight together.
__device__ __forceinline__ unsigned shift_weight(uint32_t word, int G, int64_t c, int64_t K) {
  unsigned w = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int e = (word >> (8 * i)) & 0xFF;
    if (c + i < K) w += 1u << (e >= G ? G - 1 : G - 1 - e);  // out of range: the largest shift
  }
  return w;
}

__device__ __noinline__ void plan_chunks(const GemmBatch& bt, volatile int* out, int lane,
                                         int block) {
  for (int g = 0; g < bt.count; ++g) {
    const GemmParams& p = bt.p[g];
    int chunk = p.chunk_kb;
    const uint8_t* k_exp = bt.k_exp[g];
    if (k_exp != nullptr) {
      const int spb = block / 16;                      // 16-channel segments per block
      const int64_t nseg = (static_cast<int64_t>(p.K) + 15) / 16;
      const bool vec = (reinterpret_cast<uintptr_t>(k_exp) & 15) == 0;
      unsigned wmax = 0;
      // 32 lanes cover 32 consecutive segments = 32 / spb whole blocks per round
      for (int64_t s0 = 0; s0 < nseg; s0 += 4 * 32) {
        unsigned wseg[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int64_t sg = s0 + r * 32 + lane;
          const int64_t c = sg * 16;
          uint32_t wd[4] = {0u, 0u, 0u, 0u};
          if (sg < nseg) {
            if (vec && c + 16 <= p.K) {
              const uint4 v = __ldg(reinterpret_cast<const uint4*>(k_exp + c));
              wd[0] = v.x; wd[1] = v.y; wd[2] = v.z; wd[3] = v.w;
            } else {
              for (int i = 0; i < 16 && c + i < p.K; ++i)
                wd[i >> 2] |= static_cast<uint32_t>(__ldg(k_exp + c + i)) << (8 * (i & 3));
            }
          }
          unsigned w = 0;
#pragma unroll
          for (int q = 0; q < 4; ++q) w += sg < nseg ? shift_weight(wd[q], p.G, c + 4 * q, p.K) : 0u;
          wseg[r] = w;
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          unsigned w = wseg[r];
          for (int o = 1; o < spb; o <<= 1) w += __shfl_xor_sync(0xFFFFFFFFu, w, o);
          wmax = max(wmax, w);   // every lane of a block's group holds the block's sum
        }
      }
      wmax = __reduce_max_sync(0xFFFFFFFFu, wmax);
      if (wmax > 0) {
        int64_t l = kExactSum / (static_cast<int64_t>(bt.raw_prod[g]) * wmax);
        if (l > (1 << 20)) l = 1 << 20;
        if (l > chunk) chunk = static_cast<int>(l);
      }
    }
    if (lane == 0) out[g] = chunk;
  }
}

// One operand tile of a pipeline stage: kRows rows of the M (or N) index from r0, one K
// block from k0, landing at dst (1 KB aligned) with its bytes counted on `bar`.
//   K-major: one box of kRows rows x 128 bytes of K.
//   MN-major: one box per 128 bytes of M (64 BF16 or 128 E4M3 elements) x the K block's
//   rows, placed one after another; each is a column of whole 1 KB swizzle atoms (8 K rows
//   of 128 bytes), which is the layout make_sdesc_mn_sw128 describes.
template <int kF8, bool kPair, int kRows>
__device__ __forceinline__ void load_operand(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                             int32_t k0, int32_t r0, bool mn) {
  constexpr int kBKElems = kF8 ? kBKBytes : kBKBytes / 2;
  constexpr int kMnElems = kF8 ? 128 : 64;
  if (!mn) {
    if constexpr (kPair)
      tma_load_2d_pair(dst, map, bar, k0, r0);
    else
      tma_load_2d(dst, map, bar, k0, r0);
    return;
  }
#pragma unroll
  for (int j = 0; j < kRows / kMnElems; ++j) {
    if constexpr (kPair)
      tma_load_2d_pair(dst + j * kBKElems * 128, map, bar, r0 + j * kMnElems, k0);
    else
      tma_load_2d(dst + j * kBKElems * 128, map, bar, r0 + j * kMnElems, k0);
  }
}

// The MMAs of one K block of a stage at a0 (A tile, then the B tile kABytes on), into the
// TMEM accumulator d (cleared by the block's first MMA when `first`).  An MMA takes 32
// bytes of K: 32 bytes along a K-major row, or that many 128-byte rows of an MN-major tile,
// whose 128-byte column blocks of M (N) lie a whole K block apart (a tile one block wide
// never steps to a second one, and its stride is given as one atom).
template <int kF8, int kCg, int kBRows, bool kAMn, bool kBMn>
__device__ __forceinline__ void mma_kblock(uint32_t d, uint32_t a0, bool first) {
  constexpr int kBKElems = kF8 ? kBKBytes : kBKBytes / 2;
  constexpr uint32_t kMnKStep = (kF8 ? 32 : 16) * 128;
  constexpr uint32_t kMnBlock = kBKElems * 128;
  constexpr uint32_t kStrideA = kBM * (kF8 ? 1 : 2) > 128 ? kMnBlock : 1024;
  constexpr uint32_t kStrideB = kBRows * (kF8 ? 1 : 2) > 128 ? kMnBlock : 1024;
  constexpr uint32_t idesc =
      make_idesc(kF8 ? 0u : 1u, kCg * kBM, kBN) | idesc_mn_major(kAMn, kBMn);
  const uint32_t b0 = a0 + kABytes;
#pragma unroll
  for (int k = 0; k < kBKBytes / 32; ++k) {
    const uint64_t ad = kAMn ? make_sdesc_mn_sw128(a0 + k * kMnKStep, kStrideA)
                             : make_sdesc_k_sw128(a0 + k * 32);
    const uint64_t bd = kBMn ? make_sdesc_mn_sw128(b0 + k * kMnKStep, kStrideB)
                             : make_sdesc_k_sw128(b0 + k * 32);
    const uint32_t accumulate = (!first || k > 0) ? 1u : 0u;
    if (kF8)
      tc_mma_f8<kCg>(d, ad, bd, idesc, accumulate);
    else
      tc_mma_f16<kCg>(d, ad, bd, idesc, accumulate);
  }
}

// kMulti: the K loop of a tile spans several exact chunks, whose int32 sums the epilogue
// keeps in registers; otherwise every output streams from TMEM once.
// kPair: launched as 2-CTA clusters running 256-row tiles (the host sets the cluster shape)
// kMn: some GEMM of the launch reads an operand MN-major (bt.mn); without it the copy and
// MMA loops hold the K-major form alone (measured: the MN branches in them, never taken,
// cost K-major launches 8-10%)
template <int kF8, bool kMulti, bool kPair, bool kMn>
__global__ void __launch_bounds__(kThreads, 1) shiftmm_kernel(const __grid_constant__ GemmBatch bt) {
  using L = Smem<kPair>;
  constexpr int kCg = kPair ? 2 : 1;
  constexpr int kStages = L::stages;
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {  // the swizzled layouts need 1 KB alignment
    if (threadIdx.x == 0) atomicOr(bt.status, kDevInternal);
    return;
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::bar_offset);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* tfull = bars + 2 * kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* facbar = tempty + 2;
  uint64_t* drain = facbar + 2;
  uint64_t* ufull = drain + 1;
  uint64_t* uempty = ufull + kUnitRing;
  uint64_t* facfree = uempty + kUnitRing;
  uint64_t* chunkbar = facfree + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(chunkbar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* unit_ring = reinterpret_cast<volatile int*>(smem + L::ring_offset);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kCg * kNumEpiWarps);  // the leader's: the epilogue warps of all CTAs
      mbar_init(&facbar[b], 1);                // the factor warp has filled table b
      mbar_init(&facfree[b], kNumEpiWarps);    // every epilogue warp is done with table b
    }
    mbar_init(drain, 1);
    mbar_init(chunkbar, 1);  // warp 2 has set the chunk length of every GEMM
    for (int r = 0; r < kUnitRing; ++r) {
      mbar_init(&ufull[r], 1);
      // the leader's: its MMA thread, and the producer (peer) or factor warp and every
      // epilogue warp of each CTA
      mbar_init(&uempty[r], kCg * (2 + kNumEpiWarps));
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int g = 0; g < bt.count; ++g) {
      tma_prefetch_desc(&bt.a[g]);
      tma_prefetch_desc(&bt.b[g]);
    }
  }
  if (warp == 1) {
    tmem_alloc<kCg>(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish<kCg>();
  }
  tc_fence_before();
  if constexpr (kPair)
    cluster_sync();  // both CTAs' barriers exist and their TMEM is allocated
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int units = bt.unit_end[bt.count - 1];
  constexpr int kBKElems = kF8 ? kBKBytes : kBKBytes / 2;
  // rank 0: the CTA that takes the units and issues the MMAs (a pair's leader, or a single CTA)
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;
  const int pair = static_cast<int>(blockIdx.x) / kCg;   // the CTA group's index
  const int npairs = static_cast<int>(gridDim.x) / kCg;  // CTA groups in the launch
  // the leader's unit-ring release and stage barriers; in a pair also the peer's ring and
  // the other CTA's abort flag (the epilogue forms its cluster addresses where it uses
  // them, which keeps them out of its registers)
  const uint32_t uempty_c = mapa_shared(smem_u32(uempty), 0);
  const uint32_t full_c = mapa_shared(smem_u32(full), 0);
  uint32_t peer_ring_c = 0, peer_ufull_c = 0, peer_abort_c = 0;
  if constexpr (kPair) {
    peer_ring_c = mapa_shared(smem_u32(const_cast<int*>(unit_ring)), 1);
    peer_ufull_c = mapa_shared(smem_u32(ufull), 1);
    peer_abort_c = mapa_shared(smem_u32(const_cast<int*>(abort_flag)), rank ^ 1u);
  }

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    // In a pair both CTAs load their halves of every stage: A rows m0 + 128 rank, B rows
    // (output columns) n0 + 128 rank.  The leader takes the units (from the counter, or
    // striding), publishes each to both CTAs' rings, and arms each stage's barrier for the
    // bytes of both halves; the peer's copies count their bytes on that barrier too.
    int s = 0;
    uint32_t ph = 0;
    long long issued = 0;
    bool ok = true;
    int next = pair;  // a pair's first unit is its own index
    int us = 0;
    uint32_t uph = 0;
    if (bt.segmented && !mbar_wait(chunkbar, 0, abort_flag)) ok = false;  // the segment table
    while (ok) {
      int u = next;
      RingUnit r;
      if (rank == 0) {
        // decode the unit and publish it (or, past the end, the stop mark) to the roles
        // of both CTAs
        r.g = -1;
        if (u < units) {
          int lu;
          r.g = batch_member(bt, u, &lu);
          r.w = decode_unit<kPair>(bt.p[r.g], lu);
        }
        if (!ring_wait<kPair>(&uempty[us], uph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        ring_put(unit_ring + us * 8, r);
        mbar_arrive(&ufull[us]);
        if constexpr (kPair) {
          ring_put_cluster(peer_ring_c + us * 32, r);
          mbar_arrive_cluster(peer_ufull_c + us * 8);
        }
      } else {
        if (!mbar_wait_cluster(&ufull[us], uph, abort_flag)) {
          ok = false;
          break;
        }
        r = ring_get(unit_ring + us * 8);
        mbar_arrive_cluster(uempty_c + us * 8);
      }
      if (++us == kUnitRing) {
        us = 0;
        uph ^= 1u;
      }
      if (r.g < 0) break;
      // Within the last waves of units a pair takes its next unit only once its epilogues
      // have started this one, so that no pair holds several queued units while others
      // run dry.
      const bool lazy = rank == 0 && bt.sched != nullptr && u >= bt.lazy_from;
      const int u_slot = us == 0 ? kUnitRing - 1 : us - 1;
      const uint32_t u_par = us == 0 ? uph ^ 1u : uph;
      if (rank == 0) {
        if (bt.sched == nullptr)
          next = u + npairs;
        else if (!lazy)
          next = npairs + atomicAdd(bt.sched, 1);
      }
      const int g = r.g;
      const Unit w = r.w;
      const int mn = kMn ? bt.mn[g] : 0;
      // rows past M (and columns past N) are read as zeros and never stored
      const int32_t ya = w.mb * L::tile_m + static_cast<int32_t>(rank) * kBM;
      const int32_t yb = w.nb * kBN + static_cast<int32_t>(rank) * L::b_rows;
      // a group-ordered GEMM's K loop stops at its padded width (the segment table's end)
      const int kend = bt.seg[g] != nullptr
                           ? min(w.kb1, reinterpret_cast<volatile int*>(smem + L::seg_offset)[g * kSegSlots + bt.p[g].G])
                           : w.kb1;
      for (int kb = w.kb0; kb < kend; ++kb) {
        if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t sa = smem_u32(smem + s * L::stage_bytes);
        if (rank == 0) mbar_arrive_expect_tx(&full[s], kCg * L::stage_bytes);
        if (!bt.no_copies) {
          if (!kMn || mn == 0) {
            if constexpr (kPair) {
              tma_load_2d_pair(sa, &bt.a[g], full_c + s * 8, kb * kBKElems, ya);
              tma_load_2d_pair(sa + kABytes, &bt.b[g], full_c + s * 8, kb * kBKElems, yb);
            } else {
              tma_load_2d(sa, &bt.a[g], smem_u32(&full[s]), kb * kBKElems, ya);
              tma_load_2d(sa + kABytes, &bt.b[g], smem_u32(&full[s]), kb * kBKElems, yb);
            }
          } else {
            const uint32_t bar = kPair ? full_c + s * 8 : smem_u32(&full[s]);
            load_operand<kF8, kPair, kBM>(sa, &bt.a[g], bar, kb * kBKElems, ya, mn & 1);
            load_operand<kF8, kPair, L::b_rows>(sa + kABytes, &bt.b[g], bar, kb * kBKElems, yb,
                                                mn & 2);
          }
          ++issued;
        }
        if (++s == kStages) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (ok && lazy) {
        if (!ring_wait<kPair>(&uempty[u_slot], u_par, abort_flag)) {
          ok = false;
          break;
        }
        next = npairs + atomicAdd(bt.sched, 1);
      }
    }
    if (!ok) {
      atomicOr(bt.status, kDevTimeout);
      *abort_flag = 1;
      if constexpr (kPair) st_cluster_u32(peer_abort_c, 1);
    }
    // Every issued copy must have landed before the CTAs may exit.  The leader's stage
    // barriers count both CTAs' bytes; after a timeout the peer cannot tell its own copies
    // apart there and gives them time instead (a copy lands within microseconds).
    if (rank == 0) {
      for (long long i = issued > kStages ? issued - kStages : 0; i < issued; ++i)
        mbar_wait(&full[i % kStages], static_cast<uint32_t>((i / kStages) & 1), nullptr);
    } else if (kPair && !ok) {
      const uint64_t t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 200000ull) {
      }
    }
  } else if (warp == 1 && lane == 0 && rank == 0) {
    // ------------------------------------------------- MMA issuer (the leader's)
    // In a pair: 256 x 256 MMAs; a stage is released in both CTAs, and a finished chunk
    // announced to both CTAs' epilogues, by multicast commits.
    int s = 0;
    uint32_t ph = 0;
    uint32_t c = 0;
    bool ok = !bt.planned || mbar_wait(chunkbar, 0, abort_flag);  // the chunk plan is in
    int us = 0;
    uint32_t uph = 0;
    while (ok) {
      if (!mbar_wait(&ufull[us], uph, abort_flag)) {
        ok = false;
        break;
      }
      const RingUnit r = ring_get(unit_ring + us * 8);
      mbar_arrive(&uempty[us]);
      if (++us == kUnitRing) {
        us = 0;
        uph ^= 1u;
      }
      if (r.g < 0) break;
      const int g = r.g;
      const int chunk_kb =
          bt.planned ? reinterpret_cast<volatile int*>(smem + L::chunk_offset)[g] : bt.p[g].chunk_kb;
      const Unit w = r.w;
      const volatile int* segkb =
          bt.seg[g] != nullptr ? reinterpret_cast<volatile int*>(smem + L::seg_offset) + g * kSegSlots : nullptr;
      const int kend = segkb != nullptr ? min(w.kb1, segkb[bt.p[g].G]) : w.kb1;
      const int mn = kMn ? bt.mn[g] : 0;
      int kce;
      for (int kc = w.kb0; kc < kend && ok; kc = kce) {
        int sh_unused;
        kce = chunk_end(segkb, bt.p[g].G, kc, kend, chunk_kb, &sh_unused);
        const uint32_t b = c & 1u, tph = (c >> 1) & 1u;
        if (!ring_wait<kPair>(&tempty[b], tph ^ 1u, abort_flag)) {  // every CTA's epilogue
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
          const uint32_t a0 = smem_u32(smem + s * L::stage_bytes);
          const bool first = kb == kc;
          if constexpr (!kMn) {
            mma_kblock<kF8, kCg, L::b_rows, false, false>(d, a0, first);
          } else {
            switch (mn) {  // the operand layouts as compile-time descriptor steps
              case 0: mma_kblock<kF8, kCg, L::b_rows, false, false>(d, a0, first); break;
              case 1: mma_kblock<kF8, kCg, L::b_rows, true, false>(d, a0, first); break;
              case 2: mma_kblock<kF8, kCg, L::b_rows, false, true>(d, a0, first); break;
              default: mma_kblock<kF8, kCg, L::b_rows, true, true>(d, a0, first); break;
            }
          }
          tc_commit<kCg>(smem_u32(&empty[s]), 0x3);  // frees the stage (in both CTAs)
          if (++s == kStages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit<kCg>(smem_u32(&tfull[b]), 0x3);  // chunk complete in TMEM buffer b
        ++c;
      }
    }
    if (!ok) {
      atomicOr(bt.status, kDevTimeout);
      *abort_flag = 1;
      if constexpr (kPair) st_cluster_u32(peer_abort_c, 1);
    }
    tc_commit<kCg>(smem_u32(drain), 0x1);  // every MMA issued has completed
    mbar_wait(drain, 0, nullptr);
  } else if (warp == kFacWarp) {
    // --------------------------------------------------- chunk plan, column factors
    if (bt.planned) {
      plan_chunks(bt, reinterpret_cast<volatile int*>(smem + L::chunk_offset), lane, kBKElems);
      volatile int* segkb = reinterpret_cast<volatile int*>(smem + L::seg_offset);
      for (int g = 0; g < bt.count; ++g)
        if (bt.seg[g] != nullptr && lane <= bt.p[g].G)
          segkb[g * kSegSlots + lane] = __ldg(bt.seg[g] + lane) / kBKElems;
      __syncwarp();
      if (lane == 0) mbar_arrive(chunkbar);
    }
    factor_warp<kPair>(bt, ufull, uempty, uempty_c, unit_ring, facbar, facfree,
                reinterpret_cast<float*>(smem + L::fac_offset), abort_flag, peer_abort_c, lane);
  } else if (warp >= kEpiWarp0) {
    // --------------------------------------------------------------- epilogue
    const int q = warp & 3;                       // TMEM lanes 32q .. 32q+31 (output rows)
    const int h = (warp - kEpiWarp0) >> 2;        // column half of the 256-wide tile
    const uint32_t stage_out0 =
        smem_u32(smem + L::out_offset + (warp - kEpiWarp0) * kOutStageBytes);
    float* fac_tab = reinterpret_cast<float*>(smem + L::fac_offset);
    uint32_t c = 0;
    bool ok = !bt.planned || __all_sync(0xFFFFFFFFu, mbar_wait(chunkbar, 0, abort_flag));
    int us = 0;
    uint32_t uph = 0;
    for (int it = 0; ok; ++it) {
      if (!__all_sync(0xFFFFFFFFu, ring_wait<kPair>(&ufull[us], uph, abort_flag))) {
        ok = false;
        break;
      }
      const RingUnit r = ring_get(unit_ring + us * 8);
      __syncwarp();
      if (lane == 0) leader_arrive<kPair>(&uempty[us], kPair ? mapa_shared(smem_u32(&uempty[us]), 0) : 0u);
      if (++us == kUnitRing) {
        us = 0;
        uph ^= 1u;
      }
      if (r.g < 0) break;
      const int g = r.g;
      const GemmParams& p = bt.p[g];
      const CUtensorMap* tma_y = &bt.y[g];
      const CUtensorMap* tma_ws = &bt.ws[g];
      const Unit w = r.w;
      const int ckb =
          bt.planned ? reinterpret_cast<volatile int*>(smem + L::chunk_offset)[g] : p.chunk_kb;
      const volatile int* segkb =
          bt.seg[g] != nullptr ? reinterpret_cast<volatile int*>(smem + L::seg_offset) + g * kSegSlots : nullptr;
      const int kend = segkb != nullptr ? min(w.kb1, segkb[p.G]) : w.kb1;
      const int64_t m0 = static_cast<int64_t>(w.mb) * L::tile_m + rank * kBM;  // this CTA's rows
      const int64_t n0 = static_cast<int64_t>(w.nb) * kBN;
      float* fac = fac_tab + (it & 1) * kBN;
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
            if (lane == 0) leader_arrive<kPair>(&tempty[b], kPair ? mapa_shared(smem_u32(&tempty[b]), 0) : 0u);  // b may take the next tile
          }
          const int64_t col0 = n0 + h * 128 + s * 32;
          if (row0 >= p.M || col0 >= p.N) continue;  // warp-uniform: nothing of this box exists
          const uint32_t buf = stage_out0;
          emit_box(p, tma_y, tma_ws, v, true, smem_u32(fac + h * 128 + s * 32), rfac, buf, row0,
                           col0, lane);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&facfree[it & 1]);  // this warp is done with the table
        ++c;
      } else {
        uint32_t acc[128];  // int32 sums of the chunks
        if (kend <= w.kb0) {
          // a split of a group-ordered GEMM that lies past its padded width: no chunk
#pragma unroll
          for (int i = 0; i < 128; ++i) acc[i] = 0u;
        }
        int kce;
        for (int kc = w.kb0, ch = 0; kc < kend; kc = kce, ++ch) {
          int sh;
          kce = chunk_end(segkb, p.G, kc, kend, ckb, &sh);
          const int32_t mul = 1 << sh;  // the segment's shift (1 without a segment table)
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
            // Each FP32 value is an integer of magnitude <= 2^24.  Below 2^22, adding
            // 1.5 * 2^23 lands it in [2^23, 2^24), where the FP32 spacing is 1, so the
            // integer is the bit pattern minus that of 1.5 * 2^23: an exact conversion on
            // the FP32 and integer pipes.  The conversion unit (a fraction of their rate,
            // and the limit of short chunks) takes groups holding a larger value.
            float vmax = 0.0f;
#pragma unroll
            for (int i = 0; i < 16; ++i) vmax = fmaxf(vmax, fabsf(__uint_as_float(v[i])));
            if (__all_sync(0xFFFFFFFFu, vmax < 4194304.0f)) {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const int32_t t =
                    (__float_as_int(__fadd_rn(__uint_as_float(v[i]), 12582912.0f)) - 0x4B400000) * mul;
                acc[j * 16 + i] =
                    static_cast<uint32_t>(ch == 0 ? t : static_cast<int32_t>(acc[j * 16 + i]) + t);
              }
            } else {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const int32_t t = __float2int_rn(__uint_as_float(v[i])) * mul;
                acc[j * 16 + i] =
                    static_cast<uint32_t>(ch == 0 ? t : static_cast<int32_t>(acc[j * 16 + i]) + t);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) leader_arrive<kPair>(&tempty[b], kPair ? mapa_shared(smem_u32(&tempty[b]), 0) : 0u);  // b may take the next chunk
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
          const uint32_t buf = stage_out0;
          emit_box(p, tma_y, tma_ws, v, false, smem_u32(fac + h * 128 + s * 32), rfac, buf, row0,
                           col0, lane);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&facfree[it & 1]);  // this warp is done with the table
      }
    }
    if (!ok) {
      atomicOr(bt.status, kDevTimeout);
      *abort_flag = 1;
      if constexpr (kPair) st_cluster_u32(mapa_shared(smem_u32(const_cast<int*>(abort_flag)), rank ^ 1u), 1);
    }
    if (lane == 0) bulk_wait_read<0>();  // no store still reads shared memory at exit
  }

  // neither CTA of a pair leaves while the other may still reach its barriers, shared
  // memory or TMEM
  tc_fence_before();
  if constexpr (kPair)
    cluster_sync();
  else
    __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc<kCg>(tmem_base, kTmemCols);
  }
}

// split-K: turn the summed int32 partials into the outputs, four consecutive outputs of a
// row per thread (a split GEMM has N % 4 == 0); every load of a thread leaves at once
__global__ void __launch_bounds__(256) splitk_finalize_kernel(const GemmParams p) {
  const float a_fac = epilogue_a_factor(p);
  const int nq = p.N / 4;
  const int64_t quads = static_cast<int64_t>(p.M) * nq;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < quads;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = i / nq;
    const int64_t col = (i - row * nq) * 4;
    const int4 t4 = __ldcs(reinterpret_cast<const int4*>(p.ws) + i);
    const int tv[4] = {t4.x, t4.y, t4.z, t4.w};
    float o[4];
    long long t[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) epilogue_value(p, row, col + e, tv[e], a_fac, &o[e], &t[e]);
    if (p.colmax) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t b = __float_as_uint(o[e]) & 0x7FFFFFFFu;
        if (b != 0u) atomicMax(p.colmax + col + e, b);
      }
    }
    float* dst = p.y + row * p.ldy + col;
    if (p.vec_y) {
      *reinterpret_cast<float4*>(dst) = make_float4(o[0], o[1], o[2], o[3]);
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) dst[e] = o[e];
    }
    if (p.acc) {
#pragma unroll
      for (int e = 0; e < 4; ++e) p.acc[row * p.ld_acc + col + e] = t[e];
    }
  }
}

// The same from int64 sums (a K loop beyond the int32 range), one output per thread: the one
// dequantizing multiply of the epilogue with T converted to FP32 once (round to nearest).
__global__ void __launch_bounds__(256) splitk_finalize_wide_kernel(const GemmParams p) {
  const float a_fac = epilogue_a_factor(p);
  const long long* ws = reinterpret_cast<const long long*>(p.ws);
  const int64_t n = static_cast<int64_t>(p.M) * p.N;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = i / p.N;
    const int64_t col = i - row * p.N;
    const long long t = __ldcs(ws + i);
    float y;
    long long tc;
    if (p.mode == 0) {
      y = __fmul_rn(__ll2float_rn(t), __fmul_rn(a_fac, __ldg(p.b_scale + col)));
      tc = t;
    } else {
      const int er = __ldg(p.row_exp + row), ec = __ldg(p.col_exp + col);
      y = __fmul_rn(__fmul_rn(__ll2float_rn(t), pow2_neg(er + ec)), a_fac);
      tc = t << (2 * (p.G - 1) - er - ec);
    }
    p.y[row * p.ldy + col] = y;
    if (p.colmax) {
      const uint32_t b = __float_as_uint(y) & 0x7FFFFFFFu;
      if (b != 0u) atomicMax(p.colmax + col, b);
    }
    if (p.acc) p.acc[row * p.ld_acc + col] = tc;
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

// MN-major operand: K rows of `mn` elements, leading dimension ld (elements), the M (or N)
// index contiguous: boxes of 128 bytes of M x one K block of rows, 128-byte swizzle, zero
// fill outside the tensor
static int make_operand_map_mn(CUtensorMap* map, const void* base, int64_t mn, int64_t K,
                               int64_t ld, int elem_bytes) {
  auto fn = encode_fn();
  if (!fn) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  const CUtensorMapDataType dt =
      elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(mn), static_cast<cuuint64_t>(K)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(ld * elem_bytes)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBKBytes / elem_bytes),
                       static_cast<cuuint32_t>(kBKBytes / elem_bytes)};
  cuuint32_t estride[2] = {1, 1};
  const CUresult r = fn(map, dt, 2, const_cast<void*>(base), gdim, gstride, box, estride,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SQ_ECUDA, "cuTensorMapEncodeTiled (MN-major) failed (%d)", static_cast<int>(r));
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
  int wide;  // max|T| can pass 2^31: every split stays within int32, splits add in int64
};

// max |product| of one inner index as the tensor core sees it: q_A q_B 2^(G-1) with the
// shift folded into B (forward, loss propagation), or q_A q_B with the shifts applied
// after the sum (the weight gradient; a group-ordered GEMM, whose chunks are shifted whole)
static int64_t max_product(int which, int bits, int G, bool seg = false) {
  const int64_t Q = q_of_bits(bits);
  return (which == 2 || seg) ? Q * Q : (Q * Q) << (G - 1);
}

// max |T| per inner index: the shifted product, however the shift is applied
static int64_t max_total_product(int which, int bits, int G) { return max_product(which, bits, G); }

// The exactness limit of the FP32 accumulation, checked before anything touches the device:
// one K block of worst-case products must stay within 2^24 (the chunks are whole K blocks).
// K itself is not limited: past the int32 range the K loop is split (see make_plan).
static int check_exact_range(int which, int64_t K, int bits, int G, bool seg = false) {
  (void)K;
  const int64_t P = max_product(which, bits, G, seg);
  const int bk = kBKBytes / code_bytes(code_type(bits, G));
  if (kExactSum / P < bk)
    return fail(SQ_EUNSUPPORTED,
                "bits=%d with n_groups=%d: one %d-wide K block can exceed the exact FP32 sum range",
                bits, G, bk);
  return SQ_OK;
}

// The int32 limit of a sum that is added across ranks as int32 (the sharded weight
// gradient): max|T| = max|product| K must stay below 2^31.
static int check_int32_range(int which, int64_t K, int bits, int G) {
  const int64_t P = max_product(which, bits, G);
  if (P * K > INT32_MAX)
    return fail(SQ_EUNSUPPORTED,
                "inner dimension %lld exceeds the exact int32 range for bits=%d, n_groups=%d "
                "(max |T| = %lld * K)",
                static_cast<long long>(K), bits, G, static_cast<long long>(P));
  return check_exact_range(which, K, bits, G);
}

// Tiles of 128 (pair: 256) x 256 outputs spread over `workers` (SMs, or CTA pairs).
// max_splits: 1 never splits K; 0 lets the worker count alone decide.
static int make_plan(int which, int64_t M, int64_t N, int64_t K, int bits, int G, int workers,
                     int max_splits, bool pair, Plan* pl, bool seg = false) {
  const int st = check_exact_range(which, K, bits, G, seg);
  if (st != SQ_OK) return st;
  const int64_t P = max_product(which, bits, G, seg);
  pl->elem_bytes = code_bytes(code_type(bits, G));
  const int bk = kBKBytes / pl->elem_bytes;
  pl->chunk_kb = static_cast<int>((kExactSum / P) / bk);
  if (pl->chunk_kb > (1 << 20)) pl->chunk_kb = 1 << 20;
  const int tile_m = pair ? 2 * kBM : kBM;
  pl->m_tiles = static_cast<int>((M + tile_m - 1) / tile_m);
  pl->n_tiles = static_cast<int>((N + kBN - 1) / kBN);
  pl->kb_total = static_cast<int>((K + bk - 1) / bk);
  const int64_t tiles = static_cast<int64_t>(pl->m_tiles) * pl->n_tiles;
  int splits = 1;
  if (max_splits != 1 && tiles < workers && pl->kb_total >= 4) {
    splits = static_cast<int>(workers / tiles);
    if (splits > pl->kb_total / 2) splits = pl->kb_total / 2;
    if (max_splits > 1 && splits > max_splits) splits = max_splits;
    if (splits < 1) splits = 1;
  }
  // Past the int32 range every split keeps its K loop within it (its int32 register sums
  // stay exact) and the splits add in int64: at least this many, whatever max_splits says.
  const int64_t kb_int32 = (INT32_MAX / max_total_product(which, bits, G)) / bk;  // >= 1
  pl->wide = pl->kb_total > kb_int32 ? 1 : 0;
  if (pl->wide) {
    const int need = static_cast<int>((pl->kb_total + kb_int32 - 1) / kb_int32);
    if (splits < need) splits = need;
  }
  pl->kb_per_split = (pl->kb_total + splits - 1) / splits;
  pl->splits = (pl->kb_total + pl->kb_per_split - 1) / pl->kb_per_split;
  return SQ_OK;
}

// Split-K workspace of one GEMM: the partial sums [M, N] (int32, or int64 past the int32
// range), zeroed before every launch that uses them, rounded up to 256 bytes.
static size_t split_ws_bytes(int64_t M, int64_t N, bool wide = false) {
  const size_t eb = wide ? sizeof(long long) : sizeof(int);
  return (static_cast<size_t>(M) * static_cast<size_t>(N) * eb + 255) & ~size_t(255);
}
// The layer launch's workspace starts with the unit counter of its dynamic schedule.
constexpr size_t kSchedBytes = 256;

template <int kF8, bool kMulti, bool kPair, bool kMn>
static int configure_kernel(int dev) {
  static bool done[64] = {};
  if (dev >= 0 && dev < 64 && done[dev]) return SQ_OK;
  const cudaError_t err = cudaFuncSetAttribute(shiftmm_kernel<kF8, kMulti, kPair, kMn>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(Smem<kPair>::bytes));
  if (err != cudaSuccess) return cuda_fail(err, "cudaFuncSetAttribute");
  if (dev >= 0 && dev < 64) done[dev] = true;
  return SQ_OK;
}

// CTA pairs of the GEMM kernel resident at once: one per two SMs, fewer where the GPU's
// SM groups leave single SMs over.  -1 without a device.
static int device_pairs(int* dev_out) {
  static int cached[64] = {};
  int dev = 0;
  const int sms = device_sms(&dev);
  if (sms <= 0) return -1;
  if (dev_out) *dev_out = dev;
  if (dev >= 0 && dev < 64 && cached[dev] > 0) return cached[dev];
  int pairs = sms / 2;
  if (configure_kernel<1, false, true, false>(dev) == SQ_OK) {
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * pairs);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = Smem<true>::bytes;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, shiftmm_kernel<1, false, true, false>, &cfg) !=
        cudaSuccess)
      cudaGetLastError();  // an unanswered query leaves no error behind
    else if (n > 0 && n < pairs)
      pairs = n;
  }
  if (pairs < 1) pairs = 1;
  if (dev >= 0 && dev < 64) cached[dev] = pairs;
  return pairs;
}

// One GEMM of a launch: out[M, N] = A[M, K] B[N, K]^T with the operand roles of `which`
// (0 forward, 1 loss propagation, 2 weight gradient).
struct GemmJob {
  int which;
  const void* a;
  int64_t lda;
  const void* b;
  int64_t ldb;
  int64_t M, N, K;
  const float* a_scale;
  const float* b_scale;
  const uint8_t* row_exp;
  const uint8_t* col_exp;
  float* y;
  int64_t ldy;
  int64_t* acc;
  int64_t ld_acc;
  void* ws;
  size_t ws_bytes;
  const uint8_t* k_exp;  // exponents of the inner channels (forward, loss propagation), or null
  int partial;  // weight gradient: int32 sums into ws (the caller's), no dequantizing pass
  float* colmax;  // per-column max |output| [N], formed by the epilogue, or null
  const int* seg;  // group order of the inner index (device table), or null
  // operands stored MN-major: a as [K, lda] with M contiguous, b as [K, ldb] with N
  // contiguous (the weight gradient on the codes' own layout); else K-major
  int a_mn, b_mn;
};

static const char* job_name(int which) {
  static const char* names[3] = {"gemm_fwd", "gemm_dgrad", "gemm_wgrad"};
  return names[which];
}

// Argument checks of one GEMM; *launch is false when there is nothing for the kernel to do
// (an empty output, or K == 0 whose zero result is written here with memsets).
static int check_job(const GemmJob& j, int bits, int G, int32_t* dev_status, cudaStream_t s,
                     bool* launch) {
  const char* nm = job_name(j.which);
  *launch = false;
  if (!bits_ok(bits) || !groups_ok(G))
    return fail(SQ_EINVAL, "%s: bits must be in [2, 8] and n_groups in [1, 8]", nm);
  if (j.M < 0 || j.N < 0 || j.K < 0) return fail(SQ_EINVAL, "%s: negative size", nm);
  if (j.M > INT32_MAX || j.N > INT32_MAX || j.K > INT32_MAX)
    return fail(SQ_EUNSUPPORTED, "%s: dimensions beyond 2^31", nm);
  if (dev_status == nullptr) return fail(SQ_EINVAL, "%s: dev_status is required", nm);
  if (j.M == 0 || j.N == 0) return SQ_OK;
  if (!j.partial) {  // a partial call writes int32 sums only, no fp32 output
    if (j.y == nullptr || j.ldy < j.N) return fail(SQ_EINVAL, "%s: output is NULL or its ld < N", nm);
    if (j.acc != nullptr && j.ld_acc < j.N) return fail(SQ_EINVAL, "%s: ld_acc < N", nm);
  }
  // the kernel reads the scales and exponents of every tile (a partial call too)
  if (j.a_scale == nullptr || j.b_scale == nullptr)
    return fail(SQ_EINVAL, "%s: scales are required", nm);
  if (j.which == 2 && (j.row_exp == nullptr || j.col_exp == nullptr))
    return fail(SQ_EINVAL, "%s: exponents are required", nm);
  if (j.K == 0 && j.partial) {
    const cudaError_t err = cudaMemsetAsync(j.ws, 0, static_cast<size_t>(j.M) * j.N * sizeof(int), s);
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemsetAsync");
  }
  if (j.K == 0) {
    // an empty inner sum: T = 0 everywhere
    cudaError_t err = cudaMemset2DAsync(j.y, j.ldy * sizeof(float), 0, j.N * sizeof(float), j.M, s);
    if (err == cudaSuccess && j.acc)
      err = cudaMemset2DAsync(j.acc, j.ld_acc * sizeof(int64_t), 0, j.N * sizeof(int64_t), j.M, s);
    return err == cudaSuccess ? SQ_OK : cuda_fail(err, "cudaMemset2DAsync");
  }
  if (j.a == nullptr || j.b == nullptr) return fail(SQ_EINVAL, "%s: codes are NULL", nm);
  if (j.lda < (j.a_mn ? j.M : j.K) || j.ldb < (j.b_mn ? j.N : j.K))
    return fail(SQ_EINVAL, "%s: operand ld smaller than its row", nm);
  const int eb = code_bytes(code_type(bits, G));
  if (!aligned16(j.a) || !aligned16(j.b) || (j.lda * eb) % 16 != 0 || (j.ldb * eb) % 16 != 0)
    return fail(SQ_EALIGN, "%s: operand pointers must be 16-byte aligned and ld * %d bytes a "
                "multiple of 16", nm, eb);
  const int st = check_exact_range(j.which, j.K, bits, G, j.seg != nullptr);
  if (st != SQ_OK) return st;
  *launch = true;
  return SQ_OK;
}

// Tiles and K splits of one checked GEMM: the SM count decides the splits, up to
// max_splits, and a split needs a workspace for the [M, N] int32 partial sums (added by TMA
// into N-element rows, which must stay 16-byte aligned).
static int plan_job(const GemmJob& j, int bits, int G, int workers, int max_splits, bool pair,
                    Plan* pl) {
  const bool sg = j.seg != nullptr;
  const int st = make_plan(j.which, j.M, j.N, j.K, bits, G, workers, max_splits, pair, pl, sg);
  if (st != SQ_OK || pl->splits <= 1 || j.partial) return st;  // partial: ws is the output
  if (pl->wide) {
    // int64 sums need their workspace; there is no unsplit way to stay exact
    if (j.ws == nullptr || j.ws_bytes < split_ws_bytes(j.M, j.N, true) || !aligned16(j.ws))
      return fail(SQ_EUNSUPPORTED,
                  "%s: inner dimension %lld exceeds the exact int32 range for bits=%d, "
                  "n_groups=%d; int64 accumulation needs a 16-byte aligned workspace of %zu bytes "
                  "(shiftquant_gemm_workspace_bytes)",
                  job_name(j.which), static_cast<long long>(j.K), bits, G,
                  split_ws_bytes(j.M, j.N, true));
    return SQ_OK;
  }
  if (j.ws == nullptr || j.ws_bytes < split_ws_bytes(j.M, j.N) || !aligned16(j.ws) || j.N % 4 != 0)
    return make_plan(j.which, j.M, j.N, j.K, bits, G, workers, 1, pair, pl, sg);
  return SQ_OK;
}

// Pair tiles where a launch's units run long K loops, so that the tensor core sets the
// pace; with short K loops the epilogue does, and single tiles run it faster.  Decided
// from single-tile plans: the average K blocks per unit.  Measured on layer launches:
// pairs 18% faster at 118 K blocks (16384 x 4096 x 11008), 2% at 27 (12608 x 768 x 3072),
// even at 25, 4% slower at 14.5 and 18% slower at 5 (12544 x 2304 x 256, E4M3).
constexpr int kPairMinKb = 26;
static bool pair_mode(const GemmJob* const* jobs, int n, int bits, int G, int sms, int pairs) {
  if (pairs <= 0) return false;
  double units = 0.0, kb = 0.0;
  for (int i = 0; i < n; ++i) {
    const GemmJob& j = *jobs[i];
    if (j.M <= 0 || j.N <= 0 || j.K <= 0) continue;
    Plan pl;
    if (make_plan(j.which, j.M, j.N, j.K, bits, G, sms, 0, false, &pl, j.seg != nullptr) != SQ_OK)
      continue;
    const double u = static_cast<double>(pl.m_tiles) * pl.n_tiles * pl.splits;
    units += u;
    kb += u * pl.kb_per_split;
  }
  return units > 0.0 && kb >= kPairMinKb * units;
}

// Sharing the launch with other GEMMs, a split GEMM needs fewer splits: just enough that
// its units stay well inside the launch's expected length.  Every split adds the whole
// output once more to the L2 reductions, whose throughput is far below a plain store's.
// Unit cost model, in K-block times: the K loop plus about 8 for the epilogue.
static int balance_splits(GemmJob* const* jobs, int n, int bits, int G, int workers, bool pair,
                          Plan* plans) {
  if (n <= 1) return SQ_OK;
  constexpr double kEpiKb = 8.0;
  double work = 0.0;  // the batch's total cost, with every split GEMM at its maximum
  for (int g = 0; g < n; ++g)
    work += static_cast<double>(plans[g].m_tiles) * plans[g].n_tiles * plans[g].splits *
            (plans[g].kb_per_split + kEpiKb);
  for (int g = 0; g < n; ++g) {
    if (plans[g].splits <= 1) continue;
    const double tiles = static_cast<double>(plans[g].m_tiles) * plans[g].n_tiles;
    int s = 1;
    for (; s < plans[g].splits; ++s) {
      const double kbs = static_cast<double>((plans[g].kb_total + s - 1) / s);
      const double w = work - tiles * plans[g].splits * (plans[g].kb_per_split + kEpiKb) +
                       tiles * s * (kbs + kEpiKb);
      if (kbs + kEpiKb <= 0.8 * w / workers) break;
    }
    if (s < plans[g].splits) {
      const int st = plan_job(*jobs[g], bits, G, workers, s, pair, &plans[g]);
      if (st != SQ_OK) return st;
    }
  }
  return SQ_OK;
}

// Slot g of the batch for one planned GEMM: tensor maps and parameters.
static int prepare_job(const GemmJob& j, const Plan* pl, int bits, int G, int32_t* dev_status,
                       bool pair, GemmBatch* bt, int g) {
  int st;
  const int eb = pl->elem_bytes;
  st = j.a_mn ? make_operand_map_mn(&bt->a[g], j.a, j.M, j.K, j.lda, eb)
              : make_operand_map(&bt->a[g], j.a, j.M, j.K, j.lda, eb, kBM);
  if (st != SQ_OK) return st;
  st = j.b_mn ? make_operand_map_mn(&bt->b[g], j.b, j.N, j.K, j.ldb, eb)
              : make_operand_map(&bt->b[g], j.b, j.N, j.K, j.ldb, eb, pair ? kBN / 2 : kBN);
  if (st != SQ_OK) return st;
  bt->mn[g] = (j.a_mn ? 1 : 0) | (j.b_mn ? 2 : 0);
  GemmParams& p = bt->p[g];
  p.M = static_cast<int>(j.M);
  p.N = static_cast<int>(j.N);
  p.K = static_cast<int>(j.K);
  p.m_tiles = pl->m_tiles;
  p.n_tiles = pl->n_tiles;
  p.splits = pl->splits;
  p.kb_total = pl->kb_total;
  p.kb_per_split = pl->kb_per_split;
  p.chunk_kb = pl->chunk_kb;
  // exponent-sized chunks pay where worst-case chunks would split a unit three ways or more
  // (8-bit); elsewhere the planning only costs time
  bt->k_exp[g] = (j.which == 2 || j.seg != nullptr || pl->kb_per_split <= 2 * pl->chunk_kb)
                    ? nullptr
                    : j.k_exp;
  bt->seg[g] = j.seg;
  bt->raw_prod[g] = q_of_bits(bits) * q_of_bits(bits);
  p.mode = j.which == 2 ? 1 : 0;
  p.G = G;
  p.vec_y = (j.ldy % 4 == 0) && aligned16(j.y);
  p.a_scale = j.a_scale;
  p.b_scale = j.b_scale;
  p.row_exp = j.row_exp;
  p.col_exp = j.col_exp;
  p.y = j.y;
  p.ldy = j.ldy;
  p.acc = reinterpret_cast<long long*>(j.acc);
  p.ld_acc = j.ld_acc;
  p.ws = (pl->splits > 1 || j.partial) ? static_cast<int*>(j.ws) : nullptr;
  p.wide = pl->wide;
  p.colmax = reinterpret_cast<unsigned*>(j.colmax);
  p.status = dev_status;
  memset(&bt->y[g], 0, sizeof(CUtensorMap));
  memset(&bt->ws[g], 0, sizeof(CUtensorMap));
  if (p.ws && !p.wide)
    st = make_output_map(&bt->ws[g], p.ws, j.M, j.N, j.N, CU_TENSOR_MAP_DATA_TYPE_INT32);
  else if (p.vec_y)
    st = make_output_map(&bt->y[g], j.y, j.M, j.N, j.ldy, CU_TENSOR_MAP_DATA_TYPE_FLOAT32);
  return st;
}

template <int kF8, bool kMulti, bool kPair, bool kMn>
static int launch_kernel(const GemmBatch& bt, int grid, int dev, cudaStream_t s) {
  const int st = configure_kernel<kF8, kMulti, kPair, kMn>(dev);
  if (st != SQ_OK) return st;
  cudaError_t err;
  if constexpr (kPair) {
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = Smem<true>::bytes;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    err = cudaLaunchKernelEx(&cfg, shiftmm_kernel<kF8, kMulti, true, kMn>, bt);
    if (err == cudaSuccess) err = cudaGetLastError();
  } else {
    shiftmm_kernel<kF8, kMulti, false, kMn><<<grid, kThreads, Smem<false>::bytes, s>>>(bt);
    err = cudaGetLastError();
  }
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "shiftmm_kernel launch");
}

template <int kF8, bool kMn>
static int launch_variant(const GemmBatch& bt, int grid, int dev, cudaStream_t s, bool multi,
                          bool pair) {
  if (pair)
    return multi ? launch_kernel<kF8, true, true, kMn>(bt, grid, dev, s)
                 : launch_kernel<kF8, false, true, kMn>(bt, grid, dev, s);
  return multi ? launch_kernel<kF8, true, false, kMn>(bt, grid, dev, s)
               : launch_kernel<kF8, false, false, kMn>(bt, grid, dev, s);
}

// Checks, plans and launches up to kMaxBatch GEMMs (all with the same bits / n_groups) as
// one persistent kernel; split-K partial sums are zeroed before and finalized after it.
// sched (may be null): a unit counter, zeroed here before the launch, through which the
// CTAs take their units as they free up -- for batches whose units differ in length.
// Without one each CTA strides over the unit list.
static int run_jobs(GemmJob* jobs, int njobs, int bits, int G, int32_t* dev_status, void* stream,
                    int* sched, int max_ctas = 0, bool no_copies = false) {
  cudaStream_t s = as_stream(stream);
  int live[kMaxBatch];
  int nlive = 0;
  for (int i = 0; i < njobs; ++i)
    if (jobs[i].colmax != nullptr && (reinterpret_cast<uintptr_t>(jobs[i].colmax) & 3u) != 0)
      return fail(SQ_EALIGN, "%s: column-range output must be 4-byte aligned", job_name(jobs[i].which));
  for (int i = 0; i < njobs; ++i) {
    bool launch = false;
    const int st = check_job(jobs[i], bits, G, dev_status, s, &launch);
    if (st != SQ_OK) return st;
    if (launch) live[nlive++] = i;
  }
  // column ranges start at 0 (an output with no rows, or K == 0, keeps them there)
  for (int i = 0; i < njobs; ++i) {
    if (jobs[i].colmax == nullptr || jobs[i].N <= 0) continue;
    const cudaError_t err = cudaMemsetAsync(jobs[i].colmax, 0, static_cast<size_t>(jobs[i].N) * sizeof(float), s);
    if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  }
  if (nlive == 0) return SQ_OK;
  int dev = 0;
  const int sms = device_sms(&dev);
  if (sms <= 0) return fail(SQ_ECUDA, "%s: no current CUDA device", job_name(jobs[live[0]].which));
  GemmBatch bt;
  memset(&bt, 0, sizeof(bt));
  Plan plans[kMaxBatch];
  GemmJob* lj[kMaxBatch];
  for (int g = 0; g < nlive; ++g) lj[g] = &jobs[live[g]];
  const bool partial = nlive == 1 && lj[0]->partial;  // only single-GEMM calls are partial
  const int pairs = device_pairs(nullptr);
  const bool pair = pair_mode(lj, nlive, bits, G, sms, pairs);
  const int workers = pair ? pairs : sms;  // CTA groups resident at once
  for (int g = 0; g < nlive; ++g) {
    const int st = plan_job(*lj[g], bits, G, workers, 0, pair, &plans[g]);
    if (st != SQ_OK) return st;
  }
  int st = balance_splits(lj, nlive, bits, G, workers, pair, plans);
  if (st != SQ_OK) return st;
  for (int g = 0; g < nlive; ++g)
    if ((st = prepare_job(*lj[g], &plans[g], bits, G, dev_status, pair, &bt, g)) != SQ_OK)
      return st;
  // longest K loop per unit first: the short units then fill in behind the long ones
  for (int a = 0; a < nlive; ++a)
    for (int b = a + 1; b < nlive; ++b)
      if (plans[b].kb_per_split > plans[a].kb_per_split) {
        const GemmParams tp = bt.p[a]; bt.p[a] = bt.p[b]; bt.p[b] = tp;
        const Plan tl = plans[a]; plans[a] = plans[b]; plans[b] = tl;
        CUtensorMap t;
        t = bt.a[a]; bt.a[a] = bt.a[b]; bt.a[b] = t;
        t = bt.b[a]; bt.b[a] = bt.b[b]; bt.b[b] = t;
        t = bt.y[a]; bt.y[a] = bt.y[b]; bt.y[b] = t;
        t = bt.ws[a]; bt.ws[a] = bt.ws[b]; bt.ws[b] = t;
        const uint8_t* te = bt.k_exp[a]; bt.k_exp[a] = bt.k_exp[b]; bt.k_exp[b] = te;
        const int* ts = bt.seg[a]; bt.seg[a] = bt.seg[b]; bt.seg[b] = ts;
        const int tr = bt.raw_prod[a]; bt.raw_prod[a] = bt.raw_prod[b]; bt.raw_prod[b] = tr;
        const int tm = bt.mn[a]; bt.mn[a] = bt.mn[b]; bt.mn[b] = tm;
      }
  int units = 0;
  bool multi = false;
  for (int g = 0; g < nlive; ++g) {
    units += plans[g].m_tiles * plans[g].n_tiles * plans[g].splits;
    bt.unit_end[g] = units;
    multi |= plans[g].kb_per_split > plans[g].chunk_kb;  // a unit spans several exact chunks
    multi |= bt.seg[g] != nullptr;  // chunks end at segment boundaries and carry their shifts
  }
  bt.count = nlive;
  bt.status = dev_status;
  bt.sched = sched;
  bt.no_copies = no_copies ? 1 : 0;
  bt.planned = 0;
  bt.segmented = 0;
  for (int g = 0; g < nlive; ++g) {
    bt.planned |= bt.k_exp[g] != nullptr || bt.seg[g] != nullptr;
    bt.segmented |= bt.seg[g] != nullptr;
  }
  // zero the counter and the partial sums, with one memset for the regions that follow the
  // counter back to back
  char* zero_from = reinterpret_cast<char*>(sched);
  char* zero_end = sched ? zero_from + kSchedBytes : nullptr;
  cudaError_t err;
  for (int g = 0; g < nlive; ++g) {
    if (!bt.p[g].ws) continue;
    char* w = reinterpret_cast<char*>(bt.p[g].ws);
    // a partial call's sums go to the caller's buffer of exactly M N words
    const size_t b = partial ? static_cast<size_t>(bt.p[g].M) * bt.p[g].N * sizeof(int)
                             : split_ws_bytes(bt.p[g].M, bt.p[g].N, bt.p[g].wide != 0);
    if (zero_end != nullptr && w == zero_end) {
      zero_end = w + b;
      continue;
    }
    err = cudaMemsetAsync(w, 0, b, s);
    if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  }
  if (zero_from != nullptr) {
    err = cudaMemsetAsync(zero_from, 0, static_cast<size_t>(zero_end - zero_from), s);
    if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
  }
  // CTA groups (pairs, or single CTAs); a cap on the CTAs leaves at least one group
  const int cg = pair ? 2 : 1;
  int ngroups = units < workers ? units : workers;
  if (max_ctas > 0 && ngroups > max_ctas / cg) ngroups = max_ctas / cg > 0 ? max_ctas / cg : 1;
  const int grid = cg * ngroups;
  // A CTA group holds up to about stages / K-blocks + 2 units of the last (shortest) GEMM
  // at once: its operand ring and two TMEM buffers.  Over that many final waves it takes
  // one unit at a time, so the groups run out of work together.
  {
    const int kb = plans[nlive - 1].kb_per_split > 0 ? plans[nlive - 1].kb_per_split : 1;
    const int stages = pair ? Smem<true>::stages : Smem<false>::stages;
    const int depth = 2 + (stages + kb - 1) / kb;
    const long long from = static_cast<long long>(units) - static_cast<long long>(depth) * ngroups;
    bt.lazy_from = from > 0 ? static_cast<int>(from) : 0;
  }
  bool mn = false;
  for (int g = 0; g < nlive; ++g) mn |= bt.mn[g] != 0;
  if (plans[0].elem_bytes == 1)
    st = mn ? launch_variant<1, true>(bt, grid, dev, s, multi, pair)
            : launch_variant<1, false>(bt, grid, dev, s, multi, pair);
  else
    st = mn ? launch_variant<0, true>(bt, grid, dev, s, multi, pair)
            : launch_variant<0, false>(bt, grid, dev, s, multi, pair);
  if (st != SQ_OK) return st;
  for (int g = 0; g < nlive; ++g) {
    if (!bt.p[g].ws || partial) continue;
    const int64_t items = static_cast<int64_t>(bt.p[g].M) * (bt.p[g].wide ? bt.p[g].N : bt.p[g].N / 4);
    int64_t blocks = (items + 255) / 256;
    if (blocks > static_cast<int64_t>(sms) * 16) blocks = static_cast<int64_t>(sms) * 16;
    if (bt.p[g].wide)
      splitk_finalize_wide_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(bt.p[g]);
    else
      splitk_finalize_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(bt.p[g]);
    err = cudaGetLastError();
    if (err != cudaSuccess) return cuda_fail(err, "splitk_finalize_kernel launch");
  }
  return SQ_OK;
}

static int run_gemm(int which, const void* a_codes, int64_t lda, const void* b_codes, int64_t ldb,
                    int64_t M, int64_t N, int64_t K, int bits, int G, const float* a_scale,
                    const float* b_scale, const uint8_t* row_exp, const uint8_t* col_exp,
                    float* y, int64_t ldy, int64_t* acc_out, int64_t ld_acc, void* workspace,
                    size_t workspace_bytes, int32_t* dev_status, void* stream) {
  GemmJob j{which, a_codes, lda, b_codes, ldb, M, N, K, a_scale, b_scale, row_exp, col_exp,
            y, ldy, acc_out, ld_acc, workspace, workspace_bytes};
  return run_jobs(&j, 1, bits, G, dev_status, stream, nullptr);
}

// The three GEMMs of a layer as jobs, workspace regions assigned to those that split.
static void layer_jobs(const sq_layer_gemms* a, GemmJob jobs[3], int mask) {
  jobs[0] = GemmJob{0, a->x_codes, a->ld_x, a->wf_codes, a->ld_wf, a->M, a->N, a->K, a->x_scale,
                    a->wf_scale, nullptr, nullptr, a->y, a->ld_y, a->acc_y, a->ld_acc_y, nullptr, 0};
  jobs[1] = GemmJob{1, a->g_codes, a->ld_g, a->wd_codes, a->ld_wd, a->M, a->K, a->N, a->g_scale,
                    a->wd_scale, nullptr, nullptr, a->dx, a->ld_dx, a->acc_dx, a->ld_acc_dx, nullptr, 0};
  // without a transposed copy the weight gradient reads X's (dY's) codes MN-major
  const bool x_mn = a->xt_codes == nullptr, g_mn = a->gt_codes == nullptr;
  jobs[2] = GemmJob{2, x_mn ? a->x_codes : a->xt_codes, x_mn ? a->ld_x : a->ld_xt,
                    g_mn ? a->g_codes : a->gt_codes, g_mn ? a->ld_g : a->ld_gt, a->K, a->N, a->M,
                    a->x_scale, a->g_scale, a->x_exp, a->g_exp, a->dw, a->ld_dw, a->acc_dw,
                    a->ld_acc_dw, nullptr, 0};
  jobs[2].a_mn = x_mn;
  jobs[2].b_mn = g_mn;
  jobs[0].k_exp = a->x_exp;  // the forward GEMM's inner channels are X's
  jobs[1].k_exp = a->g_exp;  // loss propagation's are dY's
  jobs[0].colmax = a->y_range;
  jobs[1].colmax = a->dx_range;
  // group-ordered inner indices: the operands span the padded width of the order
  if (a->x_seg != nullptr) {
    jobs[0].seg = a->x_seg;
    jobs[0].K = shiftquant_group_order_width(a->K, a->bits, a->n_groups);
  }
  if (a->g_seg != nullptr) {
    jobs[1].seg = a->g_seg;
    jobs[1].K = shiftquant_group_order_width(a->N, a->bits, a->n_groups);
  }
  // a GEMM left out of the mask becomes empty: nothing of it is checked or launched
  for (int i = 0; i < 3; ++i)
    if (mask != 0 && !(mask & (1 << i))) jobs[i].M = 0;
}

// Bytes of split-K workspace each GEMM of the layer would use (0: it would not split),
// a multiple of 256 bytes.
static void layer_ws_need(const GemmJob jobs[3], int bits, int G, int sms, int pairs,
                          size_t need[3]) {
  const GemmJob* jp[3] = {&jobs[0], &jobs[1], &jobs[2]};
  const bool pair = pair_mode(jp, 3, bits, G, sms, pairs);
  for (int i = 0; i < 3; ++i) {
    need[i] = 0;
    const GemmJob& j = jobs[i];
    if (j.M <= 0 || j.N <= 0 || j.K <= 0) continue;
    Plan pl;
    if (make_plan(j.which, j.M, j.N, j.K, bits, G, pair ? pairs : sms, 0, pair, &pl,
                  j.seg != nullptr) != SQ_OK)
      continue;
    if (!pl.wide && j.N % 4 != 0) continue;  // int32 splits are added by 16-byte TMA rows
    if (pl.splits > 1) need[i] = split_ws_bytes(j.M, j.N, pl.wide != 0);
  }
}

// The layer workspace: the unit counter, then a split-K region for each GEMM that would
// split, as far as the workspace reaches.  Returns the counter (null without a usable
// workspace: the launch then strides over its units and splits nothing).
static int* assign_layer_ws(GemmJob jobs[3], int bits, int G, int sms, int pairs, void* workspace,
                            size_t workspace_bytes) {
  if (workspace == nullptr || workspace_bytes < kSchedBytes || !aligned16(workspace)) return nullptr;
  if (sms > 0) {
    size_t need[3];
    layer_ws_need(jobs, bits, G, sms, pairs, need);
    size_t off = kSchedBytes;
    for (int i = 0; i < 3; ++i) {
      if (need[i] == 0 || off + need[i] > workspace_bytes) continue;
      jobs[i].ws = static_cast<char*>(workspace) + off;
      jobs[i].ws_bytes = need[i];
      off += need[i];
    }
  }
  return static_cast<int*>(workspace);
}

// ----------------------------------------------- allocation-free weight gradient
// Scratch for callers that cannot allocate device memory themselves: a fixed array in
// the library's own device image, present on every GPU that loads the library until the
// process exits.  It serves as the split-K int32 workspace of
// shiftquant_gemm_wgrad_static().
constexpr int64_t kStaticMaxOutputs = int64_t(1) << 20;  // Ci * Co
constexpr size_t kStaticScratchBytes = size_t(4) << 20;   // the int32 sums of 2^20 outputs
static __device__ __align__(256) int g_wgrad_scratch[kStaticScratchBytes / sizeof(int)];

// Device address of g_wgrad_scratch on the current device.  In host code the array's
// name only stands in for the symbol, so the address is looked up with the device
// current: on every call made outside stream capture (a device reset re-creates the
// array elsewhere, and the lookup is cheap), and the last address found is kept per device
// for calls made while `s` is being captured, which must not make that lookup.
static int static_scratch_address(void** out, cudaStream_t s) {
  static void* addr[64] = {};
  static std::mutex mu;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return cuda_fail(err, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(SQ_EUNSUPPORTED, "device index %d beyond 63", dev);
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  err = cudaStreamIsCapturing(s, &cap);
  if (err != cudaSuccess) return cuda_fail(err, "cudaStreamIsCapturing");
  std::lock_guard<std::mutex> lock(mu);
  if (cap == cudaStreamCaptureStatusNone) {
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_wgrad_scratch);
    if (err != cudaSuccess) return cuda_fail(err, "cudaGetSymbolAddress");
    addr[dev] = p;
  } else if (addr[dev] == nullptr) {
    return fail(SQ_EINVAL,
                "gemm_wgrad_static: the first call on a device must come before any stream "
                "capture (it looks up the scratch array's address)");
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
  const int pairs = device_pairs(nullptr);
  GemmJob j{};
  j.which = which;
  j.M = M;
  j.N = N;
  j.K = K;
  const GemmJob* jp = &j;
  const bool pair = pair_mode(&jp, 1, bits, n_groups, sms, pairs);
  Plan pl;
  if (make_plan(which, M, N, K, bits, n_groups, pair ? pairs : sms, 0, pair, &pl) != SQ_OK) return 0;
  if (!pl.wide && N % 4 != 0) return 0;
  return pl.splits > 1 ? split_ws_bytes(M, N, pl.wide != 0) : 0;
}

extern "C" sq_status shiftquant_gemm_wgrad_partial(
    const void* xt_codes, int64_t ldx, const float* x_scale, const uint8_t* x_exp,
    const void* gt_codes, int64_t ldg, const float* g_scale, const uint8_t* g_exp, int64_t Ci,
    int64_t Co, int64_t T, int64_t total_tokens, int bits, int n_groups, int32_t* t_out,
    int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "gemm_wgrad_partial: bits must be in [2, 8] and n_groups in [1, 8]");
  if (Ci < 0 || Co < 0 || T < 0 || total_tokens < T)
    return fail(SQ_EINVAL, "gemm_wgrad_partial: negative size or total_tokens < T");
  if (Ci == 0 || Co == 0) return SQ_OK;
  if (t_out == nullptr || !aligned16(t_out) || Co % 4 != 0)
    return fail(SQ_EALIGN, "gemm_wgrad_partial: t_out must be 16-byte aligned and Co a multiple of 4");
  // the summed partials must stay in the exact int32 range for the whole token count
  int st = check_int32_range(2, total_tokens, bits, n_groups);
  if (st != SQ_OK) return st;
  GemmJob j{2, xt_codes, ldx, gt_codes, ldg, Ci, Co, T, x_scale, g_scale, x_exp, g_exp,
            nullptr, 0, nullptr, 0, t_out, static_cast<size_t>(Ci) * Co * sizeof(int32_t)};
  j.partial = 1;
  return run_jobs(&j, 1, bits, n_groups, dev_status, stream, nullptr);
}

extern "C" sq_status shiftquant_gemm_wgrad_finish(const int32_t* t, int64_t Ci, int64_t Co,
                                                  int bits, int n_groups, const float* x_scale,
                                                  const uint8_t* x_exp, const float* g_scale,
                                                  const uint8_t* g_exp, float* dw, int64_t ld_dw,
                                                  int64_t* acc_out, int64_t ld_acc,
                                                  int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  if (!bits_ok(bits) || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "gemm_wgrad_finish: bits must be in [2, 8] and n_groups in [1, 8]");
  if (Ci < 0 || Co < 0) return fail(SQ_EINVAL, "gemm_wgrad_finish: negative size");
  if (Ci == 0 || Co == 0) return SQ_OK;
  if (t == nullptr || !aligned16(t) || Co % 4 != 0)
    return fail(SQ_EALIGN, "gemm_wgrad_finish: t must be 16-byte aligned and Co a multiple of 4");
  if (dw == nullptr || ld_dw < Co || x_scale == nullptr || g_scale == nullptr ||
      x_exp == nullptr || g_exp == nullptr || dev_status == nullptr ||
      (acc_out != nullptr && ld_acc < Co))
    return fail(SQ_EINVAL, "gemm_wgrad_finish: NULL argument or ld < Co");
  int dev = 0;
  const int sms = device_sms(&dev);
  if (sms <= 0) return fail(SQ_ECUDA, "gemm_wgrad_finish: no current CUDA device");
  GemmParams p;
  memset(&p, 0, sizeof(p));
  p.M = static_cast<int>(Ci);
  p.N = static_cast<int>(Co);
  p.mode = 1;
  p.G = n_groups;
  p.vec_y = (ld_dw % 4 == 0) && aligned16(dw);
  p.a_scale = x_scale;
  p.b_scale = g_scale;
  p.row_exp = x_exp;
  p.col_exp = g_exp;
  p.y = dw;
  p.ldy = ld_dw;
  p.acc = reinterpret_cast<long long*>(acc_out);
  p.ld_acc = ld_acc;
  p.ws = const_cast<int*>(t);
  p.status = dev_status;
  if (Ci > INT32_MAX || Co > INT32_MAX)
    return fail(SQ_EUNSUPPORTED, "gemm_wgrad_finish: dimensions beyond 2^31");
  const int64_t quads = Ci * (Co / 4);
  int64_t blocks = (quads + 255) / 256;
  if (blocks > static_cast<int64_t>(sms) * 16) blocks = static_cast<int64_t>(sms) * 16;
  splitk_finalize_kernel<<<static_cast<unsigned>(blocks), 256, 0, as_stream(stream)>>>(p);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, "splitk_finalize_kernel launch");
}

extern "C" sq_status shiftquant_gemm_wgrad_static(
    const void* xt_codes, int64_t ldx, const float* x_scale, const uint8_t* x_exp,
    const void* gt_codes, int64_t ldg, const float* g_scale, const uint8_t* g_exp, int64_t Ci,
    int64_t Co, int64_t T, int bits, int n_groups, float* dw, int64_t ld_dw, int64_t* acc_out,
    int64_t ld_acc, int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  // compared by division, so that no product of huge sizes can overflow
  if (Ci > 0 && Co > 0 && (Ci > kStaticMaxOutputs || Co > kStaticMaxOutputs / Ci))
    return fail(SQ_EUNSUPPORTED,
                "gemm_wgrad_static: Ci = %lld, Co = %lld exceed the %lld outputs of the "
                "library's static scratch; use shiftquant_gemm_wgrad with a caller workspace",
                static_cast<long long>(Ci), static_cast<long long>(Co),
                static_cast<long long>(kStaticMaxOutputs));
  void* scratch = nullptr;
  if (Ci > 0 && Co > 0 && T > 0) {
    const int st = static_scratch_address(&scratch, as_stream(stream));
    if (st != SQ_OK) return st;
  }
  return run_gemm(2, xt_codes, ldx, gt_codes, ldg, Ci, Co, T, bits, n_groups, x_scale, g_scale,
                  x_exp, g_exp, dw, ld_dw, acc_out, ld_acc, scratch,
                  scratch ? kStaticScratchBytes : 0, dev_status, stream);
}

extern "C" sq_status shiftquant_gemm_layer(const sq_layer_gemms* args, void* workspace,
                                           size_t workspace_bytes, int32_t* dev_status,
                                           void* stream) {
  fail(SQ_OK, "");
  if (args == nullptr) return fail(SQ_EINVAL, "gemm_layer: args is NULL");
  if (!bits_ok(args->bits) || !groups_ok(args->n_groups))
    return fail(SQ_EINVAL, "gemm_layer: bits must be in [2, 8] and n_groups in [1, 8]");
  if (args->gemm_mask < 0 || args->gemm_mask > 7 || args->max_ctas < 0)
    return fail(SQ_EINVAL, "gemm_layer: gemm_mask must be in [0, 7] and max_ctas >= 0");
  const bool wgrad = args->gemm_mask == 0 || (args->gemm_mask & 4);
  if (wgrad && ((args->xt_codes == nullptr && args->x_seg != nullptr) ||
                (args->gt_codes == nullptr && args->g_seg != nullptr)))
    return fail(SQ_EINVAL, "gemm_layer: a group-ordered operand needs its transposed copy "
                "(xt_codes / gt_codes) for the weight gradient");
  GemmJob jobs[3];
  layer_jobs(args, jobs, args->gemm_mask);
  const int sms = device_sms(nullptr);
  const int pairs = device_pairs(nullptr);
  int* sched =
      assign_layer_ws(jobs, args->bits, args->n_groups, sms, pairs, workspace, workspace_bytes);
  return run_jobs(jobs, 3, args->bits, args->n_groups, dev_status, stream, sched, args->max_ctas);
}

extern "C" sq_status shiftquant_selftest_wait_timeout(const void* a_codes, int64_t lda,
                                                      const float* a_scale, const void* b_codes,
                                                      int64_t ldb, const float* b_scale, int64_t M,
                                                      int64_t N, int64_t K, int bits, int n_groups,
                                                      float* y, int64_t ldy, int32_t* dev_status,
                                                      void* stream) {
  fail(SQ_OK, "");
  if (M <= 0 || N <= 0 || K <= 0)
    return fail(SQ_EINVAL, "selftest_wait_timeout: the launch needs a non-empty GEMM");
  if (M > 4096 || N > 4096 || K > 4096)
    return fail(SQ_EINVAL, "selftest_wait_timeout: M, N and K must be at most 4096");
  GemmJob j{0, a_codes, lda, b_codes, ldb, M, N, K, a_scale, b_scale, nullptr, nullptr,
            y, ldy, nullptr, 0, nullptr, 0};
  return run_jobs(&j, 1, bits, n_groups, dev_status, stream, nullptr, 0, true);
}

static size_t layer_workspace_bytes(int64_t M, int64_t K, int64_t N, int bits, int n_groups,
                                    bool grouped) {
  if (!bits_ok(bits) || !groups_ok(n_groups)) return 0;
  const int sms = device_sms(nullptr);
  if (sms <= 0) return 0;
  const int pairs = device_pairs(nullptr);
  sq_layer_gemms a;
  memset(&a, 0, sizeof(a));
  a.M = M;
  a.K = K;
  a.N = N;
  a.bits = bits;
  a.n_groups = n_groups;
  if (grouped) {  // the plan reads only whether a table exists: a stand-in address serves
    a.x_seg = reinterpret_cast<const int32_t*>(static_cast<uintptr_t>(256));
    a.g_seg = a.x_seg;
  }
  GemmJob jobs[3];
  layer_jobs(&a, jobs, 0);
  size_t need[3];
  layer_ws_need(jobs, bits, n_groups, sms, pairs, need);
  return kSchedBytes + need[0] + need[1] + need[2];
}

extern "C" size_t shiftquant_gemm_layer_workspace_bytes(int64_t M, int64_t K, int64_t N, int bits,
                                                        int n_groups) {
  return layer_workspace_bytes(M, K, N, bits, n_groups, false);
}

extern "C" size_t shiftquant_gemm_layer_workspace_bytes_grouped(int64_t M, int64_t K, int64_t N,
                                                                int bits, int n_groups) {
  return layer_workspace_bytes(M, K, N, bits, n_groups, true);
}

extern "C" int shiftquant_gemm_layer_kernel_launches(int64_t M, int64_t K, int64_t N, int bits,
                                                     int n_groups, size_t workspace_bytes,
                                                     int gemm_mask) {
  if (!bits_ok(bits) || !groups_ok(n_groups) || M < 0 || K < 0 || N < 0 || gemm_mask < 0 ||
      gemm_mask > 7)
    return -1;
  const int sms = device_sms(nullptr);
  if (sms <= 0) return -1;
  const int pairs = device_pairs(nullptr);
  sq_layer_gemms a;
  memset(&a, 0, sizeof(a));
  a.M = M;
  a.K = K;
  a.N = N;
  GemmJob jobs[3];
  layer_jobs(&a, jobs, gemm_mask);
  // the plan looks at the workspace's size and alignment only: a stand-in address serves
  assign_layer_ws(jobs, bits, n_groups, sms, pairs, workspace_bytes ? reinterpret_cast<void*>(4096) : nullptr,
                  workspace_bytes);
  Plan plans[kMaxBatch];
  GemmJob* lj[kMaxBatch];
  int n = 0;
  for (int i = 0; i < 3; ++i)
    if (jobs[i].M != 0 && jobs[i].N != 0 && jobs[i].K != 0) lj[n++] = &jobs[i];
  if (n == 0) return 0;
  const bool pair = pair_mode(lj, n, bits, n_groups, sms, pairs);
  const int workers = pair ? pairs : sms;
  for (int g = 0; g < n; ++g)
    if (plan_job(*lj[g], bits, n_groups, workers, 0, pair, &plans[g]) != SQ_OK) return -1;
  if (balance_splits(lj, n, bits, n_groups, workers, pair, plans) != SQ_OK) return -1;
  int launches = 1;
  for (int g = 0; g < n; ++g) launches += plans[g].splits > 1;
  return launches;
}

// Whether the weight gradient of a layer launch should read X's and dY's codes in place
// (MN-major operands) rather than transposed copies.  Measured on GB300: an MMA with an
// MN-major operand (either or both) runs 8% (E4M3) to 16-20% (BF16) slower than the K-major
// form once the tensor core sets the pace -- pair tiles, a full wave of unsplit units with
// long K loops (16384 x 4096 x 11008: 729 -> 924 us; 4096^3: 95 -> 113 us) -- and within
// 2-4% where the launch is bound by split-K reductions or epilogues (12608 x 3072 x 768,
// 12544 x 2304 x 256), where dropping the copies' quantizer writes wins.
extern "C" int shiftquant_gemm_layer_wgrad_in_place(int64_t M, int64_t K, int64_t N, int bits,
                                                    int n_groups) {
  const int pair = shiftquant_gemm_layer_cta_pairs(M, K, N, bits, n_groups, 0);
  if (pair < 0) return -1;
  if (pair == 0) return 1;
  const int pairs = device_pairs(nullptr);
  Plan pl;
  if (make_plan(2, K, N, M, bits, n_groups, pairs, 0, true, &pl) != SQ_OK) return -1;
  const int64_t units = static_cast<int64_t>(pl.m_tiles) * pl.n_tiles * pl.splits;
  const bool mma_bound = pl.splits == 1 && 2 * units >= pairs && pl.kb_per_split >= 64;
  return mma_bound ? 0 : 1;
}

extern "C" int shiftquant_gemm_layer_cta_pairs(int64_t M, int64_t K, int64_t N, int bits,
                                               int n_groups, int gemm_mask) {
  if (!bits_ok(bits) || !groups_ok(n_groups) || M < 0 || K < 0 || N < 0 || gemm_mask < 0 ||
      gemm_mask > 7)
    return -1;
  const int sms = device_sms(nullptr);
  if (sms <= 0) return -1;
  const int pairs = device_pairs(nullptr);
  sq_layer_gemms a;
  memset(&a, 0, sizeof(a));
  a.M = M;
  a.K = K;
  a.N = N;
  GemmJob jobs[3];
  layer_jobs(&a, jobs, gemm_mask);
  const GemmJob* lj[3];
  int n = 0;
  for (int i = 0; i < 3; ++i) {
    if (jobs[i].M == 0 || jobs[i].N == 0 || jobs[i].K == 0) continue;
    if (check_exact_range(jobs[i].which, jobs[i].K, bits, n_groups) != SQ_OK) return -1;
    lj[n++] = &jobs[i];
  }
  if (n == 0) return -1;
  return pair_mode(lj, n, bits, n_groups, sms, pairs) ? 1 : 0;
}
