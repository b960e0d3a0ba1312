// Packed sub-byte storage (Sec. 5.2: with N_G = 4 the grouping map takes exactly 2 bits):
// codes of at most 4 bits two per byte, and the grouping map in 1 / 2 / 4-bit fields.
//
// The tensor cores of sm_103a have no integer inputs and no 4-bit format that holds the
// integers -7..7 (E2M1 lacks 5 and 7), so a GEMM reads codes as E4M3 bytes; the packed form
// is the storage of a quantized tensor kept between its quantization and its use -- an
// activation saved for the backward pass takes half the bytes -- and is expanded back to
// the operand format before the GEMM that reads it.  Both directions are streaming HBM
// passes: sixteen codes per thread, 16-byte loads and 8-byte stores where rows allow.
//
// Layout: element c of a row in byte c / 2 of the packed row, the low nibble for even c,
// as a 4-bit two's complement; map field of channel c at bit (c mod (8 / w)) w of byte
// c / (8 / w), w = 1, 2, 4 for N_G <= 2, <= 4, <= 8.
#include <cuda_fp16.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include "sq_device.cuh"
#include "sq_host.h"

namespace sq {

template <typename CodeT>
__device__ __forceinline__ int code_value(CodeT v);

template <>
__device__ __forceinline__ int code_value<uint8_t>(uint8_t v) {
  const __half_raw h = __nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(v), __NV_E4M3);
  return static_cast<int>(__half2float(__half(h)));
}

template <>
__device__ __forceinline__ int code_value<uint16_t>(uint16_t v) {
  return static_cast<int>(__uint_as_float(static_cast<uint32_t>(v) << 16));
}

template <typename CodeT>
__device__ __forceinline__ CodeT code_of(int q);

template <>
__device__ __forceinline__ uint8_t code_of<uint8_t>(int q) {
  return static_cast<uint8_t>(__nv_cvt_float_to_fp8(static_cast<float>(q), __NV_SATFINITE, __NV_E4M3));
}

template <>
__device__ __forceinline__ uint16_t code_of<uint16_t>(int q) {
  return static_cast<uint16_t>(__float_as_uint(static_cast<float>(q)) >> 16);
}

constexpr int kPackCodes = 16;  // codes per thread (8 packed bytes)
constexpr int kPackRows = 8;    // rows of a block (blockDim.y); blockDim.x = 32 chunks

// Two E4M3 codes (bytes 0 and 1 of `pair`) as biased integers: one conversion to a binary16
// pair, then + 1536 in binary16, where the spacing is 1 on [1024, 2048), so each half's
// bit pattern is 0x6600 (the pattern of 1536) plus its integer q.  Exact for the integers
// |q| <= 448 a quantizer writes (a fraction, which none writes, rounds to nearest).  As
// 0x6600 is a multiple of 16, the low four bits of a half are already q's nibble, and
// q lies in [-8, 7] exactly when (half + 8) & 0xFFF0 == 0x6600.
__device__ __forceinline__ uint32_t e4m3_pair_biased(uint32_t pair) {
  const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2(static_cast<__nv_fp8x2_storage_t>(pair), __NV_E4M3);
  const __half2 s = __hadd2(*reinterpret_cast<const __half2*>(&h), __half2(__half(1536.0f), __half(1536.0f)));
  return *reinterpret_cast<const uint32_t*>(&s);
}

// The E4M3 bytes of eight 4-bit two's complement codes (the nibbles of w, code k in bits
// 4k .. 4k+3) by byte permutes: the bytes of 0..7 and of -8..-1 are two 8-byte tables,
// each code's low three bits select within a table and its sign bit picks the table.
// prmt.b32 in its default mode: byte n of the result is byte (c >> 4n) & 7 of {b, a}, or,
// with bit 3 of that selector nibble set, that byte's sign bit replicated
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

__device__ __forceinline__ uint2 e4m3_of_nibbles(uint32_t w) {
  constexpr uint32_t kPos0 = 0x44403800u, kPos1 = 0x4E4C4A48u;   // 0, 1, 2, 3 | 4, 5, 6, 7
  constexpr uint32_t kNeg0 = 0xCACCCED0u, kNeg1 = 0xB8C0C4C8u;   // -8, -7, -6, -5 | -4 .. -1
  const uint32_t ws = w << 4;   // each even code's sign now at bit 7 of its byte
  uint2 out;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t sel = (w >> (16 * h)) & 0x7777u;
    const uint32_t pos = prmt(kPos0, kPos1, sel);
    const uint32_t neg = prmt(kNeg0, kNeg1, sel);
    // 0xFF in the bytes whose code is negative (sign-replicating permute of the sign bits:
    // code 2j's sign is bit 7 of byte j of ws, code 2j+1's bit 7 of byte j of w)
    const uint32_t mask = prmt(ws, w, h == 0 ? 0xD9C8u : 0xFBEAu);
    const uint32_t v = (pos & ~mask) | (neg & mask);
    if (h == 0) out.x = v; else out.y = v;
  }
  return out;
}

constexpr int kPackRowsInFlight = 4;   // rows a thread loads before working on them

// The 16 codes of a chunk as words (two BF16 or four E4M3 codes a word, low code first).
template <typename CodeT>
struct CodeChunk {
  uint32_t w[kPackCodes * sizeof(CodeT) / 4];
};

template <typename CodeT>
__device__ __forceinline__ CodeChunk<CodeT> load_chunk(const CodeT* src, int64_t c0, int64_t C, bool full) {
  constexpr int kWords = kPackCodes * static_cast<int>(sizeof(CodeT)) / 4;
  CodeChunk<CodeT> ch;
  if (full) {
#pragma unroll
    for (int k = 0; k < kWords / 4; ++k) {
      const uint4 t = __ldcs(reinterpret_cast<const uint4*>(src) + k);
      ch.w[4 * k] = t.x;
      ch.w[4 * k + 1] = t.y;
      ch.w[4 * k + 2] = t.z;
      ch.w[4 * k + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int k = 0; k < kWords; ++k) ch.w[k] = 0u;
#pragma unroll
    for (int k = 0; k < kPackCodes; ++k)
      if (c0 + k < C)
        ch.w[k * sizeof(CodeT) / 4] |= static_cast<uint32_t>(src[k])
                                       << (8 * sizeof(CodeT) * (k % (4 / sizeof(CodeT))));
  }
  return ch;
}

// the chunk's 16 nibbles (code k in bits 4 (k mod 8) of word k / 8); bad: a code outside
// [-8, 7]
template <typename CodeT>
__device__ __forceinline__ uint2 pack_chunk(const CodeChunk<CodeT>& ch, bool& bad) {
  uint32_t w[2] = {0u, 0u};
  if constexpr (sizeof(CodeT) == 1) {
    uint32_t off = 0u;   // bits outside 0x000F000F: a code outside [-8, 7]
#pragma unroll
    for (int k = 0; k < kPackCodes; k += 2) {
      const uint32_t b = e4m3_pair_biased((ch.w[k >> 2] >> (8 * (k & 3))) & 0xFFFFu);
      off |= (b + 0x00080008u) ^ 0x66006600u;
      w[k >> 3] |= ((b & 0xFu) | ((b >> 12) & 0xF0u)) << (4 * (k & 7));
    }
    bad |= (off & 0xFFF0FFF0u) != 0u;
  } else {
#pragma unroll
    for (int k = 0; k < kPackCodes; k += 2) {
      const int q0 = code_value<CodeT>(static_cast<CodeT>(ch.w[k >> 1] & 0xFFFFu));
      const int q1 = code_value<CodeT>(static_cast<CodeT>(ch.w[k >> 1] >> 16));
      bad |= static_cast<unsigned>(q0 + 8) > 15u || static_cast<unsigned>(q1 + 8) > 15u;
      w[k >> 3] |= (static_cast<uint32_t>(q0 & 0xF) | (static_cast<uint32_t>(q1 & 0xF) << 4)) << (4 * (k & 7));
    }
  }
  return make_uint2(w[0], w[1]);
}

// codes [R, ld] -> packed [R, ldp]; a code outside [-8, 7] (not a 4-bit code) is packed as
// its low nibble and flags SQ_DEV_INTERNAL.  Thread (x, y) of block (bx, by) packs the 16
// codes of chunk 32 bx + x of rows by 8 + y, then every 8 gridDim.y-th row, loading
// kPackRowsInFlight rows before packing them.
template <typename CodeT>
__global__ void __launch_bounds__(256) pack4_kernel(const CodeT* __restrict__ codes, int64_t R,
                                                    int64_t C, int64_t ld, uint8_t* __restrict__ out,
                                                    int64_t ldp, int vec, int* __restrict__ status) {
  constexpr int U = kPackRowsInFlight;
  const int64_t c0 = (static_cast<int64_t>(blockIdx.x) * 32 + threadIdx.x) * kPackCodes;
  if (c0 >= C) return;
  const bool full = vec && c0 + kPackCodes <= C;
  const int64_t nbytes = ((C < c0 + kPackCodes ? C : c0 + kPackCodes) - c0 + 1) / 2;
  const int64_t S = static_cast<int64_t>(gridDim.y) * kPackRows;
  bool bad = false;
  for (int64_t r = static_cast<int64_t>(blockIdx.y) * kPackRows + threadIdx.y; r < R; r += U * S) {
    CodeChunk<CodeT> in[U];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (r + u * S < R) in[u] = load_chunk(codes + (r + u * S) * ld + c0, c0, C, full);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (r + u * S >= R) break;
      const uint2 w = pack_chunk(in[u], bad);
      uint8_t* dst = out + (r + u * S) * ldp + c0 / 2;
      if (full) {
        *reinterpret_cast<uint2*>(dst) = w;
      } else {
#pragma unroll
        for (int k = 0; k < kPackCodes / 2; ++k)
          if (k < nbytes) dst[k] = static_cast<uint8_t>((k < 4 ? w.x : w.y) >> (8 * (k & 3)));
      }
    }
  }
  if (bad) atomicOr(status, kDevInternal);
}

template <typename CodeT>
__global__ void __launch_bounds__(256) unpack4_kernel(const uint8_t* __restrict__ in, int64_t ldp,
                                                      int64_t R, int64_t C, CodeT* __restrict__ codes,
                                                      int64_t ld, int vec) {
  constexpr int U = kPackRowsInFlight;
  const int64_t c0 = (static_cast<int64_t>(blockIdx.x) * 32 + threadIdx.x) * kPackCodes;
  if (c0 >= C) return;
  const bool full = vec && c0 + kPackCodes <= C;
  const int64_t nbytes = ((C < c0 + kPackCodes ? C : c0 + kPackCodes) - c0 + 1) / 2;
  const int64_t S = static_cast<int64_t>(gridDim.y) * kPackRows;
  for (int64_t r = static_cast<int64_t>(blockIdx.y) * kPackRows + threadIdx.y; r < R; r += U * S) {
    uint2 pw[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      pw[u] = make_uint2(0u, 0u);
      if (r + u * S >= R) continue;
      const uint8_t* src = in + (r + u * S) * ldp + c0 / 2;
      if (full) {
        pw[u] = __ldcs(reinterpret_cast<const uint2*>(src));
      } else {
#pragma unroll
        for (int k = 0; k < kPackCodes / 2; ++k)
          if (k < nbytes) (k < 4 ? pw[u].x : pw[u].y) |= static_cast<uint32_t>(src[k]) << (8 * (k & 3));
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (r + u * S >= R) break;
      CodeT* dst = codes + (r + u * S) * ld + c0;
      if constexpr (sizeof(CodeT) == 1) {
        const uint2 lo = e4m3_of_nibbles(pw[u].x), hi = e4m3_of_nibbles(pw[u].y);
        if (full) {
          *reinterpret_cast<uint4*>(dst) = make_uint4(lo.x, lo.y, hi.x, hi.y);
        } else {
          const uint32_t b[4] = {lo.x, lo.y, hi.x, hi.y};
#pragma unroll
          for (int k = 0; k < kPackCodes; ++k)   // constant indices: b stays in registers
            if (c0 + k < C) dst[k] = static_cast<CodeT>(b[k >> 2] >> (8 * (k & 3)));
        }
      } else {
        uint32_t cw[kPackCodes / 2];   // two BF16 codes a word
#pragma unroll
        for (int k = 0; k < kPackCodes; k += 2) {
          const uint32_t word = k < 8 ? pw[u].x : pw[u].y;
          const int n0 = (word >> (4 * (k & 7))) & 0xF, n1 = (word >> (4 * (k & 7) + 4)) & 0xF;
          cw[k >> 1] = static_cast<uint32_t>(code_of<CodeT>(n0 >= 8 ? n0 - 16 : n0)) |
                       (static_cast<uint32_t>(code_of<CodeT>(n1 >= 8 ? n1 - 16 : n1)) << 16);
        }
        if (full) {
#pragma unroll
          for (int k = 0; k < kPackCodes / 8; ++k)
            reinterpret_cast<uint4*>(dst)[k] = make_uint4(cw[4 * k], cw[4 * k + 1], cw[4 * k + 2], cw[4 * k + 3]);
        } else {
#pragma unroll
          for (int k = 0; k < kPackCodes; ++k)
            if (c0 + k < C) dst[k] = static_cast<CodeT>(cw[k >> 1] >> (16 * (k & 1)));
        }
      }
    }
  }
}

// grid of a pack / unpack launch: 32 chunks of 16 codes by 8 rows a block, about one
// resident wave (four blocks per SM); the blocks then walk the rows
static dim3 pack_grid(int64_t R, int64_t C) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    sms = 152;
  const int64_t gx = (C + 32 * kPackCodes - 1) / (32 * kPackCodes);
  int64_t gy = (R + kPackRows - 1) / kPackRows;
  const int64_t cap = (static_cast<int64_t>(sms) * 4 + gx - 1) / gx;
  if (gy > cap) gy = cap;
  if (gy > 65535) gy = 65535;
  return dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy < 1 ? 1 : gy));
}

__device__ __forceinline__ int map_bits(int G) { return G <= 2 ? 1 : (G <= 4 ? 2 : 4); }

// one packed byte per thread
__global__ void __launch_bounds__(256) pack_groups_kernel(const uint8_t* __restrict__ e, int64_t C,
                                                          int G, uint8_t* __restrict__ out) {
  const int w = map_bits(G), per = 8 / w;
  const int64_t nb = (C + per - 1) / per;
  for (int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b < nb;
       b += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    uint32_t v = 0;
    for (int k = 0; k < per && b * per + k < C; ++k)
      v |= static_cast<uint32_t>(e[b * per + k] & ((1 << w) - 1)) << (k * w);
    out[b] = static_cast<uint8_t>(v);
  }
}

__global__ void __launch_bounds__(256) unpack_groups_kernel(const uint8_t* __restrict__ in, int64_t C,
                                                            int G, uint8_t* __restrict__ e) {
  const int w = map_bits(G), per = 8 / w;
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; c < C;
       c += static_cast<int64_t>(gridDim.x) * blockDim.x)
    e[c] = static_cast<uint8_t>((in[c / per] >> ((c % per) * w)) & ((1 << w) - 1));
}

static unsigned grid_for(int64_t items) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    sms = 0;
  int64_t b = (items + 255) / 256;
  const int64_t cap = sms > 0 ? static_cast<int64_t>(sms) * 16 : 65535;
  if (b > cap) b = cap;
  return static_cast<unsigned>(b < 1 ? 1 : b);
}

static int done(const char* what) {
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? SQ_OK : cuda_fail(err, what);
}

}  // namespace sq

using namespace sq;

extern "C" sq_status shiftquant_pack_codes(const void* codes, int64_t rows, int64_t cols,
                                           int64_t ld, int bits, int n_groups, uint8_t* packed,
                                           int64_t ld_packed, int32_t* dev_status, void* stream) {
  fail(SQ_OK, "");
  if (!bits_ok(bits) || bits > 4 || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "pack_codes: codes of 2 to 4 bits (n_groups in [1, 8]) only");
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "pack_codes: negative size");
  if (rows == 0 || cols == 0) return SQ_OK;
  if (codes == nullptr || packed == nullptr || dev_status == nullptr || ld < cols ||
      ld_packed < (cols + 1) / 2)
    return fail(SQ_EINVAL, "pack_codes: NULL argument or leading dimension too small");
  const int cb = code_bytes(code_type(bits, n_groups));
  const int vec = aligned16(codes) && (ld * cb) % 16 == 0 &&
                  (reinterpret_cast<uintptr_t>(packed) & 7u) == 0 && ld_packed % 8 == 0;
  cudaStream_t s = as_stream(stream);
  const dim3 grid = pack_grid(rows, cols), block(32, kPackRows);
  if (cb == 1)
    pack4_kernel<uint8_t><<<grid, block, 0, s>>>(static_cast<const uint8_t*>(codes), rows, cols, ld,
                                                 packed, ld_packed, vec, dev_status);
  else
    pack4_kernel<uint16_t><<<grid, block, 0, s>>>(static_cast<const uint16_t*>(codes), rows, cols, ld,
                                                  packed, ld_packed, vec, dev_status);
  return done("pack4_kernel launch");
}

extern "C" sq_status shiftquant_unpack_codes(const uint8_t* packed, int64_t ld_packed, int64_t rows,
                                             int64_t cols, int bits, int n_groups, void* codes,
                                             int64_t ld, void* stream) {
  fail(SQ_OK, "");
  if (!bits_ok(bits) || bits > 4 || !groups_ok(n_groups))
    return fail(SQ_EINVAL, "unpack_codes: codes of 2 to 4 bits (n_groups in [1, 8]) only");
  if (rows < 0 || cols < 0) return fail(SQ_EINVAL, "unpack_codes: negative size");
  if (rows == 0 || cols == 0) return SQ_OK;
  if (codes == nullptr || packed == nullptr || ld < cols || ld_packed < (cols + 1) / 2)
    return fail(SQ_EINVAL, "unpack_codes: NULL argument or leading dimension too small");
  const int cb = code_bytes(code_type(bits, n_groups));
  const int vec = aligned16(codes) && (ld * cb) % 16 == 0 &&
                  (reinterpret_cast<uintptr_t>(packed) & 7u) == 0 && ld_packed % 8 == 0;
  cudaStream_t s = as_stream(stream);
  const dim3 grid = pack_grid(rows, cols), block(32, kPackRows);
  if (cb == 1)
    unpack4_kernel<uint8_t><<<grid, block, 0, s>>>(packed, ld_packed, rows, cols,
                                                   static_cast<uint8_t*>(codes), ld, vec);
  else
    unpack4_kernel<uint16_t><<<grid, block, 0, s>>>(packed, ld_packed, rows, cols,
                                                    static_cast<uint16_t*>(codes), ld, vec);
  return done("unpack4_kernel launch");
}

extern "C" int64_t shiftquant_packed_groups_bytes(int64_t channels, int n_groups) {
  if (channels < 0 || !groups_ok(n_groups)) return -1;
  const int per = 8 / (n_groups <= 2 ? 1 : (n_groups <= 4 ? 2 : 4));
  return (channels + per - 1) / per;
}

extern "C" sq_status shiftquant_pack_groups(const uint8_t* exp, int64_t channels, int n_groups,
                                            uint8_t* packed, void* stream) {
  fail(SQ_OK, "");
  if (!groups_ok(n_groups) || channels < 0) return fail(SQ_EINVAL, "pack_groups: bad arguments");
  if (channels == 0) return SQ_OK;
  if (exp == nullptr || packed == nullptr) return fail(SQ_EINVAL, "pack_groups: NULL argument");
  pack_groups_kernel<<<grid_for(shiftquant_packed_groups_bytes(channels, n_groups)), 256, 0,
                       as_stream(stream)>>>(exp, channels, n_groups, packed);
  return done("pack_groups_kernel launch");
}

extern "C" sq_status shiftquant_unpack_groups(const uint8_t* packed, int64_t channels, int n_groups,
                                              uint8_t* exp, void* stream) {
  fail(SQ_OK, "");
  if (!groups_ok(n_groups) || channels < 0) return fail(SQ_EINVAL, "unpack_groups: bad arguments");
  if (channels == 0) return SQ_OK;
  if (exp == nullptr || packed == nullptr) return fail(SQ_EINVAL, "unpack_groups: NULL argument");
  unpack_groups_kernel<<<grid_for(channels), 256, 0, as_stream(stream)>>>(packed, channels, n_groups,
                                                                          exp);
  return done("unpack_groups_kernel launch");
}
