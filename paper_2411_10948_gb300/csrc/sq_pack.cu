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

// codes [R, ld] -> packed [R, ldp]; a code outside [-8, 7] (not a 4-bit code) is packed as
// its low nibble and flags SQ_DEV_INTERNAL
template <typename CodeT>
__global__ void __launch_bounds__(256) pack4_kernel(const CodeT* __restrict__ codes, int64_t R,
                                                    int64_t C, int64_t ld, uint8_t* __restrict__ out,
                                                    int64_t ldp, int vec, int* __restrict__ status) {
  const int64_t per_row = (C + kPackCodes - 1) / kPackCodes;
  const int64_t n = R * per_row;
  bool bad = false;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / per_row;
    const int64_t c0 = (i - r * per_row) * kPackCodes;
    const CodeT* src = codes + r * ld + c0;
    alignas(16) CodeT v[kPackCodes];
    if (vec && c0 + kPackCodes <= C) {
#pragma unroll
      for (int k = 0; k < kPackCodes * static_cast<int>(sizeof(CodeT)) / 16; ++k)
        reinterpret_cast<uint4*>(v)[k] = __ldcs(reinterpret_cast<const uint4*>(src) + k);
    } else {
#pragma unroll
      for (int k = 0; k < kPackCodes; ++k) v[k] = c0 + k < C ? src[k] : CodeT(0);
    }
    uint32_t w[2] = {0u, 0u};
#pragma unroll
    for (int k = 0; k < kPackCodes; ++k) {
      const int q = code_value<CodeT>(v[k]);
      bad |= q < -8 || q > 7;
      w[k >> 3] |= static_cast<uint32_t>(q & 0xF) << (4 * (k & 7));
    }
    uint8_t* dst = out + r * ldp + c0 / 2;
    const int64_t nbytes = ((C < c0 + kPackCodes ? C : c0 + kPackCodes) - c0 + 1) / 2;
    if (vec && nbytes == kPackCodes / 2) {
      *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
    } else {
      for (int k = 0; k < nbytes; ++k) dst[k] = static_cast<uint8_t>(w[k >> 2] >> (8 * (k & 3)));
    }
  }
  if (bad) atomicOr(status, kDevInternal);
}

template <typename CodeT>
__global__ void __launch_bounds__(256) unpack4_kernel(const uint8_t* __restrict__ in, int64_t ldp,
                                                      int64_t R, int64_t C, CodeT* __restrict__ codes,
                                                      int64_t ld, int vec) {
  const int64_t per_row = (C + kPackCodes - 1) / kPackCodes;
  const int64_t n = R * per_row;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / per_row;
    const int64_t c0 = (i - r * per_row) * kPackCodes;
    const uint8_t* src = in + r * ldp + c0 / 2;
    const int64_t nbytes = ((C < c0 + kPackCodes ? C : c0 + kPackCodes) - c0 + 1) / 2;
    uint32_t w[2] = {0u, 0u};
    if (vec && nbytes == kPackCodes / 2) {
      const uint2 t = __ldcs(reinterpret_cast<const uint2*>(src));
      w[0] = t.x;
      w[1] = t.y;
    } else {
      for (int k = 0; k < nbytes; ++k) w[k >> 2] |= static_cast<uint32_t>(src[k]) << (8 * (k & 3));
    }
    alignas(16) CodeT v[kPackCodes];
#pragma unroll
    for (int k = 0; k < kPackCodes; ++k) {
      const int nib = (w[k >> 3] >> (4 * (k & 7))) & 0xF;
      v[k] = code_of<CodeT>(nib >= 8 ? nib - 16 : nib);
    }
    CodeT* dst = codes + r * ld + c0;
    if (vec && c0 + kPackCodes <= C) {
#pragma unroll
      for (int k = 0; k < kPackCodes * static_cast<int>(sizeof(CodeT)) / 16; ++k)
        reinterpret_cast<uint4*>(dst)[k] = reinterpret_cast<const uint4*>(v)[k];
    } else {
      for (int k = 0; k < kPackCodes && c0 + k < C; ++k) dst[k] = v[k];
    }
  }
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
  const int64_t items = rows * ((cols + kPackCodes - 1) / kPackCodes);
  cudaStream_t s = as_stream(stream);
  if (cb == 1)
    pack4_kernel<uint8_t><<<grid_for(items), 256, 0, s>>>(static_cast<const uint8_t*>(codes), rows,
                                                          cols, ld, packed, ld_packed, vec, dev_status);
  else
    pack4_kernel<uint16_t><<<grid_for(items), 256, 0, s>>>(static_cast<const uint16_t*>(codes), rows,
                                                           cols, ld, packed, ld_packed, vec, dev_status);
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
  const int64_t items = rows * ((cols + kPackCodes - 1) / kPackCodes);
  cudaStream_t s = as_stream(stream);
  if (cb == 1)
    unpack4_kernel<uint8_t><<<grid_for(items), 256, 0, s>>>(packed, ld_packed, rows, cols,
                                                            static_cast<uint8_t*>(codes), ld, vec);
  else
    unpack4_kernel<uint16_t><<<grid_for(items), 256, 0, s>>>(packed, ld_packed, rows, cols,
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
