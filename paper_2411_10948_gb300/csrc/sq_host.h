// Host-side helpers shared by the translation units of libshiftquant: error reporting,
// argument checks and the code-format rules.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

#include "../../include/shiftquant.h"

namespace sq {

// record a message for shiftquant_last_error() and return `status`
int fail(int status, const char* fmt, ...);

inline int cuda_fail(cudaError_t err, const char* what) {
  return fail(SQ_ECUDA, "%s failed: %s", what, cudaGetErrorString(err));
}

inline int q_of_bits(int bits) { return (1 << (bits - 1)) - 1; }

inline bool bits_ok(int bits) { return bits >= 2 && bits <= 8; }
inline bool groups_ok(int g) { return g >= 1 && g <= 8; }

// FP8 E4M3 represents every integer up to 16 and every 4-significant-bit integer up to
// 448, so it holds q (|q| <= 15) and the shifted weight codes q 2^(G-1) when those stay
// below 448; otherwise BF16 (8 significant bits) holds q 2^(G-1) for all bits <= 8.
inline int code_type(int bits, int groups) {
  const int Q = q_of_bits(bits);
  return (Q <= 15 && (Q << (groups - 1)) <= 448) ? SQ_CODE_E4M3 : SQ_CODE_BF16;
}

inline int code_bytes(int type) { return type == SQ_CODE_E4M3 ? 1 : 2; }

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

}  // namespace sq
