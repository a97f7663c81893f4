// FP8 weight storage, host side (dcl_fp8_quantise): bf16 weights -> E4M3 codes with one
// power-of-two scale per output row.  A serving refinement outside the paper; the format
// is E4M3 of the OCP 8-bit floating-point specification (bias 7, subnormals m * 2^-9, no
// infinities, 448 the largest magnitude).  Plain host code: integer and double
// arithmetic only, the same result on every host.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <string>

#include "../../include/dcleap.h"
#include "common.cuh"

namespace {

constexpr double kE4M3Max = 448.0;

double bf16_value(uint16_t bits) {
  const uint32_t u = (uint32_t)bits << 16;
  float f;
  std::memcpy(&f, &u, sizeof f);
  return (double)f;
}

// The least integer e with amax <= 448 * 2^e (0 when amax is 0).  ldexp is exact, so the
// comparisons decide; log2 only gives the starting guess.
int row_exponent(double amax) {
  if (!(amax > 0.0)) return 0;
  int e = (int)std::ceil(std::log2(amax / kE4M3Max));
  while (amax > std::ldexp(kE4M3Max, e)) ++e;
  while (amax <= std::ldexp(kE4M3Max, e - 1)) --e;
  return e;
}

// Code of the E4M3 value nearest to x (|x| <= 448), ties to the even mantissa, the sign
// of x kept.  Values in the binade [2^E, 2^(E+1)) are spaced 2^(E-3) (E >= -6); below
// 2^-6 the subnormals keep binade -6's spacing 2^-9.  nearbyint rounds half to even in
// the default rounding mode, and a / spacing is exact.
uint8_t e4m3_code(double x) {
  const uint8_t sign = std::signbit(x) ? 0x80 : 0x00;
  const double a = std::fabs(x);
  int ex = 0;
  std::frexp(a, &ex);  // a = f * 2^ex with f in [0.5, 1): binade ex - 1
  const int E = std::max(ex - 1, -6);
  const int n = (int)std::nearbyint(std::ldexp(a, 3 - E));  // 0..16
  int field, mant;
  if (n >= 16) {  // rounded up into the next binade
    field = E + 1 + 7;
    mant = 0;
  } else if (n >= 8) {
    field = E + 7;
    mant = n - 8;
  } else {  // only when E = -6: the subnormal n * 2^-9 (or zero)
    field = 0;
    mant = n;
  }
  return (uint8_t)(sign | (field << 3) | mant);
}

}  // namespace

extern "C" dcl_status dcl_fp8_quantise(const uint16_t* w, int64_t rows, int64_t cols, uint8_t* codes,
                                       int32_t* exps) {
  if (!w || !codes || !exps || rows < 1 || cols < 1) {
    dcl::set_thread_error("dcl_fp8_quantise: NULL pointer or rows / cols < 1");
    return DCL_ERR_INVALID_ARG;
  }
  for (int64_t n = 0; n < rows; ++n) {
    const uint16_t* row = w + n * cols;
    double amax = 0.0;
    for (int64_t k = 0; k < cols; ++k) {
      if ((row[k] & 0x7F80u) == 0x7F80u) {  // exponent all ones: infinity or NaN
        dcl::set_thread_error(("dcl_fp8_quantise: non-finite weight at row " + std::to_string(n) + ", column " +
                               std::to_string(k)).c_str());
        return DCL_ERR_INVALID_ARG;
      }
      amax = std::max(amax, std::fabs(bf16_value(row[k])));
    }
    const int e = row_exponent(amax);
    exps[n] = e;
    uint8_t* out = codes + n * cols;
    for (int64_t k = 0; k < cols; ++k) out[k] = e4m3_code(std::ldexp(bf16_value(row[k]), -e));
  }
  return DCL_OK;
}
