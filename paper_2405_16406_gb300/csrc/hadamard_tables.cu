// hadamard_tables.cu -- host construction of the small Kronecker factor H_s
// of the online rotation (Sec. 3.1, R4 of non-power-of-two size).
//
// Paley I (order q + 1, q a prime power with q = 3 mod 4): H = I + S with
// S = [[0, 1..1], [-1.., Q]] and Q[i][j] = chi(a_i - a_j), chi = +1 on the
// nonzero squares of GF(q) and -1 on the other nonzero elements.  Field
// elements are indexed as in the header: GF(p) = integers mod p; GF(27) =
// GF(3)[t]/(t^3 + 2t + 1) with index c0 + 3 c1 + 9 c2.
//
// The square set is found by squaring every nonzero element (no Euler
// criterion), with GF(27) elements held as coefficient triples.
#include <array>
#include <cstring>

#include "spinq_internal.h"

namespace spinq {
namespace {

struct Gf {
  int q;
  bool ext3;  // GF(27) as polynomials over GF(3)

  int sub(int a, int b) const {
    if (!ext3) return (a - b + q) % q;
    int r = 0;
    for (int d = 0, p = 1; d < 3; ++d, p *= 3) r += ((a / p % 3) - (b / p % 3) + 3) % 3 * p;
    return r;
  }

  int mul(int a, int b) const {
    if (!ext3) return a * b % q;
    // coefficient triples, product of degree <= 4
    std::array<int, 3> x{a % 3, a / 3 % 3, a / 9 % 3}, y{b % 3, b / 3 % 3, b / 9 % 3};
    std::array<int, 5> z{};
    for (int i = 0; i < 3; ++i)
      for (int j = 0; j < 3; ++j) z[i + j] += x[i] * y[j];
    // t^4 = t^2 + 2t and t^3 = t + 2 (from t^3 + 2t + 1 = 0 over GF(3))
    z[2] += z[4];
    z[1] += 2 * z[4];
    z[1] += z[3];
    z[0] += 2 * z[3];
    return z[0] % 3 + 3 * (z[1] % 3) + 9 * (z[2] % 3);
  }
};

}  // namespace

bool build_small_hadamard(int n, SmallHadamard* out) {
  std::memset(out, 0, sizeof(*out));
  out->n = n;
  if (n == 1) return true;
  const int q = n - 1;
  Gf f{q, q == 27};
  if (!(q == 11 || q == 19 || q == 27)) return false;
  bool square[32] = {false};
  for (int a = 1; a < q; ++a) square[f.mul(a, a)] = true;
  for (int r = 0; r < n; ++r)
    for (int c = 0; c < n; ++c) {
      int h;
      if (r == c)
        h = 1;  // I + S with S zero on the diagonal
      else if (r == 0)
        h = 1;
      else if (c == 0)
        h = -1;
      else
        h = square[f.sub(r - 1, c - 1)] ? 1 : -1;
      if (h < 0) out->neg[r] |= 1u << c;
    }
  return true;
}

}  // namespace spinq
