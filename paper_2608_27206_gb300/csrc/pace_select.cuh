// Shared pieces of the one-CTA radix selections (top-K of S_final, tail of d_i).
#pragma once
#include <cstdint>

namespace pace {

// Warp 0 of the block finds the digit of the `remaining`-th largest key among the counts
// hist[0..255] of the current digit: sel[0] = digit, sel[1] = number of keys in higher bins.
// Lane l scans bins 255 - 8l .. 248 - 8l, so a prefix over the lanes walks the bins from the
// top.  Equivalent to walking d = 255 .. 1 and stopping at the first bin whose cumulative count
// reaches `remaining` (bin 0 if none does before it).
__device__ __forceinline__ void warp_digit_search(const unsigned* hist, unsigned remaining, unsigned* sel) {
  const int lane = threadIdx.x & 31;
  const int top = 255 - 8 * lane;
  unsigned c[8];
  unsigned s = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    c[i] = hist[top - i];
    s += c[i];
  }
  unsigned incl = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  const unsigned hit = __ballot_sync(0xffffffffu, incl >= remaining);
  const int L = hit ? __ffs(hit) - 1 : 31;
  if (lane == L) {
    unsigned above = incl - s;
    int digit = top - 7;
    bool found = false;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int d = top - i;
      if (!found) {
        if (d == 0 || above + c[i] >= remaining) {
          digit = d;
          found = true;
        } else {
          above += c[i];
        }
      }
    }
    sel[0] = static_cast<unsigned>(digit);
    sel[1] = above;
  }
}

// Rank of every entry of a short list (c <= blockDim.x = 1024 keys in shared memory): gt = entries
// above list[i], ge = entries at or above it.  Each entry's count is spread over P threads (P the
// largest power of two with c P <= 1024, at most 32): thread t takes entry t / P and every P-th
// comparison, and the P partial counts meet by shuffles inside their aligned group of lanes.
// Every thread of the block calls it (its control flow is uniform per warp); it returns true on
// the one thread per entry (part 0) that holds the complete counts.
__device__ __forceinline__ bool rank_in_list(const unsigned* list, unsigned c, int& i, unsigned& gt, unsigned& ge) {
  unsigned P = 1u;
  while (P < 32u && 2u * P * c <= blockDim.x) P <<= 1;
  const unsigned t = threadIdx.x;
  gt = ge = 0u;
  i = static_cast<int>(t / P);
  if ((t & ~31u) >= c * P) return false;   // the whole warp is past the list
  const unsigned part = t & (P - 1u);
  const bool valid = static_cast<unsigned>(i) < c;
  if (valid) {
    const unsigned mine = list[i];
    for (unsigned j = part; j < c; j += P) {
      const unsigned o = list[j];
      gt += o > mine;
      ge += o >= mine;
    }
  }
  for (unsigned o = 1u; o < P; o <<= 1) {
    gt += __shfl_xor_sync(0xffffffffu, gt, static_cast<int>(o));
    ge += __shfl_xor_sync(0xffffffffu, ge, static_cast<int>(o));
  }
  return valid && part == 0u;
}

}  // namespace pace
