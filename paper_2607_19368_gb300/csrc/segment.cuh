// Problem table shared by the SimHash, segment and aggregation kernels and
// by the compress driver.  A "problem" is one token set that is compressed
// independently: the compressible region of a prompt (global backend) or one
// window (adaptive backend).
#pragma once

#include <cstdint>

namespace sls {

struct ProbDesc {
  int64_t tok_row;   // first token row (b * N + pos0); also its Phi/Q/U row base
  int64_t q1off;     // offset of its Lanczos start vector in q1
  int64_t out0;      // first output macro row (b * M + ...)
  int64_t phi_row;   // first row in Phi / Q / U (spectral problems)
  int pos0;          // position of its first token inside the prompt
  int n;             // tokens
  int m;             // macro-tokens to produce (exact budget)
  int bits;          // SimHash bits
  int spectral;      // 1 = Spectral-LSH, 0 = chunk
  int chunk_k;       // chunk backend group size k (0 = m array_split groups)
  int spec_idx;      // index in the compacted spectral list (or -1)
  int out_local;     // first output macro index inside its prompt
};

}  // namespace sls
