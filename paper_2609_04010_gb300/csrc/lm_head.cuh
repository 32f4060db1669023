// Declarations of the fused LM head + row statistics (lm_head.cu), used by the ABI.
#pragma once

#include "common.cuh"

namespace specv {

constexpr int kLmTileN = 224;  // vocab rows per tile (MMA N; 128,256 / 224 = 573 tiles, 1.9 waves)
constexpr int kLmTileM = 128;  // hidden-state rows per tile (MMA M)
struct LmLayout {
  size_t parts;  // 16 B [rows][vocab tiles]: (max, sum, argmax, token logit) per tile
  size_t end;
  int ntiles_n, ntiles_m;
};
LmLayout lm_layout(const spec_lm_head_args_t& a, size_t base);
// starve (test hook only): the producer issues no copies, so the kernel's bounded waits
// run out and it returns with SPEC_FLAG_TIMEOUT set (outputs undefined).
cudaError_t launch_lm_head(const spec_lm_head_args_t& a, const LmLayout& L, char* ws,
                           cudaStream_t stream, bool starve = false);

}  // namespace specv
