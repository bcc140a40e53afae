// Host-side work split of the decoding step, shared by its kernels' file and the C ABI.
#pragma once
#include <stddef.h>

namespace hdsfa {

struct DecodePlan {
  int G, M, ngroups, nsplit, chunk, rg;
  bool tc;  // head dim 256 with <= 128 query rows per K/V head: the tcgen05 kernel
  size_t part_o_bytes, part_ml_bytes;
};
DecodePlan decode_plan(int B, int maxT, int n, int Hq, int Hkv, int Dh, int mode, int window);
size_t decode_ws_bytes(const DecodePlan& p);

}  // namespace hdsfa
