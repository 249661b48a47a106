// stream.cuh -- how the streaming kernels cut their work.
//
// A launch streams R rows in fixed-size pieces (tiles of kTileBytes for the
// expansion, 2 KB chunks for the verification stream).  The R * pieces_per_row
// pieces are split into G contiguous ranges, one per worker (a CTA or a warp),
// so every worker moves the same number of bytes; the part of a row that falls
// in one worker's range is a "segment" of that row.
#pragma once

#include <stdint.h>

namespace rheo {

constexpr int kTileBytes = 16384;

// Static split of R * pieces_per_row pieces over G workers.
struct TileSplit {
    int64_t total;  // R * pieces_per_row
    int G;          // workers
    __host__ __device__ __forceinline__ int64_t begin(int i) const { return (int64_t)i * total / G; }
    // worker whose range holds piece t
    __host__ __device__ __forceinline__ int owner(int64_t t) const { return (int)((t * G + G - 1) / total); }
};

}  // namespace rheo
