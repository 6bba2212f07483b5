// reduce_jobs.h -- several fixed-order chunk reductions in one launch.
//
// The backward kernels leave per-chunk column partials (gate, bias, shift,
// scale and norm-scale gradients); each partial set is summed by the fixed
// fp64 order of reduce_chunks.  A job is one such sum; a batch of up to
// kMaxReduceJobs jobs runs as one launch whose CTAs each take 32 columns of
// one job (and one sample for a per-sample job), with the same per-column
// order as a job launched alone, so batching changes no result bit.
#pragma once

#include "internal.h"

namespace ff {

struct ReduceJob {
    const float* part;   // chunk partials, row = chunk, pitch ld_part floats
    int64_t ld_part;
    int ncols;           // columns [0, ncols) of each chunk row
    ChunkSpans sp;       // the chunk rows summed (per sample b: first + b count)
    int per_sample;      // 1: out[b * ld_out + j] for b < B; 0: out[j] over all chunks
    float* out;
    int64_t ld_out;
};

constexpr int kMaxReduceJobs = 8;

// Runs jobs[0 .. n) (any n >= 0, in launches of up to kMaxReduceJobs) on
// stream; B = samples of the per-sample jobs.
int reduce_chunks_batch(const ReduceJob* jobs, int n, int B, cudaStream_t stream);

// One-span job helpers.
inline ChunkSpans chunk_span(int first, int count) {
    ChunkSpans sp{};
    sp.n = 1;
    sp.first[0] = first;
    sp.count[0] = count;
    return sp;
}

}  // namespace ff
