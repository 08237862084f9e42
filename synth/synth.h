/*
 * Seeded synthetic-input generator (test and benchmark infrastructure).
 *
 * Two independent implementations of one definition (SplitMix64 counter
 * streams feeding an Irwin-Hall(12) normal, rounded to bf16 by
 * round-to-nearest-even): a host one in synth_host.c and a device one in
 * synth_dev.cu. Neither contains any arithmetic of the attention method.
 *
 * Device entry points return 0 on success, 1 on a bad argument (nothing
 * launched) and 2 on a launch error. All work is enqueued on `stream`
 * (a cudaStream_t passed as void*); nothing is allocated.
 */
#ifndef HSA_SYNTH_H
#define HSA_SYNTH_H
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif

/* out[i] = bf16(ih12(seed, offset + i)) for i < n; out is device memory of n uint16. */
int synth_dev_fill_bf16(void* out, int64_t n, uint64_t seed, int64_t offset, void* stream);

/* For r < n_rows and c < row_len:
 *   x[rows[r] * row_len + c] = bf16(float(x[...]) + vecs[r * vec_stride + c]).
 * x, rows and vecs are device pointers; vec_stride 0 adds one vector to every row.
 * rows must be distinct. */
int synth_dev_add_rows(void* x, int64_t row_len, const int64_t* rows, const float* vecs,
                       int64_t n_rows, int64_t vec_stride, void* stream);

/* K[b, t, g, e] = bf16(float(K[b, t, g, e]) + off[b, t / S, g, e]) for t < (L / S) * S;
 * K is [B, L, Hkv, d] bf16 and off is [B, L / S, Hkv, d] fp32, both on the device. */
int synth_dev_add_chunk_offsets(void* K, int B, int L, int Hkv, int d, int S, const float* off,
                                void* stream);

#ifdef __cplusplus
}
#endif
#endif
