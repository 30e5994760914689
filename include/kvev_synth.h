/*
 * kvev_synth.h -- C ABI of libkvev_synth.so, the device-side generator of the
 * seeded synthetic KV caches and window queries used by the tests and the
 * benchmark.  It is not part of the eviction method: it only fills buffers
 * with the same bits as paper_2606_15157_gb300/inputs.py computes on the host,
 * so that full-size workloads (tens of GB) need no host generation or upload.
 *
 * Generator (identical on both sides):
 *   h(i)   = SplitMix64 output of key + (i + 1) * 0x9E3779B97F4A7C15
 *   g(i)   = fp32(sum of the four 16-bit fields of h(i) - 131070) * IH4_SCALE
 *            (an Irwin-Hall(4) variate standardised to mean 0, variance 1),
 *            rounded to bf16 (nearest-even);
 *   v(i)   = low 16 bits of h(i), exponent 0xFF lowered to 0xFE.
 * `key` is the stream key computed on the host (inputs.stream_key).
 * All calls are asynchronous on `stream` (a cudaStream_t); return 0 or a
 * CUDA error code.
 */
#ifndef KVEV_SYNTH_H
#define KVEV_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define KVEV_SYNTH_API __attribute__((visibility("default")))
#else
#define KVEV_SYNTH_API
#endif

/* K of one layer, bf16 [B][H_kv][S_cap][d]: element (s, h, pos, j) = g(flat).
 * Positions < sink_tokens are scaled by sink_scale (fp32, before rounding).
 * If u != NULL (device fp32 [H_kv][d]) positions in [plant_lo, plant_hi) get
 * gamma * u[h] added (fp32, before rounding). */
KVEV_SYNTH_API int kvev_synth_k(uint16_t *dst, int B, int H_kv, int S_cap, int d, uint64_t key,
                                int sink_tokens, float sink_scale, int plant_lo, int plant_hi,
                                float gamma, const float *u, void *stream);

/* Q_win of one layer, bf16 [B][H_q][W][d]: element = g(flat); if u != NULL the
 * value is alpha * u[hq / G] + 0.1 * g(flat) (fp32, before rounding). */
KVEV_SYNTH_API int kvev_synth_q(uint16_t *dst, int B, int H_q, int W, int d, int G, uint64_t key,
                                float alpha, const float *u, void *stream);

/* count bf16 values g(index_base + i). */
KVEV_SYNTH_API int kvev_synth_gauss(uint16_t *dst, uint64_t count, uint64_t key, uint64_t index_base,
                                    void *stream);

/* count bf16 bit patterns v(index_base + i). */
KVEV_SYNTH_API int kvev_synth_bits(uint16_t *dst, uint64_t count, uint64_t key, uint64_t index_base,
                                   void *stream);

#ifdef __cplusplus
}
#endif
#endif
