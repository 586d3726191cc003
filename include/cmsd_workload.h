/*
 * cmsd_workload.h -- C ABI of libcmsd_workload.so: the device-side synthetic
 * logit generator of the decode-loop simulation (Algorithm 1 of
 * arXiv 2508.15371 run as a control loop over synthetic logits).
 *
 * This library holds no part of the method: it only produces drafter and
 * verifier logits and drafted tokens, bit-identical to the host generator
 * paper_2508_15371_gb300/workloads.py (decode_row_host).  It stands in for the
 * paper's drafter and verifier models (Sec. IV.A), which are not available.
 *
 * Row (b, i) at iteration `it` (row id r = b * (K_max + 1) + i):
 *   n1[v], n2[v] = table[u16 >> 3] with u16 the 16-bit half (v & 1) of Philox4x32-10
 *                  word (v >> 1) & 3 of counter (v >> 3, r, it, 0xC0000002 / 0xC0000003),
 *                  key (seed lo, seed hi)
 *   spike token  = (word 0 of counter (0, r, it, 0xC0000004)) * V >> 32
 *   draft[v]     = n1[v], plus heights_it[b] at the spike token (float add)
 *   target[v]    = draft[v] + 0.8f * n2[v]  (float multiply, then add)
 *   token[r]     = first argmax of draft
 * Drafter rows and tokens are written for i < k_row[b]; verifier rows for
 * i < k_row[b] + (Kt - K_max), i.e. with Kt = K_max + 1 also the row after the
 * drafted window (the verifier's extra row).  Other rows are not written.
 */
#ifndef CMSD_WORKLOAD_H
#define CMSD_WORKLOAD_H
#include <stddef.h>
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif

/* table: float[8192] device (normal quantiles at (j + 1/2) / 8192); heights_it: float[B] device
 * (spike heights of this iteration); k_row: int32[B] device (NULL = K_max);
 * Kt: verifier rows per sequence, K_max or K_max + 1;
 * draft: float [B][K_max][V] device; target: float [B][Kt][V] device;
 * tokens: int32 [B][K_max] device.
 * Returns 0, or -1 on a bad argument, -3 on a CUDA launch error. */
int cmsd_gen_decode_rows(const float* table, const float* heights_it, uint32_t it, int B, int K_max,
                         int Kt, int V, const int32_t* k_row, uint64_t seed, float* draft,
                         float* target, int32_t* tokens, void* stream);

#ifdef __cplusplus
}
#endif
#endif
