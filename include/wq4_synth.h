/*
 * wq4_synth.h -- device-side seeded generator for synthetic packed weights
 * and attention inputs.
 *
 * Not part of the method: it only fills buffers with random bits so that
 * large synthetic models (1-8B parameters) can be created directly in HBM.
 * It implements the same counter-based SplitMix64 draws as the host
 * generator (Steele, Lea and Flood, OOPSLA 2014):
 *   mix64(z)       SplitMix64 output function
 *   key(seed, sid) = mix64(seed * 0x9E3779B97F4A7C15 + sid * 0xD1B54A32D192ED03)
 *   u64(key, i)    = mix64(key + (i + 1) * 0x9E3779B97F4A7C15)      (mod 2^64)
 * and must reproduce the host generator bit for bit.
 */
#ifndef WQ4_SYNTH_H
#define WQ4_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Words [word_start, word_start + nwords) of a packed-code stream:
 * word 2m = low 32 bits of u64(key, m), word 2m+1 = high 32 bits.
 * symmetric = 0: every code uniform on 0..15 (covers the whole format).
 * symmetric != 0: then every code equal to 15 becomes 7, so codes lie in
 * 0..14 with mean 7, the range of symmetric 4-bit quantisation (|q - 7| <= 7)
 * and zero-mean weights, as trained models have; used for whole synthetic
 * models, whose activations would otherwise drift out of fp16 range.
 * W: device uint32 buffer of nwords entries; word_start and nwords even.
 * Returns 0, -1 on bad arguments, -4 on a CUDA launch failure. */
int wq4_synth_codes(uint32_t* W, int64_t word_start, int64_t nwords,
                    uint64_t seed, uint64_t sid, int symmetric, void* stream);

/* Scales [start, start + n): fp16_RNE(lo + (hi - lo) * u),
 * u = (u64(key, i) >> 11) * 2^-53, one fp64 multiply then one fp64 add,
 * a single rounding to fp16.  s: device uint16 buffer of n entries. */
int wq4_synth_scales(uint16_t* s, int64_t start, int64_t n, uint64_t seed,
                     uint64_t sid, double lo, double hi, void* stream);

/* Attention inputs [start, start + n) ("sum4"): fp16_RNE((a + b + c + d -
 * 131070) * 2^-15), a..d the four 16-bit fields of u64(key, i) (an
 * Irwin-Hall approximation of a normal draw, standard deviation 2/sqrt(3)).
 * out: device uint16 buffer of n entries. */
int wq4_synth_sum4(uint16_t* out, int64_t start, int64_t n, uint64_t seed, uint64_t sid, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* WQ4_SYNTH_H */
