/*
 * pad_moe_oracle.c -- double-precision CPU oracle for two more row-wise
 * operators the paper traces: the Hyena FFT-size padding operator and the
 * MoE group score.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is part of the oracle, not the
 * product: only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it.  It shares no code, header, table or constant
 * with the CUDA library, and it never includes anything from it.
 *
 * Hyena FFT-size padding (§6, "Representative cross-layer trace"): every row
 * of seqlen inputs is scaled and followed by zeros up to fft_size,
 *
 *   y[r][c] = scale * x[r][c]   for 0 <= c < seqlen
 *   y[r][c] = 0                 for seqlen <= c < fft_size.
 *
 * MoE group score (§2.1, "A Running Example"): the scores of a token are cut
 * into consecutive groups of `group` experts, and each group's score is the
 * largest sum of two distinct members,
 *
 *   out[t][g] = max over i != j of (v_i + v_j),  v = scores of group g,
 *
 * which equals the sum of the group's two largest values, a tied maximum
 * counting twice.  The oracle takes the pairwise definition literally: every
 * ordered pair i != j, in order, by brute force.  Scores are finite or -inf
 * (a masked expert).  The sum of two doubles that came from float32 or
 * bfloat16 values is exact.
 */
#include <math.h>
#include <stdint.h>

void oracle_pad_scale(const double *x, double *y, int64_t rows, int64_t seqlen,
                      int64_t fft_size, double scale)
{
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < fft_size; ++c)
            y[r * fft_size + c] = c < seqlen ? scale * x[r * seqlen + c] : 0.0;
}

void oracle_moe_group_top2(const double *v, double *out, int64_t tokens,
                           int64_t experts, int64_t group)
{
    const int64_t groups = experts / group;
    for (int64_t t = 0; t < tokens; ++t) {
        for (int64_t g = 0; g < groups; ++g) {
            const double *w = v + t * experts + g * group;
            double best = -INFINITY;
            for (int64_t i = 0; i < group; ++i)
                for (int64_t j = 0; j < group; ++j)
                    if (i != j && w[i] + w[j] > best)
                        best = w[i] + w[j];
            out[t * groups + g] = best;
        }
    }
}
