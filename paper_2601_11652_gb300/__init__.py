"""GB300-native (sm_103a) batched speculative-verification step of WISP (arxiv 2601.11652).

One verification step (Sec. 4.5) = ragged paged GQA attention for every
request's k+1 new tokens over its cached prefix, then the lossless in-order
acceptance and target-token draw (Eq. 1-3) over the vocabulary.  The work is
done by hand-written CUDA kernels behind the C ABI in include/wisp_verify.h;
`binding` marshals torch tensors into that ABI and nothing else.
"""
__all__ = ["binding", "workload"]
