"""GB300 microbenchmarks behind the attention kernel's design; see __main__.py."""
